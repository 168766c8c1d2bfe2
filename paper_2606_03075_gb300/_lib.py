"""ctypes loader of libtgvkv.so: symbol signatures only, no logic.

The library must have been built (``paper_2606_03075_gb300.build.build()``);
there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtgvkv.so")

c_void_p, c_int, c_int32, c_int64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int32, ctypes.c_int64
c_float, c_double, c_size_t, c_char_p = ctypes.c_float, ctypes.c_double, ctypes.c_size_t, ctypes.c_char_p


class Desc(ctypes.Structure):
    """Mirror of ``tgvkv_desc`` (include/tgvkv.h)."""
    _fields_ = [("L", c_int32), ("H_q", c_int32), ("H_kv", c_int32), ("d", c_int32),
                ("N", c_int32), ("N_v", c_int32), ("n_win", c_int32),
                ("softmax_scale", c_float), ("w_layer_stride", c_int64),
                ("budget_basis", c_int32), ("weight_mode", c_int32),
                ("keep_first", c_int32), ("keep_last", c_int32), ("budget_stat", c_int32),
                ("head_budgets", c_int32)]


BASIS_VISION, BASIS_ALL = 0, 1
WEIGHTS_GIVEN, WEIGHTS_EQ7 = 0, 1
STAT_TV, STAT_TT, STAT_UNIFORM = 0, 1, 2


_P = ctypes.POINTER(Desc)

# name -> (restype, argtypes); the exported C ABI, one entry per declaration
SIGNATURES = {
    "tgvkv_workspace_size": (c_size_t, [_P]),
    "tgvkv_vision_budget_total": (c_int64, [_P, c_double]),
    "tgvkv_budget_total": (c_int64, [_P, c_double]),
    "tgvkv_retained_rows": (c_int64, [_P, c_double]),
    "tgvkv_text_scores": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_void_p]),
    "tgvkv_score": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                            c_void_p, c_void_p, c_void_p, c_void_p]),
    "tgvkv_budget": (c_int, [_P, c_void_p, c_double, c_void_p, c_void_p, c_void_p]),
    "tgvkv_select": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                             c_void_p, c_void_p]),
    "tgvkv_select_tpr": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                 c_void_p, c_void_p, c_void_p]),
    "tgvkv_compact": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                              c_int64, c_void_p, c_void_p]),
    "tgvkv_select_compact": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_int64,
                                     c_void_p, c_void_p]),
    "tgvkv_select_compact_launches": (c_int, [_P]),
    "tgvkv_evict": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                            c_double, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                            c_void_p, c_void_p, c_void_p, c_void_p]),
    "tgvkv_evict_with_stats": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_void_p, c_double, c_void_p, c_void_p, c_void_p,
                                       c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_void_p, c_void_p]),
    "tgvkv_prefill": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                              c_void_p, c_void_p, c_void_p, c_void_p]),
    "tgvkv_workspace_init": (c_int, [_P, c_void_p, c_void_p]),
    "tgvkv_status": (c_int, [c_void_p, c_void_p]),
    "tgvkv_evict_launches": (c_int, [_P]),
    "tgvkv_decode": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_int64, c_void_p, c_void_p,
                             c_void_p, c_void_p]),
    "tgvkv_decode_launches": (c_int, [_P]),
    "tgvkv_check_wait_timeout": (c_int, [c_void_p, c_void_p]),
    "tgvkv_last_error": (c_char_p, []),
    "tgvkv_score_noalloc": (c_int, [_P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                    c_void_p, c_void_p, c_void_p]),
    "tgvkv_noalloc_status": (c_int, [c_void_p]),
}

_lib = None


def load() -> ctypes.CDLL:
    """The loaded library; raises if it was not built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with "
                "`python -c 'import __graft_entry__ as g; g.build()'` (nvcc, sm_103a). "
                "There is no CPU fallback.")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib
