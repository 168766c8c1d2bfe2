"""Python binding of the TGV-KV C ABI (include/tgvkv.h).

Argument marshalling only: each function checks that the torch tensors have
the dtype, device, contiguity and size the C call expects, passes their device
pointers and the current CUDA stream, and raises on a non-zero return code.
Every step of the computation runs in the library's CUDA kernels.  PyTorch
provides device memory and streams.
"""
from __future__ import annotations

import ctypes
import math
from dataclasses import dataclass

import torch

from . import _lib

Desc = _lib.Desc

_BF16_LIKE = (torch.bfloat16, torch.int16, torch.uint16)


class TgvkvError(RuntimeError):
    def __init__(self, code, fn):
        msg = _lib.load().tgvkv_last_error().decode()
        super().__init__(f"{fn} failed with code {code}: {msg}")
        self.code = code


BASIS = {"vision": _lib.BASIS_VISION, "all": _lib.BASIS_ALL}
WEIGHTS = {"given": _lib.WEIGHTS_GIVEN, "eq7": _lib.WEIGHTS_EQ7}
STAT = {"tv": _lib.STAT_TV, "tt": _lib.STAT_TT, "uniform": _lib.STAT_UNIFORM}


def make_desc(L, H_q, H_kv, d, N, N_v, n_win, softmax_scale=0.0, w_layer_stride=None,
              basis="vision", weights="given", keep_first=0, keep_last=0, stat="tv",
              head_budgets=False) -> Desc:
    """A problem descriptor; w_layer_stride defaults to n_win (one weight row per layer).

    basis: "vision" (r counts vision KV, every text KV kept) or "all" (r counts
    every KV, both cases of Eq. 10); weights: "given" (the caller's w~) or
    "eq7" (tgvkv_evict derives w~ by Eq. 7); keep_first / keep_last: sinks;
    stat: the statistic the layer budgets follow, "tv" / "tt" / "uniform";
    head_budgets: one budget per (layer, KV head) (tvb_stat and budgets then
    hold L * H_kv entries)."""
    return Desc(L=L, H_q=H_q, H_kv=H_kv, d=d, N=N, N_v=N_v, n_win=n_win,
                softmax_scale=float(softmax_scale),
                w_layer_stride=n_win if w_layer_stride is None else w_layer_stride,
                budget_basis=BASIS[basis], weight_mode=WEIGHTS[weights],
                keep_first=keep_first, keep_last=keep_last, budget_stat=STAT[stat],
                head_budgets=int(bool(head_budgets)))


def budget_units(desc: Desc) -> int:
    """Entries of tvb_stat and budgets: L, or L * H_kv with head budgets."""
    return desc.L * desc.H_kv if desc.head_budgets else desc.L


def desc_for_workload(wl, softmax_scale=0.0, **options) -> Desc:
    return make_desc(wl.L, wl.H_q, wl.H_kv, wl.d, wl.N, wl.N_v, wl.n_win, softmax_scale,
                     **options)


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _ptr(t, dtypes, numel, name):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype not in dtypes:
        raise TypeError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, needs {numel}")
    return ctypes.c_void_p(t.data_ptr())


def _check(code, fn):
    if code != 0:
        raise TgvkvError(code, fn)


def tgvkv_workspace_size(desc: Desc) -> int:
    n = _lib.load().tgvkv_workspace_size(ctypes.byref(desc))
    if n == 0:
        raise TgvkvError(-1, "tgvkv_workspace_size")
    return int(n)


def tgvkv_vision_budget_total(desc: Desc, ratio: float) -> int:
    n = _lib.load().tgvkv_vision_budget_total(ctypes.byref(desc), float(ratio))
    if n < 0:
        raise TgvkvError(-1, "tgvkv_vision_budget_total")
    return int(n)


def tgvkv_budget_total(desc: Desc, ratio: float) -> int:
    n = _lib.load().tgvkv_budget_total(ctypes.byref(desc), float(ratio))
    if n < 0:
        raise TgvkvError(-1, "tgvkv_budget_total")
    return int(n)


def tgvkv_retained_rows(desc: Desc, ratio: float) -> int:
    n = _lib.load().tgvkv_retained_rows(ctypes.byref(desc), float(ratio))
    if n < 0:
        raise TgvkvError(-1, "tgvkv_retained_rows")
    return int(n)


def tgvkv_workspace_init(desc: Desc, ws: torch.Tensor, stream=None):
    p = _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace")
    _check(_lib.load().tgvkv_workspace_init(ctypes.byref(desc), p, _stream(stream)),
           "tgvkv_workspace_init")


def new_workspace(desc: Desc, device=None) -> torch.Tensor:
    """A zeroed workspace tensor (uint8) for this problem."""
    ws = torch.empty(tgvkv_workspace_size(desc), dtype=torch.uint8, device=device or "cuda")
    tgvkv_workspace_init(desc, ws)
    return ws


def tgvkv_score(desc, q_text, k, modality, text_pos, w, scores, tvb_stat, ws, stream=None):
    L, Hq, Hkv, d, N, Nv, nw = desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.N_v, desc.n_win
    wrows = (L - 1) * desc.w_layer_stride + nw if nw else 0
    _check(_lib.load().tgvkv_score(
        ctypes.byref(desc),
        _ptr(q_text, _BF16_LIKE, L * Hq * nw * d, "q_text"),
        _ptr(k, _BF16_LIKE, L * Hkv * N * d, "k"),
        _ptr(modality, (torch.uint8,), N, "modality"),
        _ptr(text_pos, (torch.int32,), nw, "text_pos"),
        _ptr(w, (torch.float32,), wrows, "w"),
        _ptr(scores, (torch.float32,), L * Hkv * Nv, "scores"),
        _ptr(tvb_stat, (torch.float32,), budget_units(desc), "tvb_stat"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_score")


def tgvkv_text_scores(desc, q_text, k, modality, text_pos, text_scores, weights, ws, stream=None):
    L, Hq, Hkv, d, N, nw = desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.n_win
    _check(_lib.load().tgvkv_text_scores(
        ctypes.byref(desc),
        _ptr(q_text, _BF16_LIKE, L * Hq * nw * d, "q_text"),
        _ptr(k, _BF16_LIKE, L * Hkv * N * d, "k"),
        _ptr(modality, (torch.uint8,), N, "modality"),
        _ptr(text_pos, (torch.int32,), nw, "text_pos"),
        _ptr(text_scores, (torch.float32,), L * Hkv * (N - desc.N_v), "text_scores"),
        _ptr(weights, (torch.float32,), L * nw, "weights"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_text_scores")


def tgvkv_budget(desc, tvb_stat, ratio, budgets, ws, stream=None):
    _check(_lib.load().tgvkv_budget(
        ctypes.byref(desc),
        _ptr(tvb_stat, (torch.float32,), budget_units(desc), "tvb_stat"), float(ratio),
        _ptr(budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_budget")


def tgvkv_select(desc, scores, budgets, modality, offsets, idx, ws, stream=None):
    LH = desc.L * desc.H_kv
    _check(_lib.load().tgvkv_select(
        ctypes.byref(desc),
        _ptr(scores, (torch.float32,), LH * desc.N_v, "scores"),
        _ptr(budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(modality, (torch.uint8,), desc.N, "modality"),
        _ptr(offsets, (torch.int64,), LH + 1, "offsets"),
        _ptr(idx, (torch.int32,), 0, "idx"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_select")


def tgvkv_select_tpr(desc, scores, text_scores, budgets, modality, offsets, idx, ws, stream=None):
    LH = desc.L * desc.H_kv
    _check(_lib.load().tgvkv_select_tpr(
        ctypes.byref(desc),
        _ptr(scores, (torch.float32,), LH * desc.N_v, "scores"),
        _ptr(text_scores, (torch.float32,), LH * (desc.N - desc.N_v), "text_scores"),
        _ptr(budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(modality, (torch.uint8,), desc.N, "modality"),
        _ptr(offsets, (torch.int64,), LH + 1, "offsets"),
        _ptr(idx, (torch.int32,), 0, "idx"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_select_tpr")


def tgvkv_compact(desc, k, v, offsets, idx, k_out, v_out, ws, stream=None):
    n = desc.L * desc.H_kv * desc.N * desc.d
    capacity = min(k_out.numel(), v_out.numel()) // desc.d   # rows of the outputs
    _check(_lib.load().tgvkv_compact(
        ctypes.byref(desc),
        _ptr(k, _BF16_LIKE, n, "k"), _ptr(v, _BF16_LIKE, n, "v"),
        _ptr(offsets, (torch.int64,), desc.L * desc.H_kv + 1, "offsets"),
        _ptr(idx, (torch.int32,), 0, "idx"),
        _ptr(k_out, _BF16_LIKE, 0, "k_out"), _ptr(v_out, _BF16_LIKE, 0, "v_out"),
        capacity,
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_compact")


def tgvkv_select_compact(desc, scores, text_scores, budgets, modality, k, v, offsets, idx,
                         k_out, v_out, ws, stream=None):
    LH = desc.L * desc.H_kv
    n = LH * desc.N * desc.d
    # rows every output holds: k_out, v_out and idx alike
    capacity = min(k_out.numel() // desc.d, v_out.numel() // desc.d, idx.numel())
    _check(_lib.load().tgvkv_select_compact(
        ctypes.byref(desc),
        _ptr(scores, (torch.float32,), LH * desc.N_v, "scores"),
        _ptr(text_scores, (torch.float32,), LH * (desc.N - desc.N_v), "text_scores"),
        _ptr(budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(modality, (torch.uint8,), desc.N, "modality"),
        _ptr(k, _BF16_LIKE, n, "k"), _ptr(v, _BF16_LIKE, n, "v"),
        _ptr(offsets, (torch.int64,), LH + 1, "offsets"),
        _ptr(idx, (torch.int32,), 0, "idx"),
        _ptr(k_out, _BF16_LIKE, 0, "k_out"), _ptr(v_out, _BF16_LIKE, 0, "v_out"),
        capacity,
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_select_compact")


def tgvkv_select_compact_launches(desc: Desc) -> int:
    return int(_lib.load().tgvkv_select_compact_launches(ctypes.byref(desc)))


@dataclass
class EvictOutputs:
    scores: torch.Tensor     # fp32 [L, H_kv, N_v]
    tvb_stat: torch.Tensor   # fp32 [L]
    budgets: torch.Tensor    # int32 [L]
    offsets: torch.Tensor    # int64 [L*H_kv + 1]
    idx: torch.Tensor        # int32 [retained rows]
    k_out: torch.Tensor      # bf16 [retained rows, d]
    v_out: torch.Tensor      # bf16 [retained rows, d]


def alloc_outputs(desc: Desc, ratio: float, device=None) -> EvictOutputs:
    dev = device or "cuda"
    rows = tgvkv_retained_rows(desc, ratio)
    L, Hkv = desc.L, desc.H_kv
    return EvictOutputs(
        scores=torch.empty((L, Hkv, desc.N_v), dtype=torch.float32, device=dev),
        tvb_stat=torch.empty(budget_units(desc), dtype=torch.float32, device=dev),
        budgets=torch.empty(budget_units(desc), dtype=torch.int32, device=dev),
        offsets=torch.empty(L * Hkv + 1, dtype=torch.int64, device=dev),
        idx=torch.empty(max(rows, 1), dtype=torch.int32, device=dev),
        k_out=torch.empty((max(rows, 1), desc.d), dtype=torch.bfloat16, device=dev),
        v_out=torch.empty((max(rows, 1), desc.d), dtype=torch.bfloat16, device=dev))


def tgvkv_evict(desc, q_text, k, v, modality, text_pos, w, ratio, out: EvictOutputs, ws,
                stream=None):
    L, Hq, Hkv, d, N, Nv, nw = desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.N_v, desc.n_win
    rows = tgvkv_retained_rows(desc, ratio)
    wrows = (L - 1) * desc.w_layer_stride + nw if nw else 0
    _check(_lib.load().tgvkv_evict(
        ctypes.byref(desc),
        _ptr(q_text, _BF16_LIKE, L * Hq * nw * d, "q_text"),
        _ptr(k, _BF16_LIKE, L * Hkv * N * d, "k"),
        _ptr(v, _BF16_LIKE, L * Hkv * N * d, "v"),
        _ptr(modality, (torch.uint8,), N, "modality"),
        _ptr(text_pos, (torch.int32,), nw, "text_pos"),
        _ptr(w, (torch.float32,), wrows, "w"),
        float(ratio),
        _ptr(out.scores, (torch.float32,), L * Hkv * Nv, "scores"),
        _ptr(out.tvb_stat, (torch.float32,), budget_units(desc), "tvb_stat"),
        _ptr(out.budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(out.offsets, (torch.int64,), L * Hkv + 1, "offsets"),
        _ptr(out.idx, (torch.int32,), rows, "idx"),
        _ptr(out.k_out, _BF16_LIKE, rows * d, "k_out"),
        _ptr(out.v_out, _BF16_LIKE, rows * d, "v_out"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_evict")


def tgvkv_evict_with_stats(desc, q_text, k, v, modality, text_pos, w, ratio, row_stats,
                           out: EvictOutputs, ws, stream=None):
    """tgvkv_evict with the query rows' (m, Z, vision mass) from tgvkv_prefill."""
    L, Hq, Hkv, d, N, Nv, nw = desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.N_v, desc.n_win
    rows = tgvkv_retained_rows(desc, ratio)
    wrows = (L - 1) * desc.w_layer_stride + nw if nw else 0
    _check(_lib.load().tgvkv_evict_with_stats(
        ctypes.byref(desc),
        _ptr(q_text, _BF16_LIKE, L * Hq * nw * d, "q_text"),
        _ptr(k, _BF16_LIKE, L * Hkv * N * d, "k"),
        _ptr(v, _BF16_LIKE, L * Hkv * N * d, "v"),
        _ptr(modality, (torch.uint8,), N, "modality"),
        _ptr(text_pos, (torch.int32,), nw, "text_pos"),
        _ptr(w, (torch.float32,), wrows, "w"),
        float(ratio),
        _ptr(row_stats, (torch.float32,), 3 * L * Hq * nw, "row_stats"),
        _ptr(out.scores, (torch.float32,), L * Hkv * Nv, "scores"),
        _ptr(out.tvb_stat, (torch.float32,), budget_units(desc), "tvb_stat"),
        _ptr(out.budgets, (torch.int32,), budget_units(desc), "budgets"),
        _ptr(out.offsets, (torch.int64,), L * Hkv + 1, "offsets"),
        _ptr(out.idx, (torch.int32,), rows, "idx"),
        _ptr(out.k_out, _BF16_LIKE, rows * d, "k_out"),
        _ptr(out.v_out, _BF16_LIKE, rows * d, "v_out"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_evict_with_stats")


def tgvkv_prefill(desc, q, k, v, modality, text_pos, o, q_text, row_stats, ws, stream=None):
    """Causal prefill attention over every token, plus the eviction step's query
    rows (q_text) and their (m, Z, vision mass) (see include/tgvkv.h)."""
    L, Hq, Hkv, d, N, nw = desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.n_win
    _check(_lib.load().tgvkv_prefill(
        ctypes.byref(desc),
        _ptr(q, _BF16_LIKE, L * Hq * N * d, "q"),
        _ptr(k, _BF16_LIKE, L * Hkv * N * d, "k"),
        _ptr(v, _BF16_LIKE, L * Hkv * N * d, "v"),
        _ptr(modality, (torch.uint8,), N, "modality"),
        _ptr(text_pos, (torch.int32,), nw, "text_pos"),
        _ptr(o, _BF16_LIKE, L * Hq * N * d, "o"),
        _ptr(q_text, _BF16_LIKE, L * Hq * nw * d, "q_text"),
        _ptr(row_stats, (torch.float32,), 3 * L * Hq * nw, "row_stats"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_prefill")


def tgvkv_check_wait_timeout(ws: torch.Tensor, stream=None):
    """Launch the failure-detection self-test: a bounded wait that runs out and
    sets TGVKV_STATUS_TIMEOUT in the workspace's status word."""
    _check(_lib.load().tgvkv_check_wait_timeout(_ptr(ws, (torch.uint8,), 4, "workspace"),
                                                _stream(stream)), "tgvkv_check_wait_timeout")


def tgvkv_status(ws: torch.Tensor, stream=None) -> int:
    """Synchronise the stream, return and clear the device status bits."""
    rc = _lib.load().tgvkv_status(_ptr(ws, (torch.uint8,), 4, "workspace"), _stream(stream))
    if rc < 0:
        raise TgvkvError(-rc, "tgvkv_status")
    return rc


def tgvkv_decode(desc, q, k_rows, v_rows, offsets, out, ws, stream=None):
    """One decode step of every layer over a CSR cache (see include/tgvkv.h)."""
    L, Hq, Hkv, d = desc.L, desc.H_q, desc.H_kv, desc.d
    capacity = min(k_rows.numel(), v_rows.numel()) // d
    _check(_lib.load().tgvkv_decode(
        ctypes.byref(desc),
        _ptr(q, _BF16_LIKE, L * Hq * d, "q"),
        _ptr(k_rows, _BF16_LIKE, 0, "k_rows"),
        _ptr(v_rows, _BF16_LIKE, 0, "v_rows"),
        capacity,
        _ptr(offsets, (torch.int64,), L * Hkv + 1, "offsets"),
        _ptr(out, (torch.float32,), L * Hq * d, "out"),
        _ptr(ws, (torch.uint8,), tgvkv_workspace_size(desc), "workspace"),
        _stream(stream)), "tgvkv_decode")


def tgvkv_decode_launches(desc: Desc) -> int:
    return int(_lib.load().tgvkv_decode_launches(ctypes.byref(desc)))


def tgvkv_evict_launches(desc: Desc) -> int:
    """Kernels one tgvkv_evict call launches for this problem."""
    n = _lib.load().tgvkv_evict_launches(ctypes.byref(desc))
    if n < 0:
        raise TgvkvError(-1, "tgvkv_evict_launches")
    return int(n)


def default_scale(d: int) -> float:
    return 1.0 / math.sqrt(d)
