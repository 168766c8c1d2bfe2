"""tgvkv_score_noalloc: the scoring call for callers that cannot allocate.

Some callers receive only input and output buffers -- for example an operator
plugged into an inference runtime that owns all device memory and hands its
operators no workspace -- so they cannot provide tgvkv_score's workspace.
tgvkv_score_noalloc keeps that scratch in a fixed array inside the library.
This test calls it through the C ABI twice in a row and compares both results
with tgvkv_score's and with the fp64 oracle's Eq. 8 scores and Eq. 5 statistic
(same tolerance as the other parity tests), reading the call's status word
after each call, on a layout with several query-row tiles per KV head so that
the shared counters and partial scores in the fixed array are exercised, and
checks that an oversized problem is refused before any launch.  The file runs last so that a failure here
leaves the rest of the suite already run.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2606_03075_gb300 import synth

import _parity as P

pytestmark = pytest.mark.gpu


def _vp(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("wl", [
    synth.WORKLOADS["tiny"],
    synth.custom("noalloc_gqa", 2, 12, 2, 128,
                 [("text", 5), ("vision", 100), ("text", 9), ("vision", 77), ("text", 30)],
                 window="all_text", weights="dirichlet"),
], ids=["tiny", "gqa_3_row_tiles"])
def test_noalloc_matches_workspace_call(wl):
    assert torch.cuda.is_available()
    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import _lib, api
    lib = _lib.load()

    inp = synth.generate(wl, seed=7)
    dev = P.device_inputs(inp)
    desc = api.desc_for_workload(wl)
    stream = torch.cuda.current_stream()

    ws = api.new_workspace(desc)
    ref_s = torch.empty((wl.L, wl.H_kv, wl.N_v), dtype=torch.float32, device="cuda")
    ref_t = torch.empty(wl.L, dtype=torch.float32, device="cuda")
    api.tgvkv_score(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], dev["w"],
                    ref_s, ref_t, ws)
    assert api.tgvkv_status(ws) == 0
    # the oracle's Eq. 8 scores and Eq. 5 statistic on the same inputs
    o_s, o_t = oracle.twr_scores_tvb_stat(
        oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"]), inp["modality"],
        inp["text_pos"], np.asarray(inp["w"], np.float64), 1.0 / math.sqrt(wl.d), wl.H_kv)

    for call in range(2):
        s = torch.full((wl.L, wl.H_kv, wl.N_v), float("nan"), dtype=torch.float32, device="cuda")
        t = torch.full((wl.L,), float("nan"), dtype=torch.float32, device="cuda")
        rc = lib.tgvkv_score_noalloc(ctypes.byref(desc), _vp(dev["q"]), _vp(dev["k"]),
                                     _vp(dev["modality"]), _vp(dev["text_pos"]), _vp(dev["w"]),
                                     _vp(s), _vp(t), ctypes.c_void_p(stream.cuda_stream))
        assert rc == 0, lib.tgvkv_last_error()
        assert lib.tgvkv_noalloc_status(ctypes.c_void_p(stream.cuda_stream)) == 0
        P.assert_close(s.cpu().numpy(), ref_s.cpu().numpy(), f"scores, call {call}")
        P.assert_close(t.cpu().numpy(), ref_t.cpu().numpy(), f"tvb_stat, call {call}")
        P.assert_close(s.cpu().numpy(), o_s, f"scores vs oracle, call {call}")
        P.assert_close(t.cpu().numpy(), o_t, f"tvb_stat vs oracle, call {call}")


def test_noalloc_rejects_oversized_problem():
    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import _lib, api
    lib = _lib.load()
    wl = synth.WORKLOADS["video"]          # needs ~100 MB of scratch
    desc = api.desc_for_workload(wl)
    assert api.tgvkv_workspace_size(desc) > 8 << 20
    fake = ctypes.c_void_p(0x1000)         # never dereferenced: the call is refused first
    rc = lib.tgvkv_score_noalloc(ctypes.byref(desc), fake, fake, fake, fake, fake, fake, fake,
                                 None)
    assert rc == 2
    assert b"static scratch" in lib.tgvkv_last_error()
