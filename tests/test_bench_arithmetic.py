"""The bench's roofline arithmetic (CPU): algorithmic bytes, FLOPs and
exponential counts of a step, against values derived by hand from the
workload shapes and, for the counts, from a direct loop over (row, key) pairs."""
import numpy as np

import bench
from paper_2606_03075_gb300 import synth


def test_llava15_step_bytes_by_hand():
    wl = synth.WORKLOADS["llava15"]
    # K read once: 32 layers x 32 KV heads x 675 keys x 128 dims x 2 bytes
    k_read = 32 * 32 * 675 * 128 * 2
    # kept rows per KV head over all layers: every text row (99 per layer) plus
    # B_V = floor(0.05 * 576 * 32 + 1/2) = 922 vision rows
    assert bench.budget_total(wl, 0.05) == 922
    rows = 32 * (32 * 99 + 922)
    written = 2 * rows * 128 * 2
    assert bench.step_bytes(wl, 0.05) == (k_read + written, rows)
    q_read = 32 * 32 * 64 * 128 * 2
    scores = 32 * 32 * 576 * 4
    full = k_read + q_read + 2 * scores + 4 * rows * 128 * 2 + 4 * rows + 8 * (32 * 32 + 1)
    assert bench.full_step_bytes(wl, 0.05) == full
    sb = bench.stage_bytes(wl, 0.05)
    assert sb["score"] == k_read + q_read + scores


def test_score_flops_and_exponentials_by_counting_pairs():
    wl = synth.custom("count", 2, 6, 2, 64, [("text", 5), ("vision", 40), ("text", 3),
                                             ("vision", 20), ("text", 7)], window="all_text")
    pos = wl.text_pos
    vision = wl.modality == 1
    visible = sum(p + 1 for p in pos)
    visible_vision = sum(int(vision[:p + 1].sum()) for p in pos)
    assert bench.score_flops(wl) == 2 * wl.d * wl.L * wl.H_q * visible
    assert bench.score_exps(wl) == wl.L * wl.H_q * (visible + visible_vision)
    assert np.all(np.diff(pos) > 0)


def test_clock_rule_rejects_slowdowns_and_stuck_clocks():
    """The timing rule on clocks: a hardware or thermal slowdown, or a median
    SM clock well below the maximum with no reason given, disqualifies a timed
    region; the power cap alone does not, nor does a missing NVML."""
    ok = dict(sm_mhz=2070, sm_max_mhz=2070, reasons=[])
    assert not bench.clocks_rejected(ok)
    assert not bench.clocks_rejected(dict(ok, sm_mhz=1800, reasons=["sw_power_cap"]))
    assert not bench.clocks_rejected(dict(ok, sm_mhz=1200, reasons=["sw_power_cap"]))
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert bench.clocks_rejected(dict(ok, reasons=[r]))
        assert bench.clocks_rejected(dict(ok, reasons=["sw_power_cap", r]))
    assert bench.clocks_rejected(dict(ok, sm_mhz=1500))          # locked low, no reason
    assert not bench.clocks_rejected(dict(ok, sm_mhz=1700))      # 82% of the maximum
    assert not bench.clocks_rejected(dict(sm_mhz=None, sm_max_mhz=None, reasons=[]))


def test_traffic_hash_covers_every_included_kernel_header():
    """A recorded ncu traffic figure stays valid only while the kernel's source
    is unchanged: each kernel's hash list must hold its .cu file and every
    kernel header it includes, directly or through another header (launch.h
    declares host launchers only)."""
    import os
    import re
    csrc = os.path.join(os.path.dirname(bench.__file__), "paper_2606_03075_gb300", "csrc")

    def local_includes(name, seen):
        for inc in re.findall(r'#include "([^"]+)"', open(os.path.join(csrc, name)).read()):
            if inc not in seen and os.path.exists(os.path.join(csrc, inc)):
                seen.add(inc)
                local_includes(inc, seen)
        return seen

    for stage, files in bench.KERNEL_SOURCES.items():
        for cu in (f for f in files if f.endswith(".cu")):
            missing = local_includes(cu, set()) - set(files) - {"launch.h"}
            assert not missing, (stage, cu, missing)


def test_roof_and_mufu_rate_by_hand():
    """One layer, two query heads on one KV head, d = 64, 10 text + 100 vision +
    18 text tokens with the last 18 (positions 110..127) as query rows.
    Score launch bytes: K 128*64*2 = 16384, Q 2*18*64*2 = 4608, scores 100*4 =
    400: 21392.  FLOPs: 2*64*2 * sum_{p=110..127}(p+1) = 256 * 2151 = 550656.
    At 1000 GB/s and 1 TFLOP/s the FLOPs take longer (550.656 ns > 21.392 ns):
    tensor-bound.  Exponentials: 2 heads * (2151 + 18*100) = 7902."""
    import pytest
    wl = synth.custom("hand", 1, 2, 1, 64, [("text", 10), ("vision", 100), ("text", 18)])
    assert wl.text_pos.tolist() == list(range(110, 128))
    peaks = {"hbm_gbs": 1000.0, "bf16_tflops": 1.0}
    r = bench.kernel_roof(wl, 0.5, "score", 1.0, peaks)
    assert r["bytes_per_launch"] == 21392 and r["flops_per_launch"] == 550656
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and r["peak"] == 1.0
    assert r["achieved"] == pytest.approx(550656 / 1e-3 / 1e12)
    assert r["frac"] == pytest.approx(550656 / 1e-3 / 1e12 / 1.0)
    assert r["frac_nominal"] == pytest.approx(550656 / 1e-3 / 1e12 / 2250.0)
    # a much slower tensor peak keeps it tensor-bound; a much faster one makes
    # the bytes bind: 550656 / 1e15 s < 21392 / 1e12 s
    r = bench.kernel_roof(wl, 0.5, "score", 2.0, {"hbm_gbs": 1000.0, "bf16_tflops": 1000.0})
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 1000.0
    assert r["achieved"] == pytest.approx(21392 / 2e-3 / 1e9)
    assert r["frac"] == pytest.approx(21392 / 2e-3 / 1e9 / 1000.0)
    assert r["frac_nominal"] == pytest.approx(21392 / 2e-3 / 1e9 / 7900.0)
    # the fused tail has no FLOPs: HBM-bound on its bytes (scores read, kept
    # rows read and written, idx, offsets); r = 0.5 keeps 18 + 10 text rows and
    # B_V = floor(0.5 * 100 + 1/2) = 50 vision rows: 78 rows
    tail = 400 + 4 * 78 * 64 * 2 + 4 * 78 + 8 * 2
    assert bench.stage_bytes(wl, 0.5)["tail"] == tail
    r = bench.kernel_roof(wl, 0.5, "tail", 1.0, peaks)
    assert r["bound"] == "hbm" and r["flops_per_launch"] == 0 and r["bytes_per_launch"] == tail
    m = bench.mufu_of(wl, 1.0, 2000.0)
    assert m["exps_per_launch"] == 7902
    assert m["peak_G_per_s"] == pytest.approx(32 * 152 * 2000e6 / 1e9)
    assert m["achieved_G_per_s"] == pytest.approx(7902 / 1e-3 / 1e9)
    assert m["frac"] == pytest.approx(7902 / 1e-3 / 1e9 / (32 * 152 * 2.0))


def test_stage_bytes_rounding_and_boundaries_by_hand():
    """The same hand workload: every launch's algorithmic bytes, the budget
    total's rounding (exact rationals), the roof choice just either side of the
    point where bytes and FLOPs take equal time, rates at launch times other
    than 1 ms, and the clock rule exactly at 80% of the maximum."""
    import math as _m
    from fractions import Fraction
    import pytest
    wl = synth.custom("hand", 1, 2, 1, 64, [("text", 10), ("vision", 100), ("text", 18)])
    sb = bench.stage_bytes(wl, 0.5)
    rows = 78                                   # 28 text + 50 vision rows, one KV head
    assert bench.step_bytes(wl, 0.5) == (16384 + 2 * rows * 64 * 2, rows)
    assert sb["budget"] == 8                    # one fp32 statistic read, one int32 budget written
    assert sb["select"] == 400 + 4 * rows + 8 * 2          # scores, idx, offsets
    assert sb["compact"] == 4 * rows * 64 * 2 + 4 * rows   # kept K/V read + written, idx read
    assert sb["tail"] == 400 + 4 * rows * 64 * 2 + 4 * rows + 8 * 2
    for r, nv, L in [(0.25, 6, 1), (0.25, 5, 1), (0.25, 7, 1), (0.125, 4, 1), (0.375, 2, 1)]:
        w2 = synth.custom("r", L, 1, 1, 64, [("text", 1), ("vision", nv)])
        assert bench.budget_total(w2, r) == _m.floor(Fraction(r) * nv * L + Fraction(1, 2))
    # bytes take 21392 / 1e12 s = 21.392 ns at 1000 GB/s; the FLOPs take
    # 550656 / (T * 1e12) s: 22.03 ns at T = 25 (tensor-bound), 20.78 ns at 26.5
    assert bench.kernel_roof(wl, 0.5, "score", 0.25, {"hbm_gbs": 1000.0,
                                                      "bf16_tflops": 25.0})["bound"] == "tensor"
    r = bench.kernel_roof(wl, 0.5, "score", 0.25, {"hbm_gbs": 1000.0, "bf16_tflops": 26.5})
    assert r["bound"] == "hbm"
    assert r["achieved"] == pytest.approx(21392 / 0.25e-3 / 1e9)
    r = bench.kernel_roof(wl, 0.5, "score", 0.25, {"hbm_gbs": 1000.0, "bf16_tflops": 25.0})
    assert r["achieved"] == pytest.approx(550656 / 0.25e-3 / 1e12)
    m = bench.mufu_of(wl, 0.5, 1000.0)
    assert m["achieved_G_per_s"] == pytest.approx(7902 / 0.5e-3 / 1e9)
    assert m["peak_G_per_s"] == pytest.approx(32 * 152 * 1.0)
    # exactly 80% of the maximum is not "below 80%"
    assert not bench.clocks_rejected(dict(sm_mhz=1656.0, sm_max_mhz=2070, reasons=[]))
    assert bench.clocks_rejected(dict(sm_mhz=1655.0, sm_max_mhz=2070, reasons=[]))


def test_stage_bytes_two_layers_two_kv_heads_by_hand():
    """L = 2, H_kv = 2 (G = 2), 10 + 100 + 18 tokens, r = 0.5: B_V = floor(0.5 *
    100 * 2 + 1/2) = 100, rows = 2 * (2 * 28 + 100) = 312, scores 2*2*100*4 =
    1600 bytes, offsets 8 * (2*2 + 1) = 40 bytes."""
    wl = synth.custom("hand2", 2, 4, 2, 64, [("text", 10), ("vision", 100), ("text", 18)])
    sb = bench.stage_bytes(wl, 0.5)
    assert bench.step_bytes(wl, 0.5)[1] == 312
    assert sb["score"] == 2 * 2 * 128 * 64 * 2 + 2 * 4 * 18 * 64 * 2 + 1600
    assert sb["budget"] == 16
    assert sb["select"] == 1600 + 4 * 312 + 40
    assert sb["compact"] == 4 * 312 * 64 * 2 + 4 * 312
    assert sb["tail"] == 1600 + 4 * 312 * 64 * 2 + 4 * 312 + 40
