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
