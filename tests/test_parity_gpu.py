"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Small cases (several row and key tiles, ragged tails, grouped-query heads,
interleaved text, d = 64 and 128, edge cases) are checked in full; the four
model-shaped workloads at their full sizes are checked on sampled layers, with
the launch configuration the benchmark times.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2606_03075_gb300 import synth

import _parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def api():
    assert torch.cuda.is_available(), "the GPU tests need a CUDA device"
    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import api as _api
    return _api


def _seg_video(frames, stamp, per_frame, head, tail):
    s = [("text", head)]
    for _ in range(frames):
        s += [("text", stamp), ("vision", per_frame)]
    return s + [("text", tail)]


SMALL = {
    "ragged_mha": synth.custom("ragged_mha", 3, 4, 4, 128,
                               [("text", 13), ("vision", 150), ("text", 7), ("vision", 61),
                                ("text", 40)], ratios=(0.05, 0.3)),
    "ragged_gqa": synth.custom("ragged_gqa", 2, 12, 2, 128,
                               [("text", 5), ("vision", 100), ("text", 9), ("vision", 77),
                                ("text", 30)], window="all_text", weights="dirichlet",
                               ratios=(0.1,)),
    "d64_gqa": synth.custom("d64_gqa", 2, 8, 4, 64,
                            [("text", 20), ("vision", 180), ("text", 70)], ratios=(0.2,)),
    "video_small": synth.custom("video_small", 2, 4, 1, 128, _seg_video(8, 4, 40, 8, 16),
                                window="all_text", weights="dirichlet", ratios=(0.05,)),
    "wide_group": synth.custom("wide_group", 1, 32, 1, 128,
                               [("text", 3), ("vision", 90), ("text", 9)], ratios=(0.5,)),
}


# Heads of one row tile with 64 < G * n_win <= 128 (the score kernel's
# single-tile items) at several lengths, row counts, causal layouts and head
# dims.
ONE_TILE = {
    # grouped-query heads (G = 2, 96 rows)
    "gqa_96": synth.custom("gqa_96", 2, 8, 4, 128,
                            [("text", 11), ("vision", 400), ("text", 6), ("vision", 50),
                             ("text", 48)], ratios=(0.1,)),
    # 80 rows; vision keys after the last query row (scores 0)
    "r80_tail": synth.custom("r80_tail", 3, 4, 4, 128,
                                 [("text", 10), ("vision", 700), ("text", 80), ("vision", 300)],
                                 window=80, ratios=(0.2,)),
    # 112 rows (G = 7), Dirichlet weights, ragged N
    "r112_dirichlet": synth.custom("r112_dirichlet", 2, 14, 2, 128,
                             [("text", 7), ("vision", 900), ("text", 5), ("vision", 611),
                              ("text", 16)], window=16, weights="dirichlet", ratios=(0.05,)),
    # 128 rows spread over the sequence (rows see different key prefixes)
    "r128_causal": synth.custom("r128_causal", 2, 2, 2, 128,
                                    [("text", 20), ("vision", 500), ("text", 40), ("vision", 500),
                                     ("text", 40), ("vision", 500), ("text", 48)], window=128,
                                    ratios=(0.1,)),
    # many heads (256) per launch
    "many_heads_96": synth.custom("many_heads_96", 8, 32, 32, 128,
                            [("text", 30), ("vision", 700), ("text", 96)], ratios=(0.1,)),
    # short heads
    "short_96": synth.custom("short_96", 2, 4, 4, 128,
                               [("text", 10), ("vision", 154), ("text", 96)], ratios=(0.25,)),
    # 128 rows, long heads, ragged N
    "long_r128": synth.custom("long_r128", 1, 4, 2, 128,
                             [("text", 17), ("vision", 2800), ("text", 64)], window=64,
                             ratios=(0.05,)),
    # one KV head in all
    "one_head_96": synth.custom("one_head_96", 1, 1, 1, 128,
                                [("text", 12), ("vision", 600), ("text", 96)], ratios=(0.1,)),
    # one key tile per head
    "one_key_tile_96": synth.custom("one_key_tile_96", 2, 2, 2, 128,
                                    [("text", 4), ("vision", 20), ("text", 96)], ratios=(0.25,)),
    # d = 64, an odd number of key tiles
    "d64_96": synth.custom("d64_96", 3, 4, 4, 64,
                           [("text", 9), ("vision", 500), ("text", 25), ("vision", 70),
                            ("text", 96)], ratios=(0.1,)),
}


def _full_check(api, wl, ratio, inp=None):
    inp = inp if inp is not None else synth.generate(wl, seed=0)
    g = P.run_evict(api, wl, inp, ratio)
    assert g["status"] == 0
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"],
                       inp["w"], ratio, wl.H_kv)
    P.assert_close(g["scores"], ref["scores"], "scores")
    P.assert_close(g["stat"], ref["stat"], "tvb_stat")
    # budgets: exact from the GPU statistic; end to end they agree unless a
    # quota sits within the statistic's tolerance of a rounding boundary
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    assert int(g["budgets"].sum()) == total
    if not np.array_equal(g["budgets"], ref["budgets"]):
        q = total * ref["stat"] / ref["stat"].sum()
        assert np.min(np.abs(q - np.round(q))) < 1e-2, (g["budgets"], ref["budgets"])
    P.check_selection_and_compaction(wl, inp, g, list(range(wl.L)),
                                     ref_scores=ref["scores"] if np.array_equal(
                                         g["budgets"], ref["budgets"]) else None)
    assert g["offsets"][-1] == wl.H_kv * (wl.L * wl.N_t + total)
    return g, ref


def test_tiny(api):
    _full_check(api, synth.WORKLOADS["tiny"], 0.25)


@pytest.mark.parametrize("name", sorted(SMALL))
def test_small_layouts(api, name):
    wl = SMALL[name]
    for r in wl.ratios:
        _full_check(api, wl, r)


def test_max_length_heads(api):
    """Heads of the largest length the library accepts (N = 32768): the score
    kernel's per-head tile tables at their full size, text before and after the
    vision span, G = 2, and the select + gather in its two-launch form (its
    shared-memory tables exceed the fused kernel's at this length)."""
    wl = synth.custom("max_len", 1, 4, 2, 128,
                      [("text", 40), ("vision", 32600), ("text", 128)], window=64,
                      ratios=(0.05,))
    assert wl.N == 32768
    assert api.tgvkv_evict_launches(api.desc_for_workload(wl)) == 3
    _full_check(api, wl, 0.05)


def test_max_layers(api):
    """The most layers the library accepts (L = 1024): the score kernel's
    closing CTA sums 1024 layer masses and splits the budgets with the whole
    block (more than one warp's worth of units), and the warp-per-head select
    + gather runs 1024 sets."""
    wl = synth.custom("max_layers", 1024, 2, 1, 64,
                      [("text", 8), ("vision", 120), ("text", 16)], window=16, ratios=(0.1,))
    assert api.tgvkv_evict_launches(api.desc_for_workload(wl)) == 2
    _full_check(api, wl, 0.1)


def test_max_query_rows(api):
    """The most query rows per KV head the library accepts (G * n_win = 32768,
    256 row tiles of one head): every row tile's partial scores summed into
    the head's."""
    wl = synth.custom("max_rows", 1, 256, 1, 64,
                      [("text", 64), ("vision", 256), ("text", 128)], window=128,
                      ratios=(0.2,))
    assert wl.H_q // wl.H_kv * wl.n_win == 32768
    _full_check(api, wl, 0.2)


@pytest.mark.parametrize("name", sorted(ONE_TILE))
def test_one_tile_layouts(api, name):
    """The whole step against the oracle, then the score call alone (scores
    and statistic within tolerance, no budgets) and a second evict call
    bit-identical to the first."""
    wl = ONE_TILE[name]
    inp = synth.generate(wl, seed=3)
    g, ref = _full_check(api, wl, wl.ratios[0], inp=inp)
    dev = P.device_inputs(inp)
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    s = torch.full((wl.L, wl.H_kv, wl.N_v), float("nan"), dtype=torch.float32, device="cuda")
    t = torch.full((wl.L,), float("nan"), dtype=torch.float32, device="cuda")
    api.tgvkv_score(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], dev["w"], s, t, ws)
    assert api.tgvkv_status(ws) == 0
    P.assert_close(s.cpu().numpy(), ref["scores"], f"{name} scores (tgvkv_score)")
    P.assert_close(t.cpu().numpy(), ref["stat"], f"{name} tvb_stat (tgvkv_score)")
    g2 = P.run_evict(api, wl, inp, wl.ratios[0], dev=dev)
    assert g2["status"] == 0
    for key in ("scores", "stat", "budgets", "offsets", "idx", "k_out", "v_out"):
        np.testing.assert_array_equal(g2[key], g[key], err_msg=key)


@pytest.mark.parametrize("ratio", [0.0, 1.0])
def test_budget_extremes(api, ratio):
    g, _ = _full_check(api, SMALL["ragged_mha"], ratio)
    assert set(g["budgets"].tolist()) == ({0} if ratio == 0.0 else {SMALL["ragged_mha"].N_v})


def test_no_vision_tokens(api):
    wl = synth.custom("no_vision", 2, 2, 2, 64, [("text", 50)], ratios=(0.5,))
    g, _ = _full_check(api, wl, 0.5)
    assert g["scores"].size == 0 and np.all(g["stat"] == 0)


def test_single_query_row(api):
    wl = synth.custom("one_row", 2, 4, 2, 128,
                      [("text", 7), ("vision", 130), ("text", 1)], ratios=(0.3,))
    assert wl.n_win == 1
    _full_check(api, wl, 0.3)


def test_queries_before_any_vision(api):
    """Query rows that precede every vision key: zero TV mass everywhere, so
    the budgets split uniformly and the kept vision keys are the lowest
    positions (all scores tie at zero)."""
    wl = synth.custom("early", 3, 4, 4, 64, [("text", 30), ("vision", 64), ("text", 10)],
                      window=10, ratios=(0.25,))
    inp = synth.generate(wl, seed=1)
    inp["text_pos"] = np.arange(10, dtype=np.int32) * 3
    g, ref = _full_check(api, wl, 0.25, inp=inp)
    assert np.all(g["stat"] == 0) and np.all(g["scores"] == 0)
    assert g["budgets"].tolist() == oracle.tvb_budgets([0, 0, 0], 48, 64)


# 512 (layer, KV head) pairs with 40 query rows each: packed score items (two
# heads per row tile) and the warp-per-head select/gather of the evict path
MANY = synth.custom("many_heads", 16, 32, 32, 64, [("text", 20), ("vision", 200), ("text", 40)],
                    ratios=(0.3,))


@pytest.mark.parametrize("ratio", [0.0, 0.3, 1.0])
def test_many_small_heads(api, ratio):
    g, _ = _full_check(api, MANY, ratio)
    if ratio in (0.0, 1.0):
        assert set(g["budgets"].tolist()) == ({0} if ratio == 0.0 else {MANY.N_v})


def test_many_small_heads_all_ties(api):
    """The warp-per-head selection when every vision score ties at zero: the
    kept vision keys must be the lowest positions of each head."""
    wl = synth.custom("many_early", 16, 32, 32, 64, [("text", 30), ("vision", 200), ("text", 10)],
                      window=10, ratios=(0.25,))
    inp = synth.generate(wl, seed=2)
    inp["text_pos"] = np.arange(10, dtype=np.int32) * 3
    g, _ = _full_check(api, wl, 0.25, inp=inp)
    assert np.all(g["stat"] == 0) and np.all(g["scores"] == 0)


def test_separate_calls_match_fused(api):
    wl = SMALL["ragged_gqa"]
    ratio = 0.1
    inp = synth.generate(wl, seed=3)
    dev = P.device_inputs(inp)
    fused = P.run_evict(api, wl, inp, ratio, dev=dev)
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    out = api.alloc_outputs(desc, ratio)
    api.tgvkv_score(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], dev["w"],
                    out.scores, out.tvb_stat, ws)
    api.tgvkv_budget(desc, out.tvb_stat, ratio, out.budgets, ws)
    api.tgvkv_select(desc, out.scores, out.budgets, dev["modality"], out.offsets, out.idx, ws)
    api.tgvkv_compact(desc, dev["k"], dev["v"], out.offsets, out.idx, out.k_out, out.v_out, ws)
    assert api.tgvkv_status(ws) == 0
    rows = api.tgvkv_retained_rows(desc, ratio)
    np.testing.assert_array_equal(out.scores.cpu().numpy(), fused["scores"])
    np.testing.assert_array_equal(out.tvb_stat.cpu().numpy(), fused["stat"])
    np.testing.assert_array_equal(out.idx[:rows].cpu().numpy(), fused["idx"])
    np.testing.assert_array_equal(out.k_out[:rows].view(torch.int16).cpu().numpy(), fused["k_out"])


def test_repeat_calls_are_deterministic(api):
    wl = SMALL["video_small"]
    inp = synth.generate(wl, seed=4)
    dev = P.device_inputs(inp)
    a = P.run_evict(api, wl, inp, 0.05, dev=dev)
    b = P.run_evict(api, wl, inp, 0.05, dev=dev)
    for key in ("scores", "stat", "budgets", "offsets", "idx", "k_out", "v_out"):
        np.testing.assert_array_equal(a[key], b[key], err_msg=key)


def test_back_to_back_launches_stay_clean(api):
    """Many score launches queued back to back (no host synchronisation between
    them) on the long interleaved-video shape, whose row-tile pairs have
    different causal ranges, so a group skips ring entries and the two MMA
    issuers hand accumulator buffers to each other.  Every launch must finish
    without a timed-out wait and reproduce the first launch bit for bit."""
    wl = synth.WORKLOADS["video"]
    inp = synth.generate(wl, seed=0)
    dev = P.device_inputs(inp)
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    out = api.alloc_outputs(desc, wl.ratios[0])
    args = (desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], dev["w"])
    api.tgvkv_score(*args, out.scores, out.tvb_stat, ws)
    assert api.tgvkv_status(ws) == 0
    first = (out.scores.clone(), out.tvb_stat.clone())
    for _ in range(150):
        api.tgvkv_score(*args, out.scores, out.tvb_stat, ws)
    assert api.tgvkv_status(ws) == 0
    assert torch.equal(out.scores, first[0]) and torch.equal(out.tvb_stat, first[1])


# ---------------------------------------------------------------- single steps
def test_budget_kernel_exact(api):
    """TVB budgets from crafted statistics, including exact ties, zeros and caps."""
    cases = [([0.5, 0.3, 0.2], 7, 100), ([1.0, 1.0, 1.0], 4, 100), ([0.9, 0.05, 0.05], 6, 3),
             ([0.0, 0.0, 0.0, 0.0], 6, 10), ([0.0, 2.0, 1.0], 6, 10), ([3.0, 1.0], 8, 4)]
    rng = np.random.default_rng(0)
    for _ in range(40):
        L = int(rng.integers(1, 40))
        cap = int(rng.integers(1, 300))
        stat = (rng.random(L) ** 2).astype(np.float32)
        stat[rng.random(L) < 0.2] = 0.0
        cases.append((stat.tolist(), int(rng.integers(0, L * cap + 1)), cap))
    for stat, total, cap in cases:
        L = len(stat)
        ratio = total / float(cap * L)
        # pick a ratio whose rounded total is `total`
        desc = api.make_desc(L, 1, 1, 64, cap, cap, 1)
        if api.tgvkv_vision_budget_total(desc, ratio) != total:
            ratio = (total + 0.25) / float(cap * L)
        assert api.tgvkv_vision_budget_total(desc, ratio) == total
        s = torch.tensor(np.asarray(stat, np.float32), device="cuda")
        b = torch.empty(L, dtype=torch.int32, device="cuda")
        ws = api.new_workspace(desc)
        api.tgvkv_budget(desc, s, ratio, b, ws)
        assert api.tgvkv_status(ws) == 0
        want = oracle.tvb_budgets(np.asarray(stat, np.float32).astype(np.float64), total, cap)
        assert b.cpu().tolist() == want, (stat, total, cap)


def test_select_kernel_ties_exact(api):
    rng = np.random.default_rng(5)
    for n, L, H in [(300, 3, 2), (2000, 2, 3), (5000, 1, 1)]:
        modality = (rng.random(n) < 0.8).astype(np.uint8)
        nv = int(modality.sum())
        scores = (np.round(rng.random((L, H, nv)) * 16) / 16).astype(np.float32)
        budgets = rng.integers(0, nv + 1, L).astype(np.int32)
        budgets[0] = nv
        if L > 1:
            budgets[1] = 0
        desc = api.make_desc(L, H, H, 64, n, nv, 1)
        ws = api.new_workspace(desc)
        off = torch.empty(L * H + 1, dtype=torch.int64, device="cuda")
        idx = torch.empty(L * H * n, dtype=torch.int32, device="cuda")
        api.tgvkv_select(desc, torch.from_numpy(scores).cuda(), torch.from_numpy(budgets).cuda(),
                         torch.from_numpy(modality).cuda(), off, idx, ws)
        assert api.tgvkv_status(ws) == 0
        o_off, o_idx = oracle.tpr_select(scores, budgets, modality)
        np.testing.assert_array_equal(off.cpu().numpy(), o_off)
        np.testing.assert_array_equal(idx[:o_off[-1]].cpu().numpy(), o_idx)


@pytest.mark.parametrize("d", [64, 128])
def test_compact_kernel_bit_exact(api, d):
    rng = np.random.default_rng(d)
    L, H, n = 3, 5, 77
    k = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    v = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    sets = []
    for lg in range(L * H):
        m = int(rng.integers(0, n + 1)) if lg % 4 else (0 if lg % 8 == 0 else n)
        sets.append(np.sort(rng.choice(n, m, replace=False)))
    off = np.cumsum([0] + [s.size for s in sets]).astype(np.int64)
    idx = np.concatenate(sets).astype(np.int32)
    desc = api.make_desc(L, H, H, d, n, 0, 1)
    ws = api.new_workspace(desc)
    rows = max(int(off[-1]), 1)
    ko = torch.zeros((rows, d), dtype=torch.int16, device="cuda")
    vo = torch.zeros((rows, d), dtype=torch.int16, device="cuda")
    api.tgvkv_compact(desc, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                      torch.from_numpy(off).cuda(), torch.from_numpy(idx).cuda(), ko, vo, ws)
    assert api.tgvkv_status(ws) == 0
    rk, rv = oracle.compact(k, v, off, idx.astype(np.int64))
    np.testing.assert_array_equal(ko[:off[-1]].cpu().numpy(), rk)
    np.testing.assert_array_equal(vo[:off[-1]].cpu().numpy(), rv)


def test_compact_csr_larger_than_output(api):
    """A CSR whose total exceeds the output capacity: the kernel's own check
    sets TGVKV_STATUS_INDEX, writes the rows that fit and nothing beyond."""
    rng = np.random.default_rng(5)
    L, H, n, d = 2, 3, 40, 128
    k = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    v = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    sets = [np.sort(rng.choice(n, 30, replace=False)) for _ in range(L * H)]
    off = np.cumsum([0] + [s.size for s in sets]).astype(np.int64)
    idx = np.concatenate(sets).astype(np.int32)
    desc = api.make_desc(L, H, H, d, n, 0, 1)
    ws = api.new_workspace(desc)
    cap = 100                                   # < off[-1] = 180
    guard = 64                                  # rows past the capacity that must stay untouched
    ko = torch.zeros((cap + guard, d), dtype=torch.int16, device="cuda")
    vo = torch.zeros((cap + guard, d), dtype=torch.int16, device="cuda")
    api.tgvkv_compact(desc, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                      torch.from_numpy(off).cuda(), torch.from_numpy(idx).cuda(), ko[:cap], vo[:cap],
                      ws)
    assert api.tgvkv_status(ws) == 0x08
    rk, rv = oracle.compact(k, v, off, idx.astype(np.int64))
    np.testing.assert_array_equal(ko[:cap].cpu().numpy(), rk[:cap])
    np.testing.assert_array_equal(vo[:cap].cpu().numpy(), rv[:cap])
    assert not ko[cap:].any() and not vo[cap:].any()


def test_compact_decreasing_offsets(api):
    """Offsets that decrease: TGVKV_STATUS_INDEX, and no row written past the
    output (every access of the kernel stays in bounds)."""
    rng = np.random.default_rng(6)
    L, H, n, d = 2, 2, 40, 128
    k = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    v = rng.integers(-2 ** 15, 2 ** 15, (L, H, n, d)).astype(np.int16)
    off = np.array([0, 20, 10, 35, 50], np.int64)   # set 1 ends before it starts
    idx = rng.integers(0, n, 50).astype(np.int32)
    desc = api.make_desc(L, H, H, d, n, 0, 1)
    ws = api.new_workspace(desc)
    cap, guard = 50, 32
    ko = torch.zeros((cap + guard, d), dtype=torch.int16, device="cuda")
    vo = torch.zeros((cap + guard, d), dtype=torch.int16, device="cuda")
    api.tgvkv_compact(desc, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                      torch.from_numpy(off).cuda(), torch.from_numpy(idx).cuda(), ko[:cap], vo[:cap],
                      ws)
    assert api.tgvkv_status(ws) & 0x08
    assert not ko[cap:].any() and not vo[cap:].any()


# ---------------------------------------------------------------- full sizes
FULL = [("llava15", 0.05, (0, 31)), ("llava15", 0.20, (17,)), ("next", 0.05, (0, 31)),
        ("next", 0.10, (5,)), ("next", 0.20, (26,)), ("qwen25", 0.05, (13,)),
        ("video", 0.05, (27,))]


@pytest.mark.parametrize("name,ratio,layers", FULL)
def test_full_size_sampled(api, name, ratio, layers):
    """The bench's launch configuration at full size: scores of sampled layers,
    the statistic of EVERY layer against the oracle's fp64 Eq. 5 statistic, the
    budgets against the oracle's own budgets from that statistic (equal except
    within tolerance of a rounding boundary) and against the oracle's split of
    the GPU's statistic (exact), and the sets and rows of the sampled layers."""
    wl = synth.WORKLOADS[name]
    inp = synth.generate(wl, seed=0)
    g = P.run_evict(api, wl, inp, ratio)
    assert g["status"] == 0
    layers = list(layers)
    ref_s, ref_t = P.oracle_scores(wl, inp, layers)
    P.assert_close(g["scores"][layers], ref_s, f"{name} scores")
    P.assert_close(g["stat"][layers], ref_t, f"{name} tvb_stat")
    o_stat = P.oracle_stat_all_layers(wl, inp, seed_key=0)
    P.assert_close(g["stat"], o_stat, f"{name} tvb_stat, every layer")
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    near = P.budgets_match(g["budgets"], o_stat, total, wl.N_v)
    if near:
        print(f"{name} r={ratio}: layers {near} differ from the oracle's fp64 budgets by one "
              f"unit at a rounding boundary")
    assert np.all(g["stat"] > 0)
    P.check_selection_and_compaction(wl, inp, g, layers, ref_scores=ref_s)
    assert g["offsets"][-1] == wl.H_kv * (wl.L * wl.N_t + total)
    assert np.all(np.diff(g["offsets"]) == np.repeat(wl.N_t + g["budgets"], wl.H_kv))


def test_layer_sharded_ranks_match_full_evict(api):
    """The host logic of layer sharding with the CUDA backend: two ranks'
    layer ranges scored separately, their statistics concatenated in rank
    order (what the all-gather returns), budgets from the full vector, each
    range selected and gathered on its own -- bit-identical to one full
    tgvkv_evict.  The ranks run one after another here; nothing waits on
    another rank's kernel."""
    from paper_2606_03075_gb300 import shard
    wl = synth.custom("shard_gqa", 5, 8, 2, 128,
                      [("text", 11), ("vision", 300), ("text", 9), ("vision", 140),
                       ("text", 33)], weights="dirichlet", ratios=(0.15,))
    inp = synth.generate(wl, seed=3)
    dev = P.device_inputs(inp)
    full = P.run_evict(api, wl, inp, 0.15, dev)
    assert full["status"] == 0
    desc_full = api.desc_for_workload(wl)
    backend = shard.CudaBackend("cuda")
    world, stats, scores, spans = 2, [], [], []
    for r in range(world):
        l0, l1 = shard.layer_range(wl.L, r, world)
        d = api.make_desc(l1 - l0, wl.H_q, wl.H_kv, wl.d, wl.N, wl.N_v, wl.n_win, 0.0, wl.n_win)
        s, st = backend.score(d, dev["q"][l0:l1].contiguous(), dev["k"][l0:l1].contiguous(),
                              dev["modality"], dev["text_pos"], dev["w"][l0:l1].contiguous())
        stats.append(st), scores.append(s), spans.append((l0, l1, d))
    full_stat = torch.cat(stats)
    np.testing.assert_array_equal(full_stat.cpu().numpy(), full["stat"])
    budgets = backend.budget(desc_full, full_stat, 0.15)
    np.testing.assert_array_equal(budgets.cpu().numpy(), full["budgets"])
    H = wl.H_kv
    for (l0, l1, d), s in zip(spans, scores):
        np.testing.assert_array_equal(s.cpu().numpy(), full["scores"][l0:l1])
        off, idx, ko, vo = backend.select_compact(d, s, budgets[l0:l1].contiguous(), dev["modality"],
                                                  dev["k"][l0:l1].contiguous(),
                                                  dev["v"][l0:l1].contiguous())
        lo, hi = full["offsets"][l0 * H], full["offsets"][l1 * H]
        np.testing.assert_array_equal(off.cpu().numpy(), full["offsets"][l0 * H:l1 * H + 1] - lo)
        np.testing.assert_array_equal(idx.cpu().numpy(), full["idx"][lo:hi])
        np.testing.assert_array_equal(ko.view(torch.int16).cpu().numpy(), full["k_out"][lo:hi])
        np.testing.assert_array_equal(vo.view(torch.int16).cpu().numpy(), full["v_out"][lo:hi])


def test_head_sharded_ranks_match_full_evict(api):
    """The host logic of sharding by KV head with the CUDA backend: two ranks'
    KV heads of every layer scored separately, their per-head TV masses
    concatenated in head order (what the all-gather returns), S_l summed in head
    order -- bit-identical to one full tgvkv_evict's statistic -- budgets from
    it, each rank's heads selected and gathered on their own, every set equal
    to the full call's.  The ranks run one after another on one GPU."""
    from paper_2606_03075_gb300 import shard
    wl = synth.custom("shard_heads_gpu", 4, 12, 4, 128,
                      [("text", 11), ("vision", 300), ("text", 9), ("vision", 140),
                       ("text", 33)], weights="dirichlet", ratios=(0.15,))
    inp = synth.generate(wl, seed=4)
    dev = P.device_inputs(inp)
    full = P.run_evict(api, wl, inp, 0.15, dev)
    assert full["status"] == 0
    desc_full = api.desc_for_workload(wl)
    backend = shard.CudaBackend("cuda")
    world, G, H = 2, wl.H_q // wl.H_kv, wl.H_kv
    masses, parts = [], []
    for r in range(world):
        g0, g1 = shard.head_range(H, r, world)
        d = api.make_desc(wl.L, G * (g1 - g0), g1 - g0, wl.d, wl.N, wl.N_v, wl.n_win, 0.0, wl.n_win)
        s, m = backend.score_heads(d, dev["q"][:, G * g0:G * g1].contiguous(),
                                   dev["k"][:, g0:g1].contiguous(), dev["modality"],
                                   dev["text_pos"], dev["w"])
        masses.append(m)
        parts.append((g0, g1, d, s))
    stat = shard.layer_stat_from_heads(torch.cat(masses, dim=1))
    np.testing.assert_array_equal(stat.cpu().numpy(), full["stat"])
    budgets = backend.budget(desc_full, stat, 0.15)
    np.testing.assert_array_equal(budgets.cpu().numpy(), full["budgets"])
    for g0, g1, d, s in parts:
        np.testing.assert_array_equal(s.cpu().numpy(), full["scores"][:, g0:g1])
        off, idx, ko, vo = backend.select_compact(d, s, budgets, dev["modality"],
                                                  dev["k"][:, g0:g1].contiguous(),
                                                  dev["v"][:, g0:g1].contiguous())
        off, idx = off.cpu().numpy(), idx.cpu().numpy()
        ko, vo = ko.view(torch.int16).cpu().numpy(), vo.view(torch.int16).cpu().numpy()
        h = g1 - g0
        for l in range(wl.L):
            for gl in range(h):
                lo, hi = off[l * h + gl], off[l * h + gl + 1]
                rlo, rhi = full["offsets"][l * H + g0 + gl], full["offsets"][l * H + g0 + gl + 1]
                np.testing.assert_array_equal(idx[lo:hi], full["idx"][rlo:rhi])
                np.testing.assert_array_equal(ko[lo:hi], full["k_out"][rlo:rhi])
                np.testing.assert_array_equal(vo[lo:hi], full["v_out"][rlo:rhi])
