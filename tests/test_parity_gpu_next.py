"""GPU parity of the widened path: Eq. 9 text scores, Eq. 7 derived weights,
the all-token budget basis with both cases of Eq. 10, and sink tokens -- the
CUDA path through the C ABI against the fp64 oracle.

Tolerances: text scores and weights within 1e-3 relative (fp32 accumulation,
as the vision scores).  Vision scores computed with the GPU's derived weights
are compared with the oracle fed those same weights (1e-3); against the
oracle's own Eq. 7 weights the bound is 2e-3, the weights' relative error
adding to the attention's (the score is a positive combination of attention
entries with those weights).  Budgets, retained sets and compacted rows are
exact given the GPU's statistic and scores (integer decisions in the same
fp32 values on both sides).
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


def _video_like(frames, stamp, per_frame, head, tail):
    s = [("text", head)]
    for _ in range(frames):
        s += [("text", stamp), ("vision", per_frame)]
    return s + [("text", tail)]


CASES = {
    # several key tiles, a ragged tail, MHA with one row tile per head
    "mha_single": synth.custom("mha_single", 2, 4, 4, 128,
                               [("text", 13), ("vision", 300), ("text", 9), ("vision", 61),
                                ("text", 90)], ratios=(0.1,)),
    # two heads per row tile (<= 64 rows), d = 64
    "mha_packed_d64": synth.custom("mha_packed_d64", 3, 4, 4, 64,
                                   [("text", 20), ("vision", 180), ("text", 40)], ratios=(0.2,)),
    # grouped-query heads, several row tiles per head, text interleaved
    "gqa_pairs": synth.custom("gqa_pairs", 2, 14, 2, 128, _video_like(6, 5, 40, 9, 30),
                              window="all_text", weights="dirichlet", ratios=(0.05,)),
    # text longer than vision
    "text_heavy": synth.custom("text_heavy", 2, 8, 2, 128,
                               [("text", 150), ("vision", 64), ("text", 200)], window=120,
                               ratios=(0.3,)),
}


def _oracle_text(wl, inp, layers=None):
    return oracle.text_scores_and_weights(oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"]),
                                          inp["modality"], inp["text_pos"], 1.0 / math.sqrt(wl.d),
                                          wl.H_kv, layers)


def _run_text(api, wl, dev):
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    ts = torch.empty((wl.L, wl.H_kv, wl.N_t), dtype=torch.float32, device="cuda")
    wt = torch.empty((wl.L, wl.n_win), dtype=torch.float32, device="cuda")
    api.tgvkv_text_scores(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], ts, wt, ws)
    assert api.tgvkv_status(ws) == 0
    return ts.cpu().numpy(), wt.cpu().numpy()


@pytest.mark.parametrize("name", sorted(CASES))
def test_text_scores_and_eq7_weights(api, name):
    wl = CASES[name]
    inp = synth.generate(wl, seed=1)
    ts, wt = _run_text(api, wl, P.device_inputs(inp))
    rts, rwt = _oracle_text(wl, inp)
    P.assert_close(ts, rts, "text scores (Eq. 9)")
    P.assert_close(wt, rwt, "weights (Eq. 7)")
    assert np.allclose(wt.sum(axis=1), 1.0, rtol=1e-5)


@pytest.mark.parametrize("name,layers", [("llava15", [0, 31]), ("qwen25", [5]), ("video", [27])])
def test_text_scores_full_size_sampled(api, name, layers):
    """Full-size shapes in the launch configuration tgvkv_evict uses, checked on
    sampled layers (the oracle evaluates only those)."""
    wl = synth.WORKLOADS[name]
    inp = synth.generate(wl, seed=0)
    ts, wt = _run_text(api, wl, P.device_inputs(inp))
    rts, rwt = _oracle_text(wl, inp, layers)
    P.assert_close(ts[layers], rts[layers], "text scores (Eq. 9)")
    P.assert_close(wt[layers], rwt[layers], "weights (Eq. 7)")


def _evict(api, wl, inp, ratio, **opts):
    desc = api.desc_for_workload(wl, **opts)
    dev = P.device_inputs(inp)
    ws = api.new_workspace(desc)
    out = api.alloc_outputs(desc, ratio)
    w = None if opts.get("weights") == "eq7" else dev["w"]
    api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"], w,
                    ratio, out, ws)
    status = api.tgvkv_status(ws)
    n = int(out.offsets[-1].item())
    assert n <= api.tgvkv_retained_rows(desc, ratio)
    return dict(scores=out.scores.cpu().numpy(), stat=out.tvb_stat.cpu().numpy(),
                budgets=out.budgets.cpu().numpy().astype(np.int64),
                offsets=out.offsets.cpu().numpy(), idx=out.idx[:n].cpu().numpy().astype(np.int64),
                k_out=out.k_out[:n].view(torch.int16).cpu().numpy(),
                v_out=out.v_out[:n].view(torch.int16).cpu().numpy(), status=status, dev=dev,
                desc=desc)


@pytest.mark.parametrize("name", sorted(CASES))
def test_evict_with_eq7_weights(api, name):
    wl = CASES[name]
    inp = synth.generate(wl, seed=2)
    g = _evict(api, wl, inp, wl.ratios[0], weights="eq7")
    assert g["status"] == 0
    _, gw = _run_text(api, wl, g["dev"])
    q, k = oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"])
    scale = 1.0 / math.sqrt(wl.d)
    # the scores of the evict call, against the oracle fed the GPU's weights
    s_gw, st = oracle.twr_scores_tvb_stat(q, k, inp["modality"], inp["text_pos"],
                                          gw.astype(np.float64), scale, wl.H_kv)
    P.assert_close(g["scores"], s_gw, "scores with the GPU's Eq. 7 weights")
    P.assert_close(g["stat"], st, "tvb_stat")
    # end to end against the oracle's own Eq. 7 weights
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], None,
                       wl.ratios[0], wl.H_kv, weights="eq7")
    P.assert_close(g["scores"], ref["scores"], "scores (Eq. 7 end to end)", rtol=2e-3)
    # selection and compaction exact given the GPU's scores and budgets
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], oracle.vision_budget_total(
        wl.ratios[0], wl.N_v, wl.L), wl.N_v)
    P.check_selection_and_compaction(wl, inp, g, list(range(wl.L)))


def _check_general(wl, inp, g, ratio, basis, keep):
    """Budgets from the GPU statistic and the retained sets from the GPU scores,
    exactly as the oracle decides them."""
    if basis == "all":
        total, cap = oracle.all_budget_total(ratio, wl.N, wl.L), wl.N
    else:
        total, cap = oracle.vision_budget_total(ratio, wl.N_v, wl.L), wl.N_v
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, cap)
    ts = g.get("text_scores")
    off, idx = oracle.tpr_select_general(g["scores"], ts, g["budgets"], inp["modality"], *keep,
                                         vision_basis=basis == "vision")
    np.testing.assert_array_equal(g["offsets"], off)
    np.testing.assert_array_equal(g["idx"], idx)
    ko, vo = oracle.compact(inp["k"], inp["v"], off, idx)
    np.testing.assert_array_equal(g["k_out"], ko)
    np.testing.assert_array_equal(g["v_out"], vo)


@pytest.mark.parametrize("name", sorted(CASES))
@pytest.mark.parametrize("ratio", [0.02, 0.3, 0.9])
def test_evict_all_token_basis(api, name, ratio):
    """Ratios that put layers in both cases of Eq. 10 (b_l <= N_t: text only;
    b_l > N_t: all text plus vision)."""
    wl = CASES[name]
    inp = synth.generate(wl, seed=3)
    g = _evict(api, wl, inp, ratio, basis="all")
    assert g["status"] == 0
    ts, _ = _run_text(api, wl, g["dev"])
    g["text_scores"] = ts
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], inp["w"],
                       ratio, wl.H_kv, basis="all")
    P.assert_close(g["scores"], ref["scores"], "scores")
    P.assert_close(ts, ref["text_scores"], "text scores")
    _check_general(wl, inp, g, ratio, "all", (0, 0))
    assert g["offsets"][-1] == wl.H_kv * oracle.all_budget_total(ratio, wl.N, wl.L)


SINK_CASE = synth.custom("sinks", 3, 6, 2, 128,
                         [("vision", 6), ("text", 11), ("vision", 200), ("text", 30),
                          ("vision", 3)], window=30, ratios=(0.1,))


@pytest.mark.parametrize("basis", ["vision", "all"])
@pytest.mark.parametrize("keep", [(4, 1), (8, 5)])
@pytest.mark.parametrize("ratio", [0.0, 0.05, 0.5])
def test_evict_with_sinks(api, basis, keep, ratio):
    """Sinks on vision and text tokens at both ends of the sequence."""
    wl = SINK_CASE
    inp = synth.generate(wl, seed=4)
    g = _evict(api, wl, inp, ratio, basis=basis, keep_first=keep[0], keep_last=keep[1])
    assert g["status"] == 0
    if basis == "all":
        g["text_scores"], _ = _run_text(api, wl, g["dev"])
    _check_general(wl, inp, g, ratio, basis, keep)
    sinks = oracle.sink_positions(wl.N, *keep)
    H = wl.H_kv
    for lg in range(wl.L * H):
        assert set(sinks.tolist()) <= set(g["idx"][g["offsets"][lg]:g["offsets"][lg + 1]].tolist())


def test_select_tpr_call_matches_evict(api):
    """The separate calls (text scores, score, budget, select_tpr, compact)
    give the fused call's result under the all-token basis with sinks."""
    wl = CASES["gqa_pairs"]
    inp = synth.generate(wl, seed=5)
    ratio = 0.3
    g = _evict(api, wl, inp, ratio, basis="all", keep_first=4, keep_last=1)
    desc, dev = g["desc"], g["dev"]
    ws = api.new_workspace(desc)
    ts = torch.empty((wl.L, wl.H_kv, wl.N_t), dtype=torch.float32, device="cuda")
    wt = torch.empty((wl.L, wl.n_win), dtype=torch.float32, device="cuda")
    api.tgvkv_text_scores(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], ts, wt, ws)
    sc = torch.empty((wl.L, wl.H_kv, wl.N_v), dtype=torch.float32, device="cuda")
    st = torch.empty(wl.L, dtype=torch.float32, device="cuda")
    api.tgvkv_score(desc, dev["q"], dev["k"], dev["modality"], dev["text_pos"], dev["w"], sc, st, ws)
    bud = torch.empty(wl.L, dtype=torch.int32, device="cuda")
    api.tgvkv_budget(desc, st, ratio, bud, ws)
    rows = api.tgvkv_retained_rows(desc, ratio)
    off = torch.empty(wl.L * wl.H_kv + 1, dtype=torch.int64, device="cuda")
    idx = torch.empty(rows, dtype=torch.int32, device="cuda")
    api.tgvkv_select_tpr(desc, sc, ts, bud, dev["modality"], off, idx, ws)
    n = int(off[-1].item())
    ko = torch.empty((rows, wl.d), dtype=torch.bfloat16, device="cuda")
    vo = torch.empty_like(ko)
    api.tgvkv_compact(desc, dev["k"], dev["v"], off, idx, ko, vo, ws)
    assert api.tgvkv_status(ws) == 0
    np.testing.assert_array_equal(off.cpu().numpy(), g["offsets"])
    np.testing.assert_array_equal(idx[:n].cpu().numpy(), g["idx"])
    np.testing.assert_array_equal(ko[:n].view(torch.int16).cpu().numpy(), g["k_out"])
    with pytest.raises(api.TgvkvError):
        api.tgvkv_select(desc, sc, bud, dev["modality"], off, idx, ws)


# ---------------------------------------------------------------- decode over the compacted cache
def _decode_q(wl, seed):
    rng = np.random.default_rng(seed)
    return synth.to_bf16_bits(rng.standard_normal((wl.L, wl.H_q, wl.d)).astype(np.float32))


def _run_decode(api, desc, q_bits, k_rows, v_rows, offsets):
    ws = api.new_workspace(desc)
    out = torch.empty((desc.L, desc.H_q, desc.d), dtype=torch.float32, device="cuda")
    qd = torch.from_numpy(np.ascontiguousarray(q_bits)).cuda().view(torch.bfloat16)
    api.tgvkv_decode(desc, qd, k_rows, v_rows, offsets, out, ws)
    assert api.tgvkv_status(ws) == 0
    return out.cpu().numpy()


# A decode output is a convex combination of value rows: an entry that nearly
# cancels (|o| far below its terms) carries the fp32 accumulation error of the
# terms (~n * 6e-8 of them), so the absolute floor is 1e-5 of the head's largest
# output rather than the scores' 1e-6.
DEC_FLOOR = 1e-5


def _oracle_decode(wl, q_bits, k_bits, v_bits, offsets):
    return oracle.decode_attention(oracle.widen_bf16(q_bits), oracle.widen_bf16(k_bits),
                                   oracle.widen_bf16(v_bits), offsets, wl.H_kv,
                                   1.0 / math.sqrt(wl.d))


DECODE_CASES = dict(CASES, tiny=synth.WORKLOADS["tiny"],
                    wide_group=synth.custom("wide_group", 1, 32, 1, 128,
                                            [("text", 3), ("vision", 90), ("text", 9)],
                                            ratios=(0.5,)))


@pytest.mark.parametrize("name", sorted(DECODE_CASES))
def test_decode_over_compacted_cache(api, name):
    """A decode step over the cache tgvkv_evict compacted, against the oracle on
    the same retained rows (G > 8 takes several head batches per KV head)."""
    wl = DECODE_CASES[name]
    inp = synth.generate(wl, seed=6)
    desc = api.desc_for_workload(wl)
    dev = P.device_inputs(inp)
    ws = api.new_workspace(desc)
    ratio = wl.ratios[0]
    out = api.alloc_outputs(desc, ratio)
    api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"], dev["w"],
                    ratio, out, ws)
    assert api.tgvkv_status(ws) == 0
    n = int(out.offsets[-1].item())
    qb = _decode_q(wl, 7)
    o = _run_decode(api, desc, qb, out.k_out, out.v_out, out.offsets)
    ref = _oracle_decode(wl, qb, out.k_out[:n].view(torch.int16).cpu().numpy(),
                         out.v_out[:n].view(torch.int16).cpu().numpy(), out.offsets.cpu().numpy())
    P.assert_close(o, ref, "decode over the compacted cache", floor=DEC_FLOOR)


@pytest.mark.parametrize("name", ["llava15", "qwen25"])
def test_decode_full_size(api, name):
    """Full-size caches: the compacted cache of tgvkv_evict and the full cache
    (identity offsets), every layer and head against the oracle; qwen25 has few
    KV heads, so its rows are split over several CTAs and merged."""
    wl = synth.WORKLOADS[name]
    inp = synth.generate(wl, seed=0)
    desc = api.desc_for_workload(wl)
    dev = P.device_inputs(inp)
    ws = api.new_workspace(desc)
    ratio = wl.ratios[0]
    out = api.alloc_outputs(desc, ratio)
    api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"], dev["w"],
                    ratio, out, ws)
    assert api.tgvkv_status(ws) == 0
    qb = _decode_q(wl, 8)
    n = int(out.offsets[-1].item())
    o = _run_decode(api, desc, qb, out.k_out, out.v_out, out.offsets)
    ref = _oracle_decode(wl, qb, out.k_out[:n].view(torch.int16).cpu().numpy(),
                         out.v_out[:n].view(torch.int16).cpu().numpy(), out.offsets.cpu().numpy())
    P.assert_close(o, ref, "decode, compacted cache", floor=DEC_FLOOR)
    full_off = torch.arange(wl.L * wl.H_kv + 1, dtype=torch.int64, device="cuda") * wl.N
    of = _run_decode(api, desc, qb, dev["k"], dev["v"], full_off)
    reff = _oracle_decode(wl, qb, inp["k"].reshape(-1, wl.d), inp["v"].reshape(-1, wl.d),
                          full_off.cpu().numpy())
    P.assert_close(of, reff, "decode, full cache", floor=DEC_FLOOR)


def test_decode_empty_sets_give_zero(api):
    """No text token and a zero budget: every set is empty and the output is 0."""
    wl = synth.custom("all_vision", 2, 4, 2, 64, [("vision", 70)], window="all_text",
                      ratios=(0.0,))
    desc = api.desc_for_workload(wl)
    offsets = torch.zeros(wl.L * wl.H_kv + 1, dtype=torch.int64, device="cuda")
    rows = torch.zeros((1, wl.d), dtype=torch.bfloat16, device="cuda")
    o = _run_decode(api, desc, _decode_q(wl, 9), rows, rows, offsets)
    assert np.array_equal(o, np.zeros_like(o))


# Ragged CSR layouts around the decode kernel's boxes (8 and 32 rows): sets of
# 0, 1, 7-9, 15-17, 31-33, 63-65 and 257 rows, empty sets between full ones, a
# base offset before the first set and spare rows after the last; groups of 1,
# 4 and 12 query heads (12 takes two passes of 8 heads) at d = 64 and 128; and
# one long set that every row stream of the GPU shares (merged from all of
# their partial results).
_RAGGED_LENS = [0, 1, 7, 8, 9, 15, 16, 17, 31, 32, 33, 0, 63, 64, 65, 257, 0, 3]


def _ragged_decode(api, L, H_kv, G, d, lens, base, spare, seed):
    wl = synth.custom("ragged", L, G * H_kv, H_kv, d, [("text", 8), ("vision", 300), ("text", 8)])
    desc = api.desc_for_workload(wl)
    rng = np.random.default_rng(seed)
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64) + base
    n_rows = int(offsets[-1]) + spare
    k_bits = synth.to_bf16_bits(rng.standard_normal((n_rows, d)).astype(np.float32))
    v_bits = synth.to_bf16_bits(rng.standard_normal((n_rows, d)).astype(np.float32))
    qb = _decode_q(wl, seed + 1)
    dev = lambda b: torch.from_numpy(np.ascontiguousarray(b)).cuda().view(torch.bfloat16)
    off_d = torch.from_numpy(offsets).cuda()
    o = _run_decode(api, desc, qb, dev(k_bits), dev(v_bits), off_d)
    ref = _oracle_decode(wl, qb, k_bits, v_bits, offsets)
    return o, ref


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("G", [1, 4, 12])
def test_decode_ragged_csr(api, d, G):
    """Decode over ragged CSR layouts, element by element against the oracle."""
    L, H_kv = 3, 6
    lens = _RAGGED_LENS
    o, ref = _ragged_decode(api, L, H_kv, G, d, lens, base=5, spare=37, seed=20 + G + d)
    P.assert_close(o, ref, f"decode, ragged CSR (G={G}, d={d})", floor=DEC_FLOOR)


@pytest.mark.parametrize("G", [1, 7])
def test_decode_one_long_set(api, G):
    """One set of 40 000 rows: every row stream takes a slice of it, and the last
    stream to finish merges all partial results."""
    o, ref = _ragged_decode(api, 1, 1, G, 128, [40000], base=0, spare=0, seed=31 + G)
    P.assert_close(o, ref, f"decode, one long set (G={G})", floor=DEC_FLOOR)


def test_decode_csr_past_capacity(api):
    """A CSR whose last set runs past the rows the buffers hold: the kernel
    reads no row from capacity_rows on and reports TGVKV_STATUS_INDEX."""
    wl = synth.custom("short_cache", 1, 4, 2, 128, [("text", 8), ("vision", 300), ("text", 8)])
    desc = api.desc_for_workload(wl)
    rows = torch.zeros((100, wl.d), dtype=torch.bfloat16, device="cuda")
    offsets = torch.tensor([0, 60, 180], dtype=torch.int64, device="cuda")
    ws = api.new_workspace(desc)
    out = torch.empty((desc.L, desc.H_q, desc.d), dtype=torch.float32, device="cuda")
    qd = torch.from_numpy(_decode_q(wl, 3)).cuda().view(torch.bfloat16)
    api.tgvkv_decode(desc, qd, rows, rows, offsets, out, ws)
    assert api.tgvkv_status(ws) == 0x08


# ---------------------------------------------------------------- layer-budget statistics (Table 1a)
@pytest.mark.parametrize("name", ["mha_single", "gqa_pairs", "text_heavy"])
@pytest.mark.parametrize("stat", ["tt", "uniform"])
def test_evict_budget_statistics(api, name, stat):
    """TT budgets follow the text-key pass's text-text mass (returned as
    tvb_stat); uniform budgets ignore the statistic.  Budgets exact given the
    GPU statistic, the statistic within 1e-3, sets and rows exact."""
    wl = CASES[name]
    inp = synth.generate(wl, seed=10)
    ratio = wl.ratios[0]
    g = _evict(api, wl, inp, ratio, stat=stat)
    assert g["status"] == 0
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    if stat == "tt":
        q, k = oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"])
        tt = oracle.tt_statistic(q, k, inp["modality"], inp["text_pos"], 1.0 / math.sqrt(wl.d),
                                 wl.H_kv)
        P.assert_close(g["stat"], tt, "TT statistic")
        assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    else:
        assert g["budgets"].tolist() == oracle.tvb_budgets(np.zeros(wl.L), total, wl.N_v)
    P.check_selection_and_compaction(wl, inp, g, list(range(wl.L)))


def test_vv_statistic_with_vision_rows(api):
    """VV budgeting: tgvkv_score with the vision tokens' queries as the rows
    returns the vision-vision mass as tvb_stat; tgvkv_budget splits it."""
    base = CASES["mha_single"]
    vpos = np.flatnonzero(base.modality == 1)
    rng = np.random.default_rng(11)
    L, H_q, H_kv, d = base.L, base.H_q, base.H_kv, base.d
    qv = synth.to_bf16_bits(rng.standard_normal((L, H_q, vpos.size, d)).astype(np.float32))
    inp = synth.generate(base, seed=11)
    desc = api.make_desc(L, H_q, H_kv, d, base.N, base.N_v, int(vpos.size))
    ws = api.new_workspace(desc)
    up = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    w = torch.full((L, vpos.size), 1.0 / vpos.size, dtype=torch.float32, device="cuda")
    sc = torch.empty((L, H_kv, base.N_v), dtype=torch.float32, device="cuda")
    st = torch.empty(L, dtype=torch.float32, device="cuda")
    api.tgvkv_score(desc, up(qv).view(torch.bfloat16), up(inp["k"]).view(torch.bfloat16),
                    up(inp["modality"]), up(vpos.astype(np.int32)), w, sc, st, ws)
    bud = torch.empty(L, dtype=torch.int32, device="cuda")
    api.tgvkv_budget(desc, st, 0.2, bud, ws)
    assert api.tgvkv_status(ws) == 0
    _, vv = oracle.twr_scores_tvb_stat(oracle.widen_bf16(qv), oracle.widen_bf16(inp["k"]),
                                       inp["modality"], vpos, np.full((L, vpos.size), 1.0 / vpos.size),
                                       1.0 / math.sqrt(d), H_kv)
    P.assert_close(st.cpu().numpy(), vv, "VV statistic")
    assert bud.cpu().tolist() == oracle.tvb_budgets(st.cpu().numpy(),
                                                    oracle.vision_budget_total(0.2, base.N_v, L),
                                                    base.N_v)


# ---------------------------------------------------------------- head-adaptive budgets
@pytest.mark.parametrize("name", ["mha_single", "gqa_pairs", "mha_packed_d64"])
@pytest.mark.parametrize("basis,stat", [("vision", "tv"), ("all", "tv"), ("vision", "uniform")])
def test_evict_head_budgets(api, name, basis, stat):
    """One budget per (layer, KV head): the per-head TV masses within 1e-3,
    budgets exact from the GPU's masses, sets and rows exact."""
    wl = CASES[name]
    inp = synth.generate(wl, seed=12)
    ratio = 0.3 if basis == "all" else wl.ratios[0]
    g = _evict(api, wl, inp, ratio, basis=basis, stat=stat, head_budgets=True)
    assert g["status"] == 0
    L, H = wl.L, wl.H_kv
    if basis == "all":
        total, cap = oracle.all_budget_total(ratio, wl.N, L), wl.N
    else:
        total, cap = oracle.vision_budget_total(ratio, wl.N_v, L), wl.N_v
    stat_used = g["stat"] if stat == "tv" else np.zeros(L * H)
    if stat == "tv":
        q, k = oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"])
        ref = oracle.tv_statistic_per_head(q, k, inp["modality"], inp["text_pos"],
                                           1.0 / math.sqrt(wl.d), H)
        P.assert_close(g["stat"].reshape(L, H), ref, "per-head TV mass")
    budgets = np.asarray(oracle.tvb_budgets(stat_used, H * total, cap)).reshape(L, H)
    np.testing.assert_array_equal(g["budgets"].reshape(L, H), budgets)
    ts = _run_text(api, wl, g["dev"])[0] if basis == "all" else None
    off, idx = oracle.tpr_select_general(g["scores"], ts, budgets, inp["modality"],
                                         vision_basis=basis == "vision")
    np.testing.assert_array_equal(g["offsets"], off)
    np.testing.assert_array_equal(g["idx"], idx)
    ko, vo = oracle.compact(inp["k"], inp["v"], off, idx)
    np.testing.assert_array_equal(g["k_out"], ko)
    np.testing.assert_array_equal(g["v_out"], vo)


def test_widened_paths_back_to_back_stay_clean(api):
    """Many consecutive calls of the widened evict paths and of decode on one
    workspace: the status stays clean and every call gives the first call's
    result bit for bit (the text-key pass hands row statistics to the vision
    pass through the workspace each time)."""
    wl = CASES["gqa_pairs"]
    inp = synth.generate(wl, seed=13)
    dev = P.device_inputs(inp)
    for opts in (dict(weights="eq7"), dict(basis="all", keep_first=4, keep_last=1),
                 dict(stat="tt", head_budgets=False), dict(head_budgets=True)):
        desc = api.desc_for_workload(wl, **opts)
        ws = api.new_workspace(desc)
        out = api.alloc_outputs(desc, wl.ratios[0])
        w = None if opts.get("weights") == "eq7" else dev["w"]
        first = None
        for it in range(40):
            api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"], w,
                            wl.ratios[0], out, ws)
            if it in (0, 39):
                assert api.tgvkv_status(ws) == 0, opts
                n = int(out.offsets[-1].item())
                snap = (out.scores.cpu().numpy().copy(), out.idx[:n].cpu().numpy().copy())
                if first is None:
                    first = snap
                else:
                    np.testing.assert_array_equal(snap[0], first[0])
                    np.testing.assert_array_equal(snap[1], first[1])
        qd = torch.from_numpy(_decode_q(wl, 14)).cuda().view(torch.bfloat16)
        o1 = torch.empty((wl.L, wl.H_q, wl.d), dtype=torch.float32, device="cuda")
        o2 = torch.empty_like(o1)
        api.tgvkv_decode(desc, qd, out.k_out, out.v_out, out.offsets, o1, ws)
        for _ in range(20):
            api.tgvkv_decode(desc, qd, out.k_out, out.v_out, out.offsets, o2, ws)
        assert api.tgvkv_status(ws) == 0
        assert torch.equal(o1, o2)
