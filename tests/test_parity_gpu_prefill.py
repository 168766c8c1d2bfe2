"""GPU parity of the prefill side of the path: causal prefill attention over
every token (tgvkv_prefill) with the eviction rows' statistics it keeps, and
the eviction step that takes those statistics (tgvkv_evict_with_stats) --
the CUDA path through the C ABI against the fp64 oracle.

Tolerances, from the arithmetic of the kernel:
  * o: |gpu - oracle| <= 2^-7 sum_j A_ij |v_jc| + 1e-6.  The attention weights
    enter the value product rounded to bf16 (relative error <= 2^-9 each) and o
    is rounded to bf16 (<= 2^-9 of |o| <= sum_j A_ij |v_jc|); fp32 accumulation,
    the fp32 normaliser and ex2.approx add ~1e-6 relative.  2^-7 leaves a factor
    two over the sum of both roundings.
  * row statistics: m + log2 Z within 1e-3 of log2 sum_j exp(x_ij) (a relative
    error of 7e-4 in Z), the vision share V / Z within 1e-3 relative (plus a
    1e-6 floor), m at most 8 below the row's largest base-2 logit and not above
    it (the kernel's stale-maximum rule).
  * q_text: bit copies of the query rows.
  * the eviction with the given statistics: the bar of the eviction tests --
    scores and statistic within 1e-3 of the oracle (2e-3 with Eq. 7 weights),
    budgets, retained sets and compacted rows exact given the GPU's statistic
    and scores; TT budgeting included.
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
    # one partial tile (N = 112), d = 64
    "tiny": synth.WORKLOADS["tiny"],
    # MHA, four row tiles with a ragged last tile (N = 473)
    "mha_ragged": synth.custom("mha_ragged", 2, 4, 4, 128,
                               [("text", 13), ("vision", 300), ("text", 9), ("vision", 61),
                                ("text", 90)], ratios=(0.1, 0.5)),
    # grouped-query heads, d = 64
    "gqa_d64": synth.custom("gqa_d64", 2, 8, 2, 64,
                            [("text", 20), ("vision", 180), ("text", 70)], ratios=(0.2,)),
    # grouped-query (G = 7), text interleaved with frames, every text token a query row
    "gqa_video": synth.custom("gqa_video", 2, 14, 2, 128, _video_like(6, 5, 40, 9, 30),
                              window="all_text", weights="dirichlet", ratios=(0.05,)),
}


def _bf16(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda().view(torch.bfloat16)


def _run_prefill(api, wl, inp, dev=None):
    desc = api.desc_for_workload(wl)
    dev = dev or P.device_inputs(inp)
    q_all = _bf16(inp["q_all"])
    o = torch.empty_like(q_all)
    q_text = torch.empty((wl.L, wl.H_q, wl.n_win, wl.d), dtype=torch.bfloat16, device="cuda")
    stats = torch.empty((wl.L, wl.H_q, wl.n_win, 3), dtype=torch.float32, device="cuda")
    ws = api.new_workspace(desc)
    api.tgvkv_prefill(desc, q_all, dev["k"], dev["v"], dev["modality"], dev["text_pos"], o, q_text,
                      stats, ws)
    assert api.tgvkv_status(ws) == 0
    return o, q_text, stats


def _check_prefill(wl, inp, o, q_text, stats, layers=None):
    layers = list(range(wl.L)) if layers is None else list(layers)
    scale = 1.0 / math.sqrt(wl.d)
    q_all = oracle.widen_bf16(inp["q_all"][layers])
    k = oracle.widen_bf16(inp["k"][layers])
    v = oracle.widen_bf16(inp["v"][layers])
    o_ref, bound = oracle.prefill_attention(q_all, k, v, scale, wl.H_kv)
    o_gpu = oracle.widen_bf16(o.view(torch.int16).cpu().numpy()[layers])
    err = np.abs(o_gpu - o_ref)
    tol = 2.0 ** -7 * bound + 1e-6
    bad = err > tol
    assert not bad.any(), (f"o: {bad.sum()} of {bad.size} outside tolerance; worst excess "
                           f"{(err - tol).max()!r}")
    # the query rows, bit for bit
    np.testing.assert_array_equal(q_text.view(torch.int16).cpu().numpy()[layers],
                                  inp["q_all"][layers][:, :, inp["text_pos"]])
    # (m, Z, V) of the query rows
    lse2, vis = oracle.row_statistics(q_all, k, inp["modality"], inp["text_pos"], scale, wl.H_kv)
    st = stats.cpu().numpy().astype(np.float64)[layers]
    m, z, vm = st[..., 0], st[..., 1], st[..., 2]
    assert np.all(z > 0)
    assert np.all(np.abs(m + np.log2(z) - lse2) <= 1e-3), np.abs(m + np.log2(z) - lse2).max()
    P.assert_close(vm / z, vis, "vision share of the rows")
    # the reference maximum: at most 8 below the row maximum, not above it
    top = np.empty_like(m)
    pos = inp["text_pos"]
    for n, l in enumerate(layers):
        for h in range(wl.H_q):
            x = scale * (q_all[n, h, pos] @ k[n, h // (wl.H_q // wl.H_kv)].T) / math.log(2.0)
            x = np.where(np.arange(wl.N)[None, :] <= pos[:, None], x, -np.inf)
            top[n, h] = x.max(axis=1)
    assert np.all(m <= top + 1e-3 * np.maximum(1.0, np.abs(top)))
    assert np.all(m >= top - 8.0 - 1e-3 * np.maximum(1.0, np.abs(top)))


@pytest.mark.parametrize("name", sorted(CASES))
def test_prefill_attention_and_row_statistics(api, name):
    wl = CASES[name]
    inp = synth.generate_prefill(wl, seed=3)
    o, q_text, stats = _run_prefill(api, wl, inp)
    _check_prefill(wl, inp, o, q_text, stats)


def _run_evict_with_stats(api, wl, dev, q_text, stats, ratio, **options):
    desc = api.desc_for_workload(wl, **options)
    ws = api.new_workspace(desc)
    out = api.alloc_outputs(desc, ratio)
    api.tgvkv_evict_with_stats(desc, q_text, dev["k"], dev["v"], dev["modality"], dev["text_pos"],
                               dev["w"], ratio, stats, out, ws)
    status = api.tgvkv_status(ws)
    rows = int(out.offsets[-1].item())
    assert rows <= api.tgvkv_retained_rows(desc, ratio)
    return dict(scores=out.scores.cpu().numpy(), stat=out.tvb_stat.cpu().numpy(),
                budgets=out.budgets.cpu().numpy().astype(np.int64),
                offsets=out.offsets.cpu().numpy(),
                idx=out.idx[:rows].cpu().numpy().astype(np.int64),
                k_out=out.k_out[:rows].view(torch.int16).cpu().numpy(),
                v_out=out.v_out[:rows].view(torch.int16).cpu().numpy(), status=status)


@pytest.mark.parametrize("name", sorted(CASES))
def test_evict_with_prefill_statistics(api, name):
    """prefill -> evict with its q_text and row statistics equals the oracle's
    eviction step (which computes the row statistics itself)."""
    wl = CASES[name]
    inp = synth.generate_prefill(wl, seed=3)
    dev = P.device_inputs(inp)
    _, q_text, stats = _run_prefill(api, wl, inp, dev)
    for ratio in wl.ratios:
        g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio)
        assert g["status"] == 0
        ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"],
                           inp["w"], ratio, wl.H_kv)
        P.assert_close(g["scores"], ref["scores"], "scores")
        P.assert_close(g["stat"], ref["stat"], "tvb_stat")
        total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
        assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
        P.check_selection_and_compaction(wl, inp, g, list(range(wl.L)),
                                         ref_scores=ref["scores"] if np.array_equal(
                                             g["budgets"], ref["budgets"]) else None)
        assert g["offsets"][-1] == wl.H_kv * (wl.L * wl.N_t + total)


def _kept_gap_rule(ref, b, kept, what):
    """The kept candidates equal the oracle's top b where its b-th / (b+1)-th
    gap exceeds 1e-3; keys that differ lie within 1e-3 of the b-th score."""
    if b <= 0:
        assert not kept, (what, kept)
        return
    order = np.lexsort((np.arange(ref.size), -ref))
    want = set(order[:b].tolist())
    if kept == want:
        return
    kth = ref[order[b - 1]]
    nxt = ref[order[b]] if b < ref.size else -np.inf
    assert not (kth - nxt > P.RTOL * abs(kth)), (what, kth, nxt)
    for c in kept ^ want:
        assert abs(ref[c] - kth) <= P.RTOL * abs(kth) + 1e-12, (what, c, ref[c], kth)


@pytest.mark.parametrize("name", ["mha_ragged", "gqa_video"])
def test_evict_with_prefill_statistics_widened(api, name):
    """The same with Eq. 7 weights, the all-token basis and sinks: the text-key
    pass takes the given statistics too."""
    wl = CASES[name]
    inp = synth.generate_prefill(wl, seed=4)
    dev = P.device_inputs(inp)
    _, q_text, stats = _run_prefill(api, wl, inp, dev)
    scale = 1.0 / math.sqrt(wl.d)
    q = oracle.widen_bf16(inp["q"])
    kk = oracle.widen_bf16(inp["k"])
    ts_ref, w_ref = oracle.text_scores_and_weights(q, kk, inp["modality"], inp["text_pos"], scale,
                                                   wl.H_kv)
    vs_ref, stat_ref = oracle.twr_scores_tvb_stat(q, kk, inp["modality"], inp["text_pos"], w_ref,
                                                  scale, wl.H_kv)
    text = np.flatnonzero(inp["modality"] == 0)
    vision = np.flatnonzero(inp["modality"] == 1)
    for ratio in (0.02, 0.9):
        g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio, basis="all", weights="eq7",
                                  keep_first=4, keep_last=1)
        assert g["status"] == 0
        P.assert_close(g["scores"], vs_ref, "scores (Eq. 7 weights)", rtol=2e-3)
        P.assert_close(g["stat"], stat_ref, "tvb_stat")
        total = oracle.all_budget_total(ratio, wl.N, wl.L)
        assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N)
        sinks = set(oracle.sink_positions(wl.N, 4, 1).tolist())
        for l in range(wl.L):
            b = int(g["budgets"][l])
            for h in range(wl.H_kv):
                lo, hi = g["offsets"][l * wl.H_kv + h], g["offsets"][l * wl.H_kv + h + 1]
                kept = g["idx"][lo:hi]
                assert np.all(np.diff(kept) > 0) and sinks <= set(kept.tolist())
                np.testing.assert_array_equal(g["k_out"][lo:hi], inp["k"][l, h][kept])
                np.testing.assert_array_equal(g["v_out"][lo:hi], inp["v"][l, h][kept])
                if b > wl.N_t:      # every text key, and the top vision keys by s^V
                    assert set(text.tolist()) <= set(kept.tolist())
                    cand = [int(np.searchsorted(vision, p)) for p in kept
                            if inp["modality"][p] == 1 and p not in sinks]
                    ref = vs_ref[l, h].copy()
                    sink_v = [int(np.searchsorted(vision, p)) for p in sinks
                              if inp["modality"][p] == 1]
                    ref[sink_v] = -np.inf
                    _kept_gap_rule(ref, b - wl.N_t - len(sink_v), set(cand), (l, h))
                else:               # the top text keys by s^T, no vision beyond sinks
                    assert all(inp["modality"][p] == 0 or p in sinks for p in kept)
                    cand = [int(np.searchsorted(text, p)) for p in kept
                            if inp["modality"][p] == 0 and p not in sinks]
                    ref = ts_ref[l, h].copy()
                    sink_t = [int(np.searchsorted(text, p)) for p in sinks
                              if inp["modality"][p] == 0]
                    ref[sink_t] = -np.inf
                    _kept_gap_rule(ref, b - len(sink_t), set(cand), (l, h))


def test_evict_with_statistics_tt_budgets(api):
    """TT budgeting with given statistics: the text-key pass keeps its own row
    statistics (the TT statistic is each row's text mass), the vision pass reads
    the given ones; statistic, budgets, scores and sets against the oracle."""
    wl = CASES["mha_ragged"]
    inp = synth.generate_prefill(wl, seed=5)
    dev = P.device_inputs(inp)
    _, q_text, stats = _run_prefill(api, wl, inp, dev)
    ratio = 0.1
    g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio, stat="tt")
    assert g["status"] == 0
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], inp["w"],
                       ratio, wl.H_kv, budget_stat="tt")
    P.assert_close(g["stat"], ref["stat"], "TT statistic")
    P.assert_close(g["scores"], ref["scores"], "scores")
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    P.check_selection_and_compaction(wl, inp, g, list(range(wl.L)),
                                     ref_scores=ref["scores"] if np.array_equal(
                                         g["budgets"], ref["budgets"]) else None)


FULL = [("llava15", 0.05, (0, 31)), ("qwen25", 0.05, (13,))]


@pytest.mark.parametrize("name,ratio,layers", FULL)
def test_full_size_prefill_then_evict(api, name, ratio, layers):
    """At full size, in the launch configuration the bench times: the prefill's
    output and row statistics of sampled layers against the oracle, then the
    eviction with those statistics."""
    wl = synth.WORKLOADS[name]
    inp = synth.generate_prefill(wl, seed=0)
    dev = P.device_inputs(inp)
    o, q_text, stats = _run_prefill(api, wl, inp, dev)
    _check_prefill(wl, inp, o, q_text, stats, layers=layers[:1])
    g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio)
    assert g["status"] == 0
    layers = list(layers)
    ref_s, ref_t = P.oracle_scores(wl, inp, layers)
    P.assert_close(g["scores"][layers], ref_s, f"{name} scores")
    P.assert_close(g["stat"][layers], ref_t, f"{name} tvb_stat")
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    P.check_selection_and_compaction(wl, inp, g, layers, ref_scores=ref_s)
    assert g["offsets"][-1] == wl.H_kv * (wl.L * wl.N_t + total)


def test_prefill_without_query_rows(api):
    """The plain causal attention (no query rows: no statistics, no q_text)."""
    wl = CASES["gqa_d64"]
    inp = synth.generate_prefill(wl, seed=6)
    desc = api.make_desc(wl.L, wl.H_q, wl.H_kv, wl.d, wl.N, wl.N_v, 0)
    dev = P.device_inputs(inp)
    q_all = _bf16(inp["q_all"])
    o = torch.empty_like(q_all)
    ws = api.new_workspace(desc)
    api.tgvkv_prefill(desc, q_all, dev["k"], dev["v"], dev["modality"], None, o, None, None, ws)
    assert api.tgvkv_status(ws) == 0
    o_ref, bound = oracle.prefill_attention(oracle.widen_bf16(inp["q_all"]),
                                            oracle.widen_bf16(inp["k"]),
                                            oracle.widen_bf16(inp["v"]), 1.0 / math.sqrt(wl.d),
                                            wl.H_kv)
    err = np.abs(oracle.widen_bf16(o.view(torch.int16).cpu().numpy()) - o_ref)
    assert np.all(err <= 2.0 ** -7 * bound + 1e-6), (err - 2.0 ** -7 * bound).max()


def test_prefill_repeated_calls_bit_identical(api):
    """Back-to-back launches on one workspace give the same bits (the schedule
    does not change any sum)."""
    wl = CASES["gqa_video"]
    inp = synth.generate_prefill(wl, seed=7)
    dev = P.device_inputs(inp)
    first = [t.clone() for t in _run_prefill(api, wl, inp, dev)]
    for _ in range(5):
        again = _run_prefill(api, wl, inp, dev)
        for a, b in zip(first, again):
            assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a,
                               b.view(torch.int16) if b.dtype == torch.bfloat16 else b)


FULL_LONG = [("next", 0.05, 31, 640), ("video", 0.05, 27, 512)]


@pytest.mark.parametrize("name,ratio,layer,n_prefix", FULL_LONG)
def test_full_size_long_prefill_then_evict(api, name, ratio, layer, n_prefix):
    """The long workloads at full size: o of one layer's first n_prefix rows
    (causal rows below n_prefix see only the first n_prefix keys, so the oracle
    on the truncated sequence is exact for them), the query rows' statistics
    over all keys, then the eviction with those statistics on that layer."""
    wl = synth.WORKLOADS[name]
    inp = synth.generate_prefill(wl, seed=0)
    dev = P.device_inputs(inp)
    o, q_text, stats = _run_prefill(api, wl, inp, dev)
    scale = 1.0 / math.sqrt(wl.d)
    q1 = oracle.widen_bf16(inp["q_all"][layer:layer + 1])
    k1 = oracle.widen_bf16(inp["k"][layer:layer + 1])
    v1 = oracle.widen_bf16(inp["v"][layer:layer + 1])
    o_ref, bound = oracle.prefill_attention(q1[:, :, :n_prefix], k1[:, :, :n_prefix],
                                            v1[:, :, :n_prefix], scale, wl.H_kv)
    o_gpu = oracle.widen_bf16(o.view(torch.int16)[layer:layer + 1, :, :n_prefix].cpu().numpy())
    assert np.all(np.abs(o_gpu - o_ref) <= 2.0 ** -7 * bound + 1e-6)
    np.testing.assert_array_equal(q_text.view(torch.int16)[layer].cpu().numpy(),
                                  inp["q"][layer])
    lse2, vis = oracle.row_statistics(q1, k1, inp["modality"], inp["text_pos"], scale, wl.H_kv)
    st = stats[layer:layer + 1].cpu().numpy().astype(np.float64)
    assert np.all(np.abs(st[..., 0] + np.log2(st[..., 1]) - lse2) <= 1e-3)
    P.assert_close(st[..., 2] / st[..., 1], vis, f"{name} vision share")
    g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio)
    assert g["status"] == 0
    ref_s, ref_t = P.oracle_scores(wl, inp, [layer])
    P.assert_close(g["scores"][[layer]], ref_s, f"{name} scores")
    P.assert_close(g["stat"][[layer]], ref_t, f"{name} tvb_stat")
    total = oracle.vision_budget_total(ratio, wl.N_v, wl.L)
    assert g["budgets"].tolist() == oracle.tvb_budgets(g["stat"], total, wl.N_v)
    P.check_selection_and_compaction(wl, inp, g, [layer], ref_scores=ref_s)


def test_prefill_max_length(api):
    """Heads of the largest length the library accepts (N = 32768): the
    prefill's per-tile tables at their full size.  The first 512 rows against
    the oracle on the truncated sequence (exact for causal rows), the last row
    (which sees every key) against the oracle's attention over all of them,
    the query rows' statistics over all keys, then the eviction with them."""
    wl = synth.custom("max_len_prefill", 1, 2, 1, 64,
                      [("text", 40), ("vision", 32600), ("text", 128)], window=64,
                      ratios=(0.05,))
    assert wl.N == 32768
    inp = synth.generate_prefill(wl, seed=0)
    dev = P.device_inputs(inp)
    o, q_text, stats = _run_prefill(api, wl, inp, dev)
    scale = 1.0 / math.sqrt(wl.d)
    q1, k1, v1 = (oracle.widen_bf16(inp[n]) for n in ("q_all", "k", "v"))
    o_gpu = oracle.widen_bf16(o.view(torch.int16).cpu().numpy())
    n_prefix = 512
    o_ref, bound = oracle.prefill_attention(q1[:, :, :n_prefix], k1[:, :, :n_prefix],
                                            v1[:, :, :n_prefix], scale, wl.H_kv)
    assert np.all(np.abs(o_gpu[:, :, :n_prefix] - o_ref) <= 2.0 ** -7 * bound + 1e-6)
    # the last row: attention over the whole sequence, as one set of every row
    last, every = wl.N - 1, np.array([0, wl.N])
    o_last = oracle.decode_attention(q1[:, :, last], k1[0, 0], v1[0, 0], every, wl.H_kv, scale)
    b_last = oracle.decode_attention(q1[:, :, last], k1[0, 0], np.abs(v1[0, 0]), every, wl.H_kv,
                                     scale)
    assert np.all(np.abs(o_gpu[:, :, last] - o_last) <= 2.0 ** -7 * b_last + 1e-6)
    np.testing.assert_array_equal(q_text.view(torch.int16).cpu().numpy(), inp["q"])
    lse2, vis = oracle.row_statistics(q1, k1, inp["modality"], inp["text_pos"], scale, wl.H_kv)
    st = stats.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(st[..., 0] + np.log2(st[..., 1]) - lse2) <= 1e-3)
    P.assert_close(st[..., 2] / st[..., 1], vis, "vision share")
    g = _run_evict_with_stats(api, wl, dev, q_text, stats, 0.05)
    assert g["status"] == 0
    ref_s, ref_t = P.oracle_scores(wl, inp, [0])
    P.assert_close(g["scores"], ref_s, "scores")
    P.assert_close(g["stat"], ref_t, "tvb_stat")
    total = oracle.vision_budget_total(0.05, wl.N_v, wl.L)
    assert g["budgets"].tolist() == [total]
    P.check_selection_and_compaction(wl, inp, g, [0], ref_scores=ref_s)


@pytest.mark.parametrize("stat", ["tv", "uniform"])
def test_evict_with_statistics_head_budgets(api, stat):
    """Head-adaptive budgets with given statistics: the per-head TV masses come
    from the prefill's rows; budgets, CSR, sets and rows exact given them."""
    wl = CASES["gqa_video"]
    inp = synth.generate_prefill(wl, seed=8)
    dev = P.device_inputs(inp)
    _, q_text, stats = _run_prefill(api, wl, inp, dev)
    ratio = 0.2
    g = _run_evict_with_stats(api, wl, dev, q_text, stats, ratio, stat=stat, head_budgets=True)
    assert g["status"] == 0
    L, H = wl.L, wl.H_kv
    total = oracle.vision_budget_total(ratio, wl.N_v, L)
    if stat == "tv":
        q, k = oracle.widen_bf16(inp["q"]), oracle.widen_bf16(inp["k"])
        ref = oracle.tv_statistic_per_head(q, k, inp["modality"], inp["text_pos"],
                                           1.0 / math.sqrt(wl.d), H)
        P.assert_close(g["stat"].reshape(L, H), ref, "per-head TV mass")
    stat_used = g["stat"] if stat == "tv" else np.zeros(L * H)
    budgets = np.asarray(oracle.tvb_budgets(stat_used, H * total, wl.N_v)).reshape(L, H)
    np.testing.assert_array_equal(g["budgets"].reshape(L, H), budgets)
    off, idx = oracle.tpr_select_general(g["scores"], None, budgets, inp["modality"],
                                         vision_basis=True)
    np.testing.assert_array_equal(g["offsets"], off)
    np.testing.assert_array_equal(g["idx"], idx)
    ko, vo = oracle.compact(inp["k"], inp["v"], off, idx)
    np.testing.assert_array_equal(g["k_out"], ko)
    np.testing.assert_array_equal(g["v_out"], vo)
