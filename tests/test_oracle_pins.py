"""Pins of the fp64 oracle against facts that do not come from the oracle itself.

Each test checks the oracle against brute force, a closed form, an invariant of
the definitions, hand arithmetic or a number printed in the paper, chosen so
that a dropped term, a wrong sign or index, or a transposed operand fails one
of them.  CPU only.
"""
import math
import os

import numpy as np
import pytest

import oracle
from paper_2606_03075_gb300 import synth

RNG = np.random.default_rng(1234)


def _rand_case(L=2, H_q=4, H_kv=2, d=8, segments=(("text", 3), ("vision", 5), ("text", 2),
                                                  ("vision", 4), ("text", 3)),
               n_win=None, seed=0):
    rng = np.random.default_rng(seed)
    modality = np.concatenate([np.full(c, 1 if k == "vision" else 0, np.uint8)
                               for k, c in segments])
    text = np.flatnonzero(modality == 0)
    pos = text if n_win is None else text[-n_win:]
    n = modality.size
    q = rng.standard_normal((L, H_q, pos.size, d))
    k = rng.standard_normal((L, H_kv, n, d))
    w = rng.random((L, pos.size))
    w /= w.sum(axis=1, keepdims=True)
    return q, k, modality, pos.astype(np.int64), w


# ---------------------------------------------------------------- P1
def test_softmax_rows_sum_to_one():
    q, k, modality, pos, w = _rand_case()
    for l in range(q.shape[0]):
        for h in range(q.shape[1]):
            a = oracle.causal_text_attention(q[l, h], k[l, h // 2], pos, 0.37)
            assert np.all(np.abs(a.sum(axis=1) - 1.0) < 1e-12)
            # causal mask: nothing after each row's own position (Eq. 2, M)
            for i, p in enumerate(pos):
                assert np.all(a[i, p + 1:] == 0.0)
                assert np.all(a[i, : p + 1] > 0.0)


# ---------------------------------------------------------------- P2
def test_uniform_attention_closed_form():
    """Q = 0: every visible key gets 1/(p_i + 1) (Eq. 2), so Eq. 8 and Eq. 5
    reduce to counting."""
    q, k, modality, pos, w = _rand_case(L=1, H_q=3, H_kv=3)
    q[:] = 0.0
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 1.0, 3)
    vision = np.flatnonzero(modality == 1)
    expect = np.zeros(vision.size)
    for vi, j in enumerate(vision):
        expect[vi] = sum(w[0, i] / (p + 1) for i, p in enumerate(pos) if p >= j)
    for g in range(3):
        assert np.allclose(scores[0, g], expect, rtol=1e-13, atol=0)
    s_expect = 3 * sum(np.count_nonzero(vision <= p) / (p + 1) for p in pos)
    assert math.isclose(stat[0], s_expect, rel_tol=1e-13)


# ---------------------------------------------------------------- P3
def test_one_hot_saturation():
    """A query aligned with one key, much larger than the rest, puts all its
    attention on that key (softmax saturation)."""
    n, d = 12, 16
    keys = np.eye(d)[:n]
    pos = np.array([5, 8, 11])
    target = np.array([2, 7, 11])
    q = 80.0 * keys[target]
    a = oracle.causal_text_attention(q, keys, pos, 1.0)
    for i, t in enumerate(target):
        assert a[i, t] > 1.0 - 1e-12
        others = np.delete(a[i], t)
        assert np.all(others < 1e-12)


# ---------------------------------------------------------------- P4
def test_mass_consistency_uniform_weights():
    """With w~ = 1/n_win, summing Eq. 8 over vision keys and heads gives the
    TV mass of Eq. 5 divided by n_win (and the GQA mean divides by G)."""
    q, k, modality, pos, _ = _rand_case(L=3, H_q=6, H_kv=2, seed=5)
    n_win = pos.size
    w = np.full((3, n_win), 1.0 / n_win)
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.5, 2)
    g = 3
    for l in range(3):
        assert math.isclose(g * n_win * scores[l].sum(), stat[l], rel_tol=1e-12)
        assert 0.0 < stat[l] < 6 * n_win


# ---------------------------------------------------------------- P5
def test_tvb_budget_by_hand():
    # S = [0.5, 0.3, 0.2], B_V = 7: quotas 3.5, 2.1, 1.4 -> floors 3, 2, 1 and the
    # single leftover unit goes to the largest fraction (0.5, layer 0).
    assert oracle.tvb_budgets([0.5, 0.3, 0.2], 7, 100) == [4, 2, 1]
    # equal fractions: the leftover goes to the lower layer.
    assert oracle.tvb_budgets([1.0, 1.0, 1.0], 4, 100) == [2, 1, 1]
    assert oracle.tvb_budgets([1.0, 1.0, 1.0], 5, 100) == [2, 2, 1]
    # one layer takes everything
    assert oracle.tvb_budgets([0.37], 11, 100) == [11]
    # cap: quotas 5.4, 0.3, 0.3 with N_v = 3 -> layer 0 capped at 3; the other
    # 3 units split 1.5 / 1.5 -> 1 + 1, leftover to the lower layer.
    assert oracle.tvb_budgets([0.9, 0.05, 0.05], 6, 3) == [3, 2, 1]
    # zero statistic everywhere: uniform split
    assert oracle.tvb_budgets([0.0, 0.0, 0.0, 0.0], 6, 10) == [2, 2, 1, 1]
    # a zero layer gets nothing while others have mass
    assert oracle.tvb_budgets([0.0, 2.0, 1.0], 6, 10) == [0, 4, 2]
    # every layer capped
    assert oracle.tvb_budgets([3.0, 1.0], 8, 4) == [4, 4]
    with pytest.raises(ValueError):
        oracle.tvb_budgets([1.0, 1.0], 9, 4)


def test_tvb_budget_sums_and_caps_random():
    rng = np.random.default_rng(7)
    for _ in range(200):
        L = int(rng.integers(1, 40))
        cap = int(rng.integers(1, 50))
        total = int(rng.integers(0, L * cap + 1))
        stat = rng.random(L) ** 3
        b = oracle.tvb_budgets(stat, total, cap)
        assert sum(b) == total
        assert all(0 <= x <= cap for x in b)
        # proportionality: uncapped layers are within one unit of their quota
        # of what is left after the capped ones
        capped = [l for l in range(L) if b[l] == cap]
        free = [l for l in range(L) if l not in capped]
        rest = total - cap * len(capped)
        den = sum(stat[l] for l in free)
        for l in free:
            assert abs(b[l] - rest * stat[l] / den) < 1.0 + 1e-9


def test_vision_budget_totals():
    # B_V = floor(r * N_v * L + 1/2) for the five workloads
    cases = {("tiny", 0.25): 16, ("llava15", 0.05): 922, ("llava15", 0.20): 3686,
             ("next", 0.05): 4608, ("next", 0.10): 9216, ("next", 0.20): 18432,
             ("qwen25", 0.05): 5734, ("video", 0.05): 11469}
    for (name, r), expect in cases.items():
        wl = synth.WORKLOADS[name]
        assert oracle.vision_budget_total(r, wl.N_v, wl.L) == expect


# ---------------------------------------------------------------- P6
def test_topk_pairwise_definition():
    """Every kept vision key beats every dropped one: higher score, or the same
    score at a lower position."""
    rng = np.random.default_rng(11)
    modality = (rng.random(60) < 0.7).astype(np.uint8)
    nv = int(modality.sum())
    scores = np.round(rng.random((3, 2, nv)) * 8) / 8      # many exact ties
    budgets = [0, 5, nv]
    offsets, idx = oracle.tpr_select(scores, budgets, modality)
    vision = np.flatnonzero(modality == 1)
    rank = {int(p): r for r, p in enumerate(vision)}
    for l in range(3):
        for g in range(2):
            rows = idx[offsets[l * 2 + g]: offsets[l * 2 + g + 1]]
            kept = [rank[int(p)] for p in rows if modality[p] == 1]
            dropped = sorted(set(range(nv)) - set(kept))
            assert len(kept) == budgets[l]
            s = scores[l, g]
            for c in kept:
                for u in dropped:
                    assert s[c] > s[u] or (s[c] == s[u] and c < u)


def test_topk_all_equal_keeps_lowest_positions():
    modality = np.array([0, 1, 1, 0, 1, 1, 1, 0], np.uint8)
    scores = np.ones((1, 1, 5))
    offsets, idx = oracle.tpr_select(scores, [2], modality)
    assert idx.tolist() == [0, 1, 2, 3, 7]


# ---------------------------------------------------------------- P7
def test_retained_sets_structure():
    q, k, modality, pos, w = _rand_case(L=4, H_q=4, H_kv=2, seed=3)
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.3, 2)
    nv = int(modality.sum())
    total = oracle.vision_budget_total(0.4, nv, 4)
    budgets = oracle.tvb_budgets(stat, total, nv)
    offsets, idx = oracle.tpr_select(scores, budgets, modality)
    text = set(np.flatnonzero(modality == 0).tolist())
    nt = len(text)
    assert offsets[0] == 0 and offsets.size == 4 * 2 + 1
    for l in range(4):
        for g in range(2):
            rows = idx[offsets[l * 2 + g]: offsets[l * 2 + g + 1]]
            assert rows.size == nt + budgets[l]
            assert text <= set(rows.tolist())
            assert np.all(np.diff(rows) > 0)


# ---------------------------------------------------------------- P8
def test_table4_memory_arithmetic():
    """Compacted bytes reproduce the KV memory printed in Table 4 for a
    LLaVA-1.5-7B-sized cache (all tokens evictable, so the vision basis and the
    all-token basis coincide)."""
    path = os.path.join(os.path.dirname(__file__), "golden", "table4_kv_memory.txt")
    rows = [line.split() for line in open(path) if line.strip() and not line.startswith("#")]
    L, H_kv, d = 32, 32, 128
    rng = np.random.default_rng(2)
    for ctx, ratio, printed in rows:
        ctx, ratio, printed = int(ctx), float(ratio), float(printed)
        modality = np.ones(ctx, np.uint8)
        stat = 0.5 + rng.random(L)
        total = oracle.vision_budget_total(ratio, ctx, L)
        budgets = oracle.tvb_budgets(stat, total, ctx)
        # the per-layer budget is shared by every head of the layer, so one
        # head per layer is selected and the bytes scaled by H_kv
        scores = rng.random((L, 1, ctx))
        offsets, _ = oracle.tpr_select(scores, budgets, modality)
        gib = H_kv * oracle.compacted_kv_bytes(offsets, d) / 2.0 ** 30
        assert round(gib, 2) == printed, (ctx, ratio, gib)


# ---------------------------------------------------------------- P9
def test_brute_force_tiny():
    """Eq. 2, 5, 6, 8 summed term by term with scalar Python loops."""
    L, H_q, H_kv, d = 2, 4, 2, 5
    q, k, modality, pos, w = _rand_case(L, H_q, H_kv, d, seed=9)
    scale = 0.41
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, scale, H_kv)
    G = H_q // H_kv
    vrank = {}
    for j, m in enumerate(modality):
        if m == 1:
            vrank[j] = len(vrank)
    bs = np.zeros_like(scores)
    bstat = np.zeros(L)
    for l in range(L):
        for h in range(H_q):
            g = h // G
            for i, p in enumerate(pos):
                logits = []
                for j in range(p + 1):
                    dot = 0.0
                    for c in range(d):
                        dot += q[l, h, i, c] * k[l, g, j, c]
                    logits.append(scale * dot)
                mx = max(logits)
                e = [math.exp(x - mx) for x in logits]
                z = sum(e)
                for j in range(p + 1):
                    if modality[j] == 1:
                        a = e[j] / z
                        bstat[l] += a
                        bs[l, g, vrank[j]] += w[l, i] * a / G
    assert np.allclose(scores, bs, rtol=1e-12, atol=1e-15)
    assert np.allclose(stat, bstat, rtol=1e-12, atol=0)


# ---------------------------------------------------------------- more invariants
def test_gqa_group_mapping_and_mean():
    """A KV head's score is the mean over its own G query heads h // G == g."""
    q, k, modality, pos, w = _rand_case(L=2, H_q=6, H_kv=2, seed=21)
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.6, 2)
    for g in range(2):
        acc = 0.0
        st = 0.0
        for h in range(3 * g, 3 * g + 3):
            s1, t1 = oracle.twr_scores_tvb_stat(q[:, h:h + 1], k[:, g:g + 1], modality, pos,
                                                w, 0.6, 1)
            acc = acc + s1[:, 0]
            st = st + t1
        assert np.allclose(scores[:, g], acc / 3, rtol=1e-12, atol=1e-16)
        if g == 0:
            st0 = st
    assert np.allclose(stat, st0 + st, rtol=1e-12)


def test_key_shift_invariance():
    """Adding one vector to every key shifts each row's logits by a constant,
    which the row softmax removes."""
    q, k, modality, pos, w = _rand_case(seed=4)
    s0, t0 = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.7, 2)
    shift = np.random.default_rng(5).standard_normal(k.shape[-1])
    s1, t1 = oracle.twr_scores_tvb_stat(q, k + shift, modality, pos, w, 0.7, 2)
    assert np.allclose(s0, s1, rtol=1e-10, atol=1e-14)
    assert np.allclose(t0, t1, rtol=1e-10)


def test_scale_folds_into_queries():
    q, k, modality, pos, w = _rand_case(seed=6)
    s0, t0 = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.25, 2)
    s1, t1 = oracle.twr_scores_tvb_stat(q * 0.25, k, modality, pos, w, 1.0, 2)
    assert np.allclose(s0, s1, rtol=1e-12, atol=1e-16)
    assert np.allclose(t0, t1, rtol=1e-12)


def test_causality():
    """Keys after the last query position change nothing; query rows placed
    before the first vision key carry no text-vision mass."""
    segs = (("text", 4), ("vision", 6), ("text", 3), ("vision", 5))
    q, k, modality, pos, w = _rand_case(segments=segs, seed=8)
    pos = np.array([1, 3, 10, 12])
    q = q[:, :, :4]
    w = w[:, :4]
    s0, t0 = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.5, 2)
    k2 = k.copy()
    k2[:, :, 13:] += 3.0
    s1, t1 = oracle.twr_scores_tvb_stat(q, k2, modality, pos, w, 0.5, 2)
    assert np.array_equal(s0, s1) and np.array_equal(t0, t1)
    # the last five vision keys sit after every query row: zero score
    assert np.all(s0[:, :, 9:] == 0.0)
    early = np.array([0, 1, 2, 3])
    _, t_early = oracle.twr_scores_tvb_stat(q, k, modality, early, w, 0.5, 2)
    assert np.all(t_early == 0.0)


def test_linear_in_text_weights():
    q, k, modality, pos, w = _rand_case(seed=10)
    w2 = np.random.default_rng(3).random(w.shape)
    s_a, t_a = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.5, 2)
    s_b, t_b = oracle.twr_scores_tvb_stat(q, k, modality, pos, w2, 0.5, 2)
    s_c, t_c = oracle.twr_scores_tvb_stat(q, k, modality, pos, w + 2.0 * w2, 0.5, 2)
    assert np.allclose(s_c, s_a + 2.0 * s_b, rtol=1e-12, atol=1e-16)
    assert np.array_equal(t_a, t_b) and np.array_equal(t_a, t_c)


def test_widen_bf16_exact():
    bits = np.array([0x3F80, 0xC000, 0x3F81, 0x0001, 0x7F7F, 0x8000], np.uint16)
    vals = oracle.widen_bf16(bits)
    assert vals.tolist() == [1.0, -2.0, 1.0 + 2.0 ** -7, 2.0 ** -133,
                             (2.0 - 2.0 ** -7) * 2.0 ** 127, -0.0]


def test_compact_is_a_row_gather():
    rng = np.random.default_rng(12)
    k = rng.integers(-2 ** 15, 2 ** 15, (2, 3, 9, 4), dtype=np.int64).astype(np.int16)
    v = rng.integers(-2 ** 15, 2 ** 15, (2, 3, 9, 4), dtype=np.int64).astype(np.int16)
    sets = [[0, 2, 5], [1], [], [3, 4, 8], [0, 1, 2, 3, 4, 5, 6, 7, 8], [7]]
    offsets = np.cumsum([0] + [len(s) for s in sets])
    idx = np.array(sum(sets, []), np.int64)
    ko, vo = oracle.compact(k, v, offsets, idx)
    r = 0
    for lg, s in enumerate(sets):
        l, g = divmod(lg, 3)
        for p in s:
            assert np.array_equal(ko[r], k[l, g, p]) and np.array_equal(vo[r], v[l, g, p])
            r += 1
    assert r == ko.shape[0]


def test_evict_end_to_end_tiny():
    wl = synth.WORKLOADS["tiny"]
    inp = synth.generate(wl, seed=0)
    out = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"],
                       inp["w"], 0.25, wl.H_kv)
    assert out["budgets"].tolist() == [16]
    assert out["offsets"][-1] == wl.H_kv * (wl.N_t + 16)
    # with one layer the statistic is the whole TV mass of 8 heads x 32 rows
    assert 0.0 < out["stat"][0] < 8 * 32


def test_rows_normalised_independently_wide_range():
    """Rows whose logits differ by ~1000 are each normalised on their own:
    a row of small logits still sums to one next to a row of huge ones."""
    n, d = 6, 6
    keys = np.eye(d)
    pos = np.array([5, 5])
    q = np.stack([1000.0 * keys[3], 0.01 * keys[1]])
    a = oracle.causal_text_attention(q, keys, pos, 1.0)
    assert np.all(np.isfinite(a))
    assert np.allclose(a.sum(axis=1), 1.0, rtol=0, atol=1e-12)
    assert a[0, 3] > 1.0 - 1e-12
    assert np.all(np.abs(a[1] - 1.0 / 6.0) < 0.01)


# ---------------------------------------------------------------- Eq. 7 / Eq. 9
def _scalar_attention_rows(q, k, pos, scale, l, h, g):
    """A_{l,h}[i, j] for j <= pos[i], by scalar loops (math.exp)."""
    rows = []
    for i, p in enumerate(pos):
        logits = []
        for j in range(p + 1):
            dot = 0.0
            for c in range(q.shape[-1]):
                dot += q[l, h, i, c] * k[l, g, j, c]
            logits.append(scale * dot)
        mx = max(logits)
        e = [math.exp(x - mx) for x in logits]
        z = sum(e)
        rows.append([x / z for x in e])
    return rows


def test_text_scores_and_weights_brute_force_tiny():
    """Eq. 9 and Eq. 7 summed term by term over scalar attention entries."""
    L, H_q, H_kv, d = 2, 4, 2, 5
    q, k, modality, pos, _ = _rand_case(L, H_q, H_kv, d, seed=31)
    scale = 0.53
    ts, wt = oracle.text_scores_and_weights(q, k, modality, pos, scale, H_kv)
    G = H_q // H_kv
    trank = {}
    for j, m in enumerate(modality):
        if m == 0:
            trank[j] = len(trank)
    n_win = len(pos)
    bts = np.zeros_like(ts)
    bw = np.zeros((L, n_win))
    for l in range(L):
        num = [0.0] * n_win
        for h in range(H_q):
            g = h // G
            a = _scalar_attention_rows(q, k, pos, scale, l, h, g)
            for i, p in enumerate(pos):
                for j in range(p + 1):
                    if modality[j] == 0:
                        bts[l, g, trank[j]] += a[i][j] / G
                for jr in range(n_win):              # Eq. 7: rows i >= jr, column pos[jr]
                    if i >= jr:
                        num[jr] += a[i][pos[jr]]
        raw = [num[jr] / H_q / (n_win - jr) for jr in range(n_win)]
        tot = sum(raw)
        bw[l] = [x / tot for x in raw]
    assert np.allclose(ts, bts, rtol=1e-12, atol=1e-15)
    assert np.allclose(wt, bw, rtol=1e-12, atol=1e-15)


def test_text_and_vision_mass_partition_every_row():
    """Each causal row sums to 1 over text and vision keys, so G times the text
    scores of Eq. 9 plus the TV statistic of Eq. 5 give H_q * n_win per layer."""
    q, k, modality, pos, w = _rand_case(L=3, H_q=6, H_kv=3, d=7, seed=32)
    ts, _ = oracle.text_scores_and_weights(q, k, modality, pos, 0.45, 3)
    _, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.45, 3)
    G = 2
    total = G * ts.sum(axis=(1, 2)) + stat
    assert np.allclose(total, 6 * len(pos), rtol=1e-12)


def test_eq7_uniform_attention_closed_form():
    """Q = 0 gives A_ij = 1/(p_i + 1) on every visible key."""
    q, k, modality, pos, _ = _rand_case(L=1, H_q=2, H_kv=1, seed=33)
    q[:] = 0.0
    ts, wt = oracle.text_scores_and_weights(q, k, modality, pos, 1.0, 1)
    text = np.flatnonzero(modality == 0)
    expect_ts = np.array([sum(1.0 / (p + 1) for p in pos if p >= t) for t in text])
    assert np.allclose(ts[0, 0], expect_ts, rtol=1e-13)
    n = len(pos)
    raw = np.array([sum(1.0 / (pos[i] + 1) for i in range(j, n)) / (n - j) for j in range(n)])
    assert np.allclose(wt[0], raw / raw.sum(), rtol=1e-13)


def test_eq7_weights_normalised_and_single_row():
    q, k, modality, pos, _ = _rand_case(L=2, seed=34)
    _, wt = oracle.text_scores_and_weights(q, k, modality, pos, 0.9, 2)
    assert np.allclose(wt.sum(axis=1), 1.0, rtol=1e-14) and np.all(wt > 0)
    q1, k1, m1, p1, _ = _rand_case(L=2, n_win=1, seed=35)
    _, w1 = oracle.text_scores_and_weights(q1, k1, m1, p1, 0.9, 2)
    assert np.array_equal(w1, np.ones((2, 1)))


def test_eq7_dominant_text_token_saturates():
    """Every row attending almost only to the first window token (a dominant
    text token) puts Eq. 7's weight on that row and its Eq. 9 score at n_win."""
    q, k, modality, pos, _ = _rand_case(L=1, H_q=1, H_kv=1, d=6, seed=36)
    u = np.zeros(6)
    u[2] = 1.0
    k[0, 0] = 0.0
    k[0, 0, pos[0]] = u
    q[0, 0] = 60.0 * u
    ts, wt = oracle.text_scores_and_weights(q, k, modality, pos, 1.0, 1)
    trank = int(np.count_nonzero(modality[:pos[0]] == 0))
    assert abs(ts[0, 0, trank] - len(pos)) < 1e-9
    assert wt[0, 0] > 1 - 1e-9


def test_eq7_rejects_rows_on_vision_tokens():
    q, k, modality, pos, _ = _rand_case(seed=37)
    bad = pos.copy()
    bad[0] = int(np.flatnonzero(modality == 1)[0])
    bad.sort()
    with pytest.raises(ValueError):
        oracle.text_scores_and_weights(q, k, modality, bad, 1.0, 2)


# ---------------------------------------------------------------- Eq. 10, both cases
def _brute_select(vs, ts, b, modality, sinks, vision_basis=False):
    vision = [j for j, m in enumerate(modality) if m == 1]
    text = [j for j, m in enumerate(modality) if m == 0]
    if vision_basis or b > len(text):
        cand, sc, slots, keep = vision, vs, (b if vision_basis else b - len(text)), set(text)
    else:
        cand, sc, slots, keep = text, ts, b, set()
    keep |= set(sinks)
    free = [(-sc[r], j) for r, j in enumerate(cand) if j not in sinks]
    slots = max(0, slots - sum(1 for j in cand if j in sinks))
    for _, j in sorted(free)[:slots]:
        keep.add(j)
    return sorted(keep)


@pytest.mark.parametrize("keep", [(0, 0), (4, 1), (2, 3)])
def test_general_select_both_cases_brute_force(keep):
    rng = np.random.default_rng(38)
    modality = np.array([1, 1, 0, 0, 1, 0, 1, 1, 1, 0, 0, 1, 0, 1, 1, 0], np.uint8)
    n_t, n_v = int((modality == 0).sum()), int((modality == 1).sum())
    L, H = 6, 2
    budgets = [0, 3, n_t, n_t + 1, n_t + 5, modality.size]
    vs = rng.integers(0, 4, (L, H, n_v)).astype(np.float64)    # many ties
    ts = rng.integers(0, 4, (L, H, n_t)).astype(np.float64)
    sinks = list(oracle.sink_positions(modality.size, *keep))
    off, idx = oracle.tpr_select_general(vs, ts, budgets, modality, *keep)
    for l in range(L):
        for g in range(H):
            got = idx[off[l * H + g]:off[l * H + g + 1]].tolist()
            assert got == _brute_select(vs[l, g], ts[l, g], budgets[l], modality, sinks)
            if keep == (0, 0):
                assert len(got) == budgets[l]
            if budgets[l] > n_t:
                assert set(np.flatnonzero(modality == 0)) <= set(got)
            elif keep == (0, 0):
                assert all(modality[j] == 0 for j in got)


def test_general_select_vision_basis_is_tpr_select():
    q, k, modality, pos, w = _rand_case(L=3, seed=39)
    scores, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.8, 2)
    budgets = oracle.tvb_budgets(stat, 7, int((modality == 1).sum()))
    a = oracle.tpr_select(scores, budgets, modality)
    b = oracle.tpr_select_general(scores, None, budgets, modality, vision_basis=True)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_table4_memory_all_token_basis_mixed_layout():
    """The main-text setting counts every KV in the ratio (Section 4.3): with
    text and vision mixed, the all-token basis and Eq. 10 keep exactly
    floor(r * N * L + 1/2) rows per head, reproducing Table 4's memory."""
    path = os.path.join(os.path.dirname(__file__), "golden", "table4_kv_memory.txt")
    rows = [line.split() for line in open(path) if line.strip() and not line.startswith("#")]
    L, H_kv, d = 32, 32, 128
    rng = np.random.default_rng(40)
    for ctx, ratio, printed in rows:
        ctx, ratio, printed = int(ctx), float(ratio), float(printed)
        modality = np.zeros(ctx, np.uint8)
        modality[35:35 + 576 * (ctx // 1000)] = 1                # a text prefix, images, a question
        n_t, n_v = int((modality == 0).sum()), int((modality == 1).sum())
        stat = 0.5 + rng.random(L)
        total = oracle.all_budget_total(ratio, ctx, L)
        budgets = oracle.tvb_budgets(stat, total, ctx)
        assert sum(budgets) == total
        vs = rng.random((L, 1, n_v))
        ts = rng.random((L, 1, n_t))
        offsets, _ = oracle.tpr_select_general(vs, ts, budgets, modality)
        gib = H_kv * oracle.compacted_kv_bytes(offsets, d) / 2.0 ** 30
        assert round(gib, 2) == printed, (ctx, ratio, gib)


def test_evict_eq7_and_all_basis_tiny():
    """End to end on the oracle: Eq. 7 weights feed Eq. 8; all-token budgets
    sum to B and each head keeps b_l rows."""
    rng = np.random.default_rng(41)
    L, H_q, H_kv, d, n = 3, 4, 2, 8, 30
    modality = np.zeros(n, np.uint8)
    modality[4:22] = 1
    pos = np.flatnonzero(modality == 0)[-6:]
    qb = rng.integers(-2 ** 15, 2 ** 15, (L, H_q, pos.size, d)).astype(np.int16) & 0x3FFF
    kb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16) & 0x3FFF
    vb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16)
    w = np.full((L, pos.size), 1.0 / pos.size)
    r7 = oracle.evict(qb, kb, vb, modality, pos, w, 0.2, H_kv, weights="eq7")
    q, k = oracle.widen_bf16(qb), oracle.widen_bf16(kb)
    _, w7 = oracle.text_scores_and_weights(q, k, modality, pos, 1 / math.sqrt(d), H_kv)
    s7, _ = oracle.twr_scores_tvb_stat(q, k, modality, pos, w7, 1 / math.sqrt(d), H_kv)
    assert np.array_equal(r7["scores"], s7) and np.array_equal(r7["w"], w7)
    for ratio in (0.1, 0.3, 0.9):
        ra = oracle.evict(qb, kb, vb, modality, pos, w, ratio, H_kv, basis="all")
        assert int(ra["budgets"].sum()) == oracle.all_budget_total(ratio, n, L)
        for l in range(L):
            for g in range(H_kv):
                assert ra["offsets"][l * H_kv + g + 1] - ra["offsets"][l * H_kv + g] == ra["budgets"][l]


# ---------------------------------------------------------------- decode over the compacted cache
def _identity_csr(L, H_kv, n):
    return np.arange(L * H_kv + 1, dtype=np.int64) * n


def test_decode_full_cache_equals_causal_attention_row():
    """With every row kept, decode equals the Eq. 2 attention row of a query
    that sees all N keys, times V (the prefill definition, written separately)."""
    rng = np.random.default_rng(50)
    L, H_q, H_kv, d, n = 2, 6, 2, 8, 13
    q = rng.standard_normal((L, H_q, d))
    k = rng.standard_normal((L, H_kv, n, d))
    v = rng.standard_normal((L, H_kv, n, d))
    o = oracle.decode_attention(q, k.reshape(-1, d), v.reshape(-1, d), _identity_csr(L, H_kv, n),
                                H_kv, 0.37)
    for l in range(L):
        for h in range(H_q):
            a = oracle.causal_text_attention(q[l, h][None], k[l, h // 3], np.array([n - 1]), 0.37)
            assert np.allclose(o[l, h], (a @ v[l, h // 3])[0], rtol=1e-12, atol=1e-14)


def test_decode_uniform_and_saturated_and_empty():
    rng = np.random.default_rng(51)
    d, n = 6, 9
    k = rng.standard_normal((n, d))
    v = rng.standard_normal((n, d))
    off = np.array([0, n, n], np.int64)          # layer 0 head 0 has n rows, head 1 none
    q = np.zeros((1, 2, d))
    o = oracle.decode_attention(q, k, v, off, 2, 1.0)
    assert np.allclose(o[0, 0], v.mean(axis=0), rtol=1e-13)
    assert np.array_equal(o[0, 1], np.zeros(d))
    q[0, 0] = 80.0 * k[4] / np.linalg.norm(k[4]) ** 2 * 1.0
    k2 = k.copy()
    k2[4] *= 3.0
    o = oracle.decode_attention(q, k2, v, off, 2, 1.0)
    assert np.allclose(o[0, 0], v[4], atol=1e-9)


def test_decode_row_order_does_not_matter():
    rng = np.random.default_rng(52)
    L, H_q, H_kv, d = 2, 4, 2, 5
    lens = [3, 7, 1, 4]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    k = rng.standard_normal((off[-1], d))
    v = rng.standard_normal((off[-1], d))
    q = rng.standard_normal((L, H_q, d))
    o = oracle.decode_attention(q, k, v, off, H_kv, 0.8)
    perm = np.concatenate([off[i] + rng.permutation(lens[i]) for i in range(len(lens))])
    o2 = oracle.decode_attention(q, k[perm], v[perm], off, H_kv, 0.8)
    assert np.allclose(o, o2, rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- layer-budget statistics (Table 1a)
def test_tt_statistic_ties_to_text_scores_and_tv():
    """Eq. 5 with x = TT: the text-text mass equals G times the Eq. 9 text scores
    summed, and with the TV mass fills every row (H_q * n_win per layer)."""
    q, k, modality, pos, w = _rand_case(L=3, H_q=6, H_kv=2, d=7, seed=60)
    tt = oracle.tt_statistic(q, k, modality, pos, 0.6, 2)
    ts, _ = oracle.text_scores_and_weights(q, k, modality, pos, 0.6, 2)
    _, tv = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.6, 2)
    assert np.allclose(tt, 3 * ts.sum(axis=(1, 2)), rtol=1e-12)
    assert np.allclose(tt + tv, 6 * len(pos), rtol=1e-12)


def test_vv_statistic_is_tv_with_vision_rows_uniform_closed_form():
    """VV budgeting takes the vision tokens' queries as the rows; under uniform
    attention each vision row i puts |{j in V, j <= p_i}| / (p_i + 1) on vision keys."""
    rng = np.random.default_rng(61)
    modality = np.array([0, 0, 1, 1, 1, 0, 1, 1, 0], np.uint8)
    vpos = np.flatnonzero(modality == 1)
    L, H_q, d = 2, 3, 4
    q = np.zeros((L, H_q, vpos.size, d))
    k = rng.standard_normal((L, H_q, modality.size, d))
    w = np.full((L, vpos.size), 1.0 / vpos.size)
    _, vv = oracle.twr_scores_tvb_stat(q, k, modality, vpos, w, 1.0, H_q)
    per_row = [np.count_nonzero(modality[:p + 1] == 1) / (p + 1) for p in vpos]
    assert np.allclose(vv, H_q * sum(per_row), rtol=1e-13)


def test_evict_budget_statistics():
    rng = np.random.default_rng(62)
    L, H_q, H_kv, d, n = 4, 4, 2, 8, 40
    modality = np.zeros(n, np.uint8)
    modality[6:30] = 1
    pos = np.flatnonzero(modality == 0)[-8:]
    qb = rng.integers(-2 ** 15, 2 ** 15, (L, H_q, pos.size, d)).astype(np.int16) & 0x3FFF
    kb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16) & 0x3FFF
    vb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16)
    w = np.full((L, pos.size), 1.0 / pos.size)
    total = oracle.vision_budget_total(0.3, 24, L)
    ru = oracle.evict(qb, kb, vb, modality, pos, w, 0.3, H_kv, budget_stat="uniform")
    assert ru["budgets"].tolist() == oracle.tvb_budgets(np.zeros(L), total, 24)
    assert max(ru["budgets"]) - min(ru["budgets"]) <= 1
    rt = oracle.evict(qb, kb, vb, modality, pos, w, 0.3, H_kv, budget_stat="tt")
    q, k = oracle.widen_bf16(qb), oracle.widen_bf16(kb)
    tt = oracle.tt_statistic(q, k, modality, pos, 1 / math.sqrt(d), H_kv)
    assert np.array_equal(rt["stat"], tt)
    assert rt["budgets"].tolist() == oracle.tvb_budgets(tt, total, 24)


# ---------------------------------------------------------------- head-adaptive budgets
def test_per_head_tv_statistic_sums_to_layer_statistic():
    q, k, modality, pos, w = _rand_case(L=3, H_q=6, H_kv=3, d=7, seed=70)
    per_head = oracle.tv_statistic_per_head(q, k, modality, pos, 0.5, 3)
    _, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.5, 3)
    assert np.allclose(per_head.sum(axis=1), stat, rtol=1e-12)
    # one KV head per query head: each entry is that head's own TV mass
    one = oracle.tv_statistic_per_head(q[:, :3], k, modality, pos, 0.5, 3)
    for g in range(3):
        _, sg = oracle.twr_scores_tvb_stat(q[:, g:g + 1], k[:, g:g + 1], modality, pos, w, 0.5, 1)
        assert np.allclose(one[:, g], sg, rtol=1e-12)


@pytest.mark.parametrize("basis", ["vision", "all"])
@pytest.mark.parametrize("kind", ["tv", "uniform"])
def test_evict_head_budgets(basis, kind):
    """H_kv * B rows split over the heads; every head keeps its own count."""
    rng = np.random.default_rng(71)
    L, H_q, H_kv, d, n = 3, 4, 2, 8, 36
    modality = np.zeros(n, np.uint8)
    modality[5:28] = 1
    pos = np.flatnonzero(modality == 0)[-6:]
    qb = rng.integers(-2 ** 15, 2 ** 15, (L, H_q, pos.size, d)).astype(np.int16) & 0x3FFF
    kb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16) & 0x3FFF
    vb = rng.integers(-2 ** 15, 2 ** 15, (L, H_kv, n, d)).astype(np.int16)
    w = np.full((L, pos.size), 1.0 / pos.size)
    r = oracle.evict(qb, kb, vb, modality, pos, w, 0.3, H_kv, basis=basis, budget_stat=kind,
                     head_budgets=True)
    b = r["budgets"]
    assert b.shape == (L, H_kv)
    total = (oracle.vision_budget_total(0.3, 23, L) if basis == "vision"
             else oracle.all_budget_total(0.3, n, L))
    assert int(b.sum()) == H_kv * total
    if kind == "uniform":
        assert b.max() - b.min() <= 1
    else:
        q, k = oracle.widen_bf16(qb), oracle.widen_bf16(kb)
        st = oracle.tv_statistic_per_head(q, k, modality, pos, 1 / math.sqrt(d), H_kv)
        assert np.array_equal(r["stat"], st)
    n_t = n - 23
    for l in range(L):
        for g in range(H_kv):
            cnt = r["offsets"][l * H_kv + g + 1] - r["offsets"][l * H_kv + g]
            assert cnt == (n_t + b[l, g] if basis == "vision" else b[l, g])


# ---------------------------------------------------------------- prefill attention and its row statistics
def _prefill_case(L=2, H_q=4, H_kv=2, n=11, d=5, seed=70):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((L, H_q, n, d))
    k = rng.standard_normal((L, H_kv, n, d))
    v = rng.standard_normal((L, H_kv, n, d))
    return q, k, v


def test_prefill_attention_brute_force():
    """Eq. 2 over every row, term by term with scalar exponentials, then A V;
    G = 2, so query heads 2g and 2g+1 read KV head g."""
    q, k, v = _prefill_case()
    L, H_q, n, d = q.shape
    scale = 0.41
    o, bound = oracle.prefill_attention(q, k, v, scale, 2)
    for l in range(L):
        for h in range(H_q):
            g = h // 2
            for i in range(n):
                x = [scale * sum(q[l, h, i, c] * k[l, g, j, c] for c in range(d)) for j in range(i + 1)]
                top = max(x)
                e = [math.exp(t - top) for t in x]
                z = sum(e)
                for c in range(d):
                    ref = sum(e[j] / z * v[l, g, j, c] for j in range(i + 1))
                    mag = sum(e[j] / z * abs(v[l, g, j, c]) for j in range(i + 1))
                    assert abs(o[l, h, i, c] - ref) <= 1e-12 * (1 + abs(ref))
                    assert abs(bound[l, h, i, c] - mag) <= 1e-12 * (1 + mag)


def test_prefill_attention_closed_forms():
    """Rows of A sum to 1: equal value rows come back unchanged.  Q = 0: every
    visible key gets 1/(i + 1), so o_i is the running mean of v_0..v_i."""
    q, k, v = _prefill_case(L=1, H_q=3, H_kv=3, n=9, d=4, seed=71)
    const = np.broadcast_to(np.array([0.5, -2.0, 3.25, 0.0]), v.shape).copy()
    o, bound = oracle.prefill_attention(q, k, const, 0.9, 3)
    assert np.allclose(o, const, rtol=0, atol=1e-14)
    assert np.allclose(bound, np.abs(const), rtol=0, atol=1e-14)
    o, _ = oracle.prefill_attention(np.zeros_like(q), k, v, 0.9, 3)
    running = np.cumsum(v, axis=2) / np.arange(1, 10)[None, None, :, None]
    assert np.allclose(o, running, rtol=1e-13, atol=1e-15)
    # the first token sees only itself
    o, _ = oracle.prefill_attention(q, k, v, 0.9, 3)
    assert np.allclose(o[:, :, 0], v[:, :, 0], rtol=0, atol=1e-15)


def test_prefill_rows_at_query_positions_match_eviction_rows():
    """The prefill rows at the query positions are the eviction step's rows of
    Eq. 2 (the separately written causal_text_attention), times V."""
    q, k, v = _prefill_case(L=2, H_q=6, H_kv=2, n=12, d=4, seed=72)
    pos = np.array([3, 7, 8, 11])
    o, _ = oracle.prefill_attention(q, k, v, 0.7, 2)
    for l in range(2):
        for h in range(6):
            a = oracle.causal_text_attention(q[l, h, pos], k[l, h // 3], pos, 0.7)
            assert np.allclose(o[l, h, pos], a @ v[l, h // 3], rtol=1e-12, atol=1e-14)


def test_row_statistics_closed_form_and_eq5():
    """Q = 0: log2 of p_i + 1 visible unit terms, and the vision share is the
    fraction of vision keys among them.  Random Q: the vision shares summed over
    query heads and rows are the TVB statistic S_l of Eq. 5."""
    q, k, modality, pos, w = _rand_case(L=3, H_q=6, H_kv=2, d=7, seed=73)
    n = modality.size
    rng = np.random.default_rng(74)
    q_all = rng.standard_normal((3, 6, n, 7))
    q_all[:, :, pos] = q                       # the query rows sit at their positions
    lse2, vis = oracle.row_statistics(np.zeros_like(q_all), k, modality, pos, 0.6, 2)
    for i, p in enumerate(pos):
        assert np.allclose(lse2[:, :, i], math.log2(p + 1), rtol=0, atol=1e-13)
        assert np.allclose(vis[:, :, i], np.count_nonzero(modality[: p + 1] == 1) / (p + 1),
                           rtol=1e-13)
    lse2, vis = oracle.row_statistics(q_all, k, modality, pos, 0.6, 2)
    _, stat = oracle.twr_scores_tvb_stat(q, k, modality, pos, w, 0.6, 2)
    assert np.allclose(vis.sum(axis=(1, 2)), stat, rtol=1e-12)
    # lse2 against a direct log-sum-exp of one row
    l, h, i = 1, 4, 2
    x = [0.6 * float(q[l, h, i] @ k[l, h // 3, j]) for j in range(pos[i] + 1)]
    assert abs(lse2[l, h, i] - math.log2(sum(math.exp(t) for t in x))) < 1e-12


# ---------------------------------------------------------------- edges found by planting mistakes
def test_budget_totals_round_half_up_exact():
    """B_V and B are the nearest integer to r N L with halves rounded up,
    checked in exact rational arithmetic on ratios that are binary fractions
    (so r N L is exact in floating point): fractional parts 0, 1/4, 1/2, 3/4."""
    from fractions import Fraction
    for r, n, L in [(0.25, 6, 1), (0.25, 5, 1), (0.25, 7, 1), (0.125, 4, 1), (0.375, 2, 1),
                    (0.0, 100, 32), (1.0, 37, 3), (0.0625, 72, 3), (0.5, 3, 3)]:
        want = math.floor(Fraction(r) * n * L + Fraction(1, 2))
        assert oracle.vision_budget_total(r, n, L) == want, (r, n, L)
        assert oracle.all_budget_total(r, n, L) == want, (r, n, L)


def test_tvb_budget_zero_total_and_layer_exactly_at_cap():
    """A zero total gives zero budgets.  Eq. 5 with stat (3, 1, 5), total 4,
    cap 2, by hand: quotas 4*3/9 = 1.333, 4*1/9 = 0.444, 4*5/9 = 2.222; floors
    1, 0, 2 leave one unit, which goes to the largest fraction (layer 1):
    (1, 1, 2).  Layer 2 sits exactly at the cap, which does not exceed it, so
    nothing is re-split (re-splitting would give (2, 0, 2))."""
    assert oracle.tvb_budgets([0.3, 0.5, 0.2], 0, 10) == [0, 0, 0]
    assert oracle.tvb_budgets([3.0, 1.0, 5.0], 4, 2) == [1, 1, 2]


def test_sink_positions_by_hand():
    """The first keep_first and last keep_last positions, clipped to the
    sequence, as a sorted set."""
    assert oracle.sink_positions(10, 2, 3).tolist() == [0, 1, 7, 8, 9]
    assert oracle.sink_positions(5, 0, 0).tolist() == []
    assert oracle.sink_positions(4, 3, 3).tolist() == [0, 1, 2, 3]
    assert oracle.sink_positions(3, 0, 5).tolist() == [0, 1, 2]
    assert oracle.sink_positions(3, 5, 0).tolist() == [0, 1, 2]
    assert oracle.sink_positions(6, 0, 1).tolist() == [5]


def test_selection_without_sinks_by_default():
    """With default arguments neither the general selection nor the whole step
    keeps sinks: on a layout whose first and last tokens are vision keys with
    the lowest scores, the kept vision keys are exactly the top b by (score
    descending, position ascending), found by a plain sort."""
    modality = np.array([1, 1, 0, 1, 1, 1, 0, 0, 1, 1], np.uint8)
    vision = np.flatnonzero(modality == 1)
    text = np.flatnonzero(modality == 0)
    scores = np.array([[[0.01, 0.5, 0.4, 0.9, 0.3, 0.2, 0.02]]])
    for b in (1, 3, 5):
        _, idx = oracle.tpr_select_general(scores, None, [b], modality, vision_basis=True)
        top = sorted(range(vision.size), key=lambda i: (-scores[0, 0, i], i))[:b]
        assert idx.tolist() == sorted(text.tolist() + vision[top].tolist())
    # the whole step on such a layout: q and k random, the first and last
    # tokens vision; the kept vision keys per head are the top b_l of its scores
    rng = np.random.default_rng(7)
    L, H, d = 2, 2, 8
    modality = np.array([1, 1, 1, 0, 0, 1, 1, 1, 0, 0, 0, 1], np.uint8)
    pos = np.array([8, 9, 10])
    q = synth.to_bf16_bits(rng.standard_normal((L, H, pos.size, d)))
    k = synth.to_bf16_bits(rng.standard_normal((L, H, modality.size, d)))
    v = synth.to_bf16_bits(rng.standard_normal((L, H, modality.size, d)))
    w = np.full((L, pos.size), 1.0 / pos.size)
    ref = oracle.evict(q, k, v, modality, pos, w, 0.4, H)
    vision = np.flatnonzero(modality == 1)
    for l in range(L):
        for g in range(H):
            rows = ref["idx"][ref["offsets"][l * H + g]:ref["offsets"][l * H + g + 1]]
            s = ref["scores"][l, g]
            top = sorted(range(vision.size), key=lambda i: (-s[i], i))[:int(ref["budgets"][l])]
            assert sorted(set(rows.tolist()) & set(vision.tolist())) == sorted(vision[top].tolist())


def test_no_sets_for_no_layers():
    """Zero layers give one offset (0) and no indices."""
    modality = np.array([0, 1, 1, 0], np.uint8)
    off, idx = oracle.tpr_select(np.zeros((0, 2, 2)), [], modality)
    assert off.tolist() == [0] and idx.size == 0
    off, idx = oracle.tpr_select_general(np.zeros((0, 2, 2)), None, [], modality,
                                         vision_basis=True)
    assert off.tolist() == [0] and idx.size == 0


def test_attention_saturates_without_overflow():
    """Logits in the thousands: each softmax row is one-hot on its largest
    logit (the others are e^-1000 or less below it), so the decode output and
    every prefill row equal that key's value row exactly, with no overflow."""
    d, n = 4, 4
    k = np.eye(n, d)[None, None] * 1.0                      # orthonormal keys
    v = np.arange(n * d, dtype=np.float64).reshape(1, 1, n, d) + 1.0
    q = 1000.0 * k[:, :, ::-1].copy()                       # row i aims at key n-1-i
    o, bound = oracle.prefill_attention(q, k, v, 1.0, 1)
    for i in range(n):
        visible = np.arange(i + 1)
        logits = [1000.0 if j == n - 1 - i else 0.0 for j in visible]
        if max(logits) == 0.0:
            want = v[0, 0, :i + 1].mean(axis=0)               # all visible logits equal
        else:
            want = v[0, 0, n - 1 - i]
        np.testing.assert_allclose(o[0, 0, i], want, rtol=0, atol=1e-12)
    out = oracle.decode_attention(q[:, :, 0], k[0, 0], v[0, 0], np.array([0, n]), 1, 1.0)
    np.testing.assert_allclose(out[0, 0], v[0, 0, n - 1], rtol=0, atol=1e-12)
    out = oracle.decode_attention(-q[:, :, 0], k[0, 0], v[0, 0], np.array([0, n]), 1, 1.0)
    np.testing.assert_allclose(out[0, 0], v[0, 0, :n - 1].mean(axis=0), rtol=0, atol=1e-12)


def test_evict_one_sided_sinks_and_row_wiring():
    """The whole step with only first-token or only last-token sinks (vision
    basis), on a layout whose first and last tokens are vision keys: the sink
    is kept and takes one of the head's b_l vision slots, the other b_l - 1
    slots go to the top scores of the remaining vision keys (a plain sort);
    k_out / v_out hold the K / V rows of the kept positions (direct indexing)."""
    rng = np.random.default_rng(11)
    L, H, d = 2, 2, 8
    modality = np.array([1, 1, 1, 0, 0, 1, 1, 1, 0, 0, 0, 1], np.uint8)
    pos = np.array([8, 9, 10])
    q = synth.to_bf16_bits(rng.standard_normal((L, H, pos.size, d)))
    k = synth.to_bf16_bits(rng.standard_normal((L, H, modality.size, d)))
    v = synth.to_bf16_bits(rng.standard_normal((L, H, modality.size, d)))
    w = np.full((L, pos.size), 1.0 / pos.size)
    vision = np.flatnonzero(modality == 1)
    for first, last in ((1, 0), (0, 1)):
        sink = 0 if first else modality.size - 1
        ref = oracle.evict(q, k, v, modality, pos, w, 0.4, H, keep_first=first, keep_last=last)
        for l in range(L):
            b = int(ref["budgets"][l])
            assert b >= 1
            for g in range(H):
                lo, hi = ref["offsets"][l * H + g], ref["offsets"][l * H + g + 1]
                rows = ref["idx"][lo:hi]
                s = ref["scores"][l, g]
                rest = [i for i in range(vision.size) if vision[i] != sink]
                top = sorted(rest, key=lambda i: (-s[i], i))[:b - 1]
                want = sorted([sink] + vision[top].tolist())
                assert sorted(set(rows.tolist()) & set(vision.tolist())) == want, (first, l, g)
                np.testing.assert_array_equal(ref["k_out"][lo:hi], k[l, g][rows])
                np.testing.assert_array_equal(ref["v_out"][lo:hi], v[l, g][rows])
