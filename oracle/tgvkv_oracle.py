"""Plain, slow, fp64 CPU oracle of the TGV-KV eviction step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference arms of ``bench.py`` may import this module.  The
product path (the CUDA library and its Python binding) never calls it and shares
no code with it: not a kernel, helper, table or constant.

What is computed, in the paper's order (Section 3.3, "TGV-KV"):

1. Causal attention rows of the text queries (Eq. 2): for a text query row at
   sequence position p_i, ``A_ij = softmax_j(scale * <q_i, k_j>)`` over the keys
   ``j <= p_i`` (every modality); keys after p_i are masked with -inf.
2. Text-Vision attention (Eq. 6): the columns of those rows that belong to
   vision keys.  This is read as a *slice* of the full causal softmax (the
   paper takes A^(TV) as a block of A_l), not as a softmax restricted to vision
   keys.
3. TVB statistic (Eq. 5 with x = TV): ``S_l = sum_{h,i,j in V} A_ij`` over all
   query heads of layer l.
4. TWR vision score (Eq. 8): ``s_{l,j} = sum_i w~_{l,i} A_ij`` for vision keys
   j, with the caller's normalised text weights w~.  With grouped-query
   attention the score of a KV head is the mean over its G query heads.
5. TVB budgets: the total vision budget ``B_V = floor(r * N_v * L + 1/2)`` is
   split over layers in proportion to S_l (Eq. 5), rounded by largest
   remainder (ties to the lower layer) and capped at N_v with the excess
   re-split over the uncapped layers.
6. TPR retention (Eq. 10, case b_l > N_t, vision-budget basis of Appendix B.3):
   keep every text position and the b_l vision positions with the largest
   score (ties to the lower position), in ascending position order.
7. Compaction: the K and V rows of the retained positions, copied bit for bit.

Beyond that hot path (same file, same conventions):

8. Text scores (Eq. 9): ``s^T_{l,t} = sum_{i} A_{i,t}`` over the query rows
   for every text key t (rows before t contribute 0 through the causal mask),
   per KV head as the mean over its G query heads, like Eq. 8.
9. Derived text weights (Eq. 7): for the query row j (itself a text token at
   position p_j), ``w_{l,j} = sum_{i >= j} A_{i,p_j} / (n_win - j)`` -- the
   column sum of the text-text slice over the rows at or after j, divided by
   their number -- averaged over the H_q query heads of the layer and then
   L1-normalised over j to give w~ (the paper leaves the normalisation
   unstated; the sum is the reading taken here).
10. All-token budget basis: ``B = floor(r * N * L + 1/2)`` rows per head over
   all layers, split by the same Eq. 5 rule with cap N.
11. TPR with both cases of Eq. 10 and sink tokens: if b_l > N_t every text
   position is kept plus the top (b_l - N_t) vision positions by s^V;
   otherwise the top b_l text positions by s^T and no vision.  Sink positions
   (the first ``keep_first`` and last ``keep_last`` tokens, Appendix A.2
   "Implementation Details") are always kept and count against the part of the
   budget of their own modality.

12. Other layer-budget statistics (Table 1a, Eq. 5 with x in {VV, TT}):
   ``S^TT_l = sum_{h,i} sum_{j in T} A_ij`` over the query rows; VV is the TV
   statistic of item 3 computed with the vision tokens' queries as the rows;
   uniform budgeting splits an all-zero statistic.
13. Head-adaptive budgets (an extension: the paper budgets per layer only,
   Section 3.2): the statistic of a (layer, KV head) is the TV mass of its G
   query heads; ``H_kv * B`` rows are split over the L * H_kv heads by the
   same rule (cap N_v, or N under the all-token basis), and each head keeps its
   own budget.
14. Decode over the compacted cache (the consumer of the step, Section 3.1
   "Decode Phase"): a new token's query of head h attends to the retained
   rows of its KV head g = h // G, ``o = softmax(scale * q K_I^T) V_I``; a head
   with no retained row gives 0.
15. Prefill attention and the row statistics it leaves (the producer side of
   the step, Section 3.1 "Prefill Phase" with Eq. 2 over every row): each
   token i attends causally to the keys j <= i, ``o_i = sum_j A_ij v_j``; at
   the query positions p_i the rows' log-normaliser and vision mass
   ``sum_{j in V} A_ij`` are what Eq. 5 / Eq. 6 need, so a prefill that keeps
   them spares the eviction step its own pass over the row statistics.

Floating point: inputs are bf16 bit patterns widened exactly to float64; all
arithmetic is float64.  The paper states no precision.

Parity status: every function here is pinned by the CPU tests in
``tests/test_oracle_pins.py`` (brute force, closed forms, invariants and the
byte arithmetic of Table 4).
"""
from __future__ import annotations

import math

import numpy as np


# --------------------------------------------------------------------------
# input widening
# --------------------------------------------------------------------------
def widen_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16 or int16 storage) -> exact float64 values."""
    u = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# Eq. 2 / Eq. 6: causal attention rows of the text queries
# --------------------------------------------------------------------------
def causal_text_attention(q_rows: np.ndarray, keys: np.ndarray,
                          text_pos: np.ndarray, scale: float) -> np.ndarray:
    """Rows of A = softmax(QK^T + M) for the given text queries (Eq. 2).

    q_rows:   [n_win, d] float64 queries of one head.
    keys:     [N, d] float64 keys of the matching KV head.
    text_pos: [n_win] sequence positions of the query rows.
    Returns A: [n_win, N]; A[i, j] = 0 for j > text_pos[i] (the causal mask M).
    """
    n = keys.shape[0]
    logits = scale * (q_rows @ keys.T)
    visible = np.arange(n)[None, :] <= np.asarray(text_pos)[:, None]
    logits = np.where(visible, logits, -np.inf)
    row_max = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - row_max)
    return e / e.sum(axis=1, keepdims=True)


# --------------------------------------------------------------------------
# Eq. 5 (x = TV), Eq. 6, Eq. 8: TWR scores and the TVB statistic
# --------------------------------------------------------------------------
def twr_scores_tvb_stat(q: np.ndarray, k: np.ndarray, modality: np.ndarray,
                        text_pos: np.ndarray, w: np.ndarray, scale: float,
                        n_kv_heads: int, layers=None):
    """Vision importance scores (Eq. 8) and per-layer TV attention sums (Eq. 5).

    q:        [L, H_q, n_win, d] float64 text queries Q^(T)_l.
    k:        [L, H_kv, N, d] float64 key cache.
    modality: [N] 1 = vision key, 0 = text key.
    text_pos: [n_win] ascending positions of the query rows.
    w:        [L, n_win] float64 normalised text weights w~_l.
    layers:   optional subset of layer indices to evaluate (others stay 0).

    Returns (scores [L, H_kv, N_v], stat [L]):
      scores[l, g, v] = (1/G) sum_{h in group g} sum_i w~_{l,i} A^(TV)_{l,h}[i, v]
      stat[l]         = sum_h sum_i sum_v A^(TV)_{l,h}[i, v]
    where v runs over the vision keys in position order.
    """
    n_layers, n_q_heads = q.shape[0], q.shape[1]
    group = n_q_heads // n_kv_heads
    vision = np.flatnonzero(np.asarray(modality) == 1)
    scores = np.zeros((n_layers, n_kv_heads, vision.size))
    stat = np.zeros(n_layers)
    for l in (range(n_layers) if layers is None else layers):
        for h in range(n_q_heads):
            g = h // group
            a = causal_text_attention(q[l, h], k[l, g], text_pos, scale)
            a_tv = a[:, vision]                      # Eq. 6: slice of A_l
            stat[l] += a_tv.sum()                    # Eq. 5 numerator, x = TV
            scores[l, g] += (w[l] @ a_tv) / group    # Eq. 8, mean over the group
    return scores, stat


# --------------------------------------------------------------------------
# Eq. 9 text scores and Eq. 7 derived text weights
# --------------------------------------------------------------------------
def text_scores_and_weights(q: np.ndarray, k: np.ndarray, modality: np.ndarray,
                            text_pos: np.ndarray, scale: float, n_kv_heads: int,
                            layers=None):
    """Text-key importance (Eq. 9) and the normalised text weights (Eq. 7).

    q, k, modality, text_pos as in twr_scores_tvb_stat; every query row must
    sit on a text token.  Returns (text_scores [L, H_kv, N_t], weights
    [L, n_win]):
      text_scores[l, g, t] = (1/G) sum_{h in g} sum_i A_{l,h}[i, t]        (Eq. 9)
      w_{l,j} = (1/H_q) sum_h sum_{i >= j} A_{l,h}[i, p_j] / (n_win - j)   (Eq. 7)
      weights[l, j] = w_{l,j} / sum_j' w_{l,j'}
    where t runs over the text keys in position order.
    """
    modality = np.asarray(modality)
    text_pos = np.asarray(text_pos)
    if np.any(modality[text_pos] != 0):
        raise ValueError("a query row sits on a vision token")
    n_layers, n_q_heads, n_win = q.shape[0], q.shape[1], q.shape[2]
    group = n_q_heads // n_kv_heads
    text = np.flatnonzero(modality == 0)
    t_scores = np.zeros((n_layers, n_kv_heads, text.size))
    weights = np.zeros((n_layers, n_win))
    rows_at_or_after = n_win - np.arange(n_win)          # |{i : i >= j}|
    for l in (range(n_layers) if layers is None else layers):
        w_sum = np.zeros(n_win)
        for h in range(n_q_heads):
            g = h // group
            a = causal_text_attention(q[l, h], k[l, g], text_pos, scale)
            a_tt = a[:, text]                            # the text-text slice of A_l
            t_scores[l, g] += a_tt.sum(axis=0) / group   # Eq. 9, mean over the group
            w_sum += a[:, text_pos].sum(axis=0)          # Eq. 7 numerators (rows i >= j)
        w = w_sum / n_q_heads / rows_at_or_after
        weights[l] = w / w.sum()
    return t_scores, weights


def tv_statistic_per_head(q: np.ndarray, k: np.ndarray, modality: np.ndarray,
                          text_pos: np.ndarray, scale: float, n_kv_heads: int) -> np.ndarray:
    """[L, H_kv]: the TV mass (Eq. 5, x = TV) of the G query heads of each KV head."""
    n_layers, n_q_heads = q.shape[0], q.shape[1]
    group = n_q_heads // n_kv_heads
    vision = np.flatnonzero(np.asarray(modality) == 1)
    stat = np.zeros((n_layers, n_kv_heads))
    for l in range(n_layers):
        for h in range(n_q_heads):
            a = causal_text_attention(q[l, h], k[l, h // group], text_pos, scale)
            stat[l, h // group] += a[:, vision].sum()
    return stat


def head_budget(budgets, l: int, g: int) -> int:
    """b of head (l, g): budgets is per layer [L] or per head [L, H_kv]."""
    b = np.asarray(budgets)
    return int(b[l]) if b.ndim == 1 else int(b[l, g])


def tt_statistic(q: np.ndarray, k: np.ndarray, modality: np.ndarray, text_pos: np.ndarray,
                 scale: float, n_kv_heads: int) -> np.ndarray:
    """Eq. 5 with x = TT: per layer, the attention mass of the query rows on the
    text keys, summed over every query head."""
    n_layers, n_q_heads = q.shape[0], q.shape[1]
    group = n_q_heads // n_kv_heads
    text = np.flatnonzero(np.asarray(modality) == 0)
    stat = np.zeros(n_layers)
    for l in range(n_layers):
        for h in range(n_q_heads):
            a = causal_text_attention(q[l, h], k[l, h // group], text_pos, scale)
            stat[l] += a[:, text].sum()
    return stat


# --------------------------------------------------------------------------
# TVB: per-layer budgets from the statistic (Eq. 5)
# --------------------------------------------------------------------------
def vision_budget_total(ratio: float, n_vision: int, n_layers: int) -> int:
    """B_V = floor(r * N_v * L + 1/2): vision KV kept over all layers."""
    return int(math.floor(ratio * float(n_vision * n_layers) + 0.5))


def all_budget_total(ratio: float, n_tokens: int, n_layers: int) -> int:
    """B = floor(r * N * L + 1/2): KV rows kept per head over all layers when the
    ratio counts every token (the main-text setting of Table 4)."""
    return int(math.floor(ratio * float(n_tokens * n_layers) + 0.5))


def tvb_budgets(stat, total: int, cap: int) -> list[int]:
    """Split ``total`` vision slots over layers in proportion to ``stat``.

    Eq. 5 gives each layer the fraction stat[l] / sum(stat).  Integer budgets
    take floor(total * fraction) and hand the leftover units, one each, to the
    layers with the largest fractional parts (ties: lower layer).  A layer
    whose budget exceeds ``cap`` (= N_v) is set to ``cap`` and dropped; the
    rest is split again over the remaining layers by the same rule.  With a
    zero statistic everywhere the split is uniform.
    """
    n_layers = len(stat)
    if total < 0 or total > n_layers * cap:
        raise ValueError("total budget outside [0, L * N_v]")
    budgets = [0] * n_layers
    active = list(range(n_layers))
    remaining = total
    while active:
        denom = 0.0
        for l in active:
            denom += float(stat[l])
        quota = {}
        for l in active:
            if denom > 0.0:
                quota[l] = float(remaining) * float(stat[l]) / denom
            else:
                quota[l] = float(remaining) / float(len(active))
        base = {l: int(math.floor(quota[l])) for l in active}
        leftover = remaining - sum(base.values())
        by_fraction = sorted(active, key=lambda l: (-(quota[l] - base[l]), l))
        for l in by_fraction[:leftover]:
            base[l] += 1
        over = [l for l in active if base[l] > cap]
        if not over:
            for l in active:
                budgets[l] = base[l]
            return budgets
        for l in over:
            budgets[l] = cap
            active.remove(l)
            remaining -= cap
    return budgets


# --------------------------------------------------------------------------
# TPR: retained index sets (Eq. 10, case b_l > N_t on the vision basis)
# --------------------------------------------------------------------------
def tpr_select(scores: np.ndarray, budgets, modality: np.ndarray):
    """Retained positions per (layer, KV head) as CSR (offsets, idx).

    scores:  [L, H_kv, N_v] vision scores (any float precision).
    budgets: [L] vision budget b_l of each layer, or [L, H_kv] one per head.
    Each set is all text positions plus the b_l vision positions ranked first
    by (score descending, position ascending), listed in ascending position
    order.  offsets has L*H_kv+1 entries, row-major over (layer, head).
    """
    modality = np.asarray(modality)
    vision = np.flatnonzero(modality == 1)
    text = np.flatnonzero(modality == 0)
    n_layers, n_kv_heads, n_vision = scores.shape
    offsets = [0]
    kept = []
    for l in range(n_layers):
        for g in range(n_kv_heads):
            s = scores[l, g]
            order = np.lexsort((np.arange(n_vision), -s))   # score desc, pos asc
            chosen = vision[order[:head_budget(budgets, l, g)]]
            rows = np.sort(np.concatenate([text, chosen]))
            kept.append(rows)
            offsets.append(offsets[-1] + rows.size)
    idx = np.concatenate(kept).astype(np.int64) if kept else np.zeros(0, np.int64)
    return np.asarray(offsets, dtype=np.int64), idx


def sink_positions(n_tokens: int, keep_first: int, keep_last: int) -> np.ndarray:
    """The always-kept positions: the first keep_first and the last keep_last."""
    first = np.arange(min(keep_first, n_tokens))
    last = np.arange(max(0, n_tokens - keep_last), n_tokens)
    return np.union1d(first, last).astype(np.int64)


def tpr_select_general(v_scores: np.ndarray, t_scores, budgets, modality: np.ndarray,
                       keep_first: int = 0, keep_last: int = 0, vision_basis: bool = False):
    """Retained positions per (layer, KV head) by both cases of Eq. 10, with sinks.

    v_scores: [L, H_kv, N_v] vision scores s^V; t_scores: [L, H_kv, N_t] text
    scores s^T (only read for layers with b_l <= N_t).  budgets: [L] rows b_l
    of each head of layer l over all tokens.
      b_l > N_t:  every text position, plus the (b_l - N_t) top vision positions
      b_l <= N_t: the b_l top text positions, no vision position
    With vision_basis the budgets count vision rows only and the first case
    holds for every layer (b_l vision slots on top of all text; t_scores is not
    read).  Ranking is (score descending, position ascending).  Sinks are kept
    in any case; a sink of the ranked modality takes one of its slots (if slots
    are fewer than sinks, every sink is still kept).  Returns CSR (offsets,
    idx), positions ascending within a head.
    """
    modality = np.asarray(modality)
    vision = np.flatnonzero(modality == 1)
    text = np.flatnonzero(modality == 0)
    n_tokens = modality.size
    sinks = sink_positions(n_tokens, keep_first, keep_last)
    is_sink = np.zeros(n_tokens, bool)
    is_sink[sinks] = True
    n_layers, n_kv_heads = v_scores.shape[0], v_scores.shape[1]
    offsets = [0]
    kept = []
    for l in range(n_layers):
        for g in range(n_kv_heads):
            b = head_budget(budgets, l, g)
            if vision_basis or b > text.size:
                slots = b if vision_basis else b - text.size
                cand, s, always = vision, v_scores[l, g], text
            else:
                cand, s, slots, always = text, t_scores[l, g], b, np.zeros(0, np.int64)
            free = ~is_sink[cand]
            slots = max(0, slots - int(np.count_nonzero(~free)))
            order = np.lexsort((cand[free], -s[free]))          # score desc, pos asc
            chosen = cand[free][order[:slots]]
            rows = np.union1d(np.union1d(always, sinks), chosen)
            kept.append(rows.astype(np.int64))
            offsets.append(offsets[-1] + rows.size)
    idx = np.concatenate(kept) if kept else np.zeros(0, np.int64)
    return np.asarray(offsets, dtype=np.int64), idx


# --------------------------------------------------------------------------
# Compaction of the retained KV
# --------------------------------------------------------------------------
def compact(k_bits: np.ndarray, v_bits: np.ndarray, offsets, idx):
    """Gather K/V rows of the retained positions (bit copies).

    k_bits, v_bits: [L, H_kv, N, d] raw 16-bit storage.
    Returns (k_out, v_out) of shape [offsets[-1], d].
    """
    n_layers, n_kv_heads, _, d = k_bits.shape
    total = int(offsets[-1])
    k_out = np.zeros((total, d), dtype=k_bits.dtype)
    v_out = np.zeros((total, d), dtype=v_bits.dtype)
    for l in range(n_layers):
        for g in range(n_kv_heads):
            lo, hi = int(offsets[l * n_kv_heads + g]), int(offsets[l * n_kv_heads + g + 1])
            rows = idx[lo:hi]
            k_out[lo:hi] = k_bits[l, g, rows]
            v_out[lo:hi] = v_bits[l, g, rows]
    return k_out, v_out


def compacted_kv_bytes(offsets, head_dim: int, elem_bytes: int = 2) -> int:
    """Bytes of the compacted cache: K and V rows of every retained position."""
    return 2 * int(offsets[-1]) * head_dim * elem_bytes


# --------------------------------------------------------------------------
# Decode over the compacted cache
# --------------------------------------------------------------------------
def decode_attention(q: np.ndarray, k_rows: np.ndarray, v_rows: np.ndarray, offsets,
                     n_kv_heads: int, scale: float) -> np.ndarray:
    """One decode step of every layer over the compacted cache.

    q:       [L, H_q, d] float64 queries of the new token.
    k_rows, v_rows: [rows, d] float64 retained keys / values (CSR over (l, g)).
    offsets: [L*H_kv + 1] CSR offsets.
    Returns o [L, H_q, d]: o[l, h] = sum_r softmax_r(scale * <q[l,h], k_r>) v_r over
    the rows r of set (l, h // G); zero for an empty set.
    """
    n_layers, n_q_heads, d = q.shape
    group = n_q_heads // n_kv_heads
    out = np.zeros((n_layers, n_q_heads, d))
    for l in range(n_layers):
        for h in range(n_q_heads):
            lg = l * n_kv_heads + h // group
            lo, hi = int(offsets[lg]), int(offsets[lg + 1])
            if hi == lo:
                continue
            logits = scale * (k_rows[lo:hi] @ q[l, h])
            e = np.exp(logits - logits.max())
            out[l, h] = (e / e.sum()) @ v_rows[lo:hi]
    return out


# --------------------------------------------------------------------------
# Prefill attention over every token, and the row statistics it leaves
# --------------------------------------------------------------------------
def prefill_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
                      n_kv_heads: int):
    """Causal attention of every token of the prefill (Eq. 2 for all N rows,
    then the attention-weighted sum of the value rows).

    q: [L, H_q, N, d] float64 queries of every token; k, v: [L, H_kv, N, d].
    Returns (o, bound), both [L, H_q, N, d], with g = h // G:
      o[l, h, i]     = sum_{j <= i} A_ij v[l, g, j],  A_i = softmax_j(scale <q_i, k_j>)
      bound[l, h, i] = sum_{j <= i} A_ij |v[l, g, j]|  (the size of the terms, which
                       sets how far a rounded computation of o may stray)
    """
    n_layers, n_q_heads, n, _ = q.shape
    group = n_q_heads // n_kv_heads
    visible = np.tril(np.ones((n, n), dtype=bool))     # key j visible from row i iff j <= i
    o = np.zeros_like(q)
    bound = np.zeros_like(q)
    for l in range(n_layers):
        for h in range(n_q_heads):
            g = h // group
            logits = np.where(visible, scale * (q[l, h] @ k[l, g].T), -np.inf)
            e = np.exp(logits - logits.max(axis=1, keepdims=True))
            a = e / e.sum(axis=1, keepdims=True)
            o[l, h] = a @ v[l, g]
            bound[l, h] = a @ np.abs(v[l, g])
    return o, bound


def row_statistics(q: np.ndarray, k: np.ndarray, modality: np.ndarray, text_pos: np.ndarray,
                   scale: float, n_kv_heads: int):
    """The eviction step's per-row quantities at the query positions (Eq. 2, 5, 6).

    q: [L, H_q, N, d] float64 queries of every token; the query row i of the
    step is the token at position p_i = text_pos[i].  k: [L, H_kv, N, d].
    Returns (lse2, vision), both [L, H_q, n_win]:
      lse2[l, h, i]   = log2 sum_{j <= p_i} exp(scale <q_{p_i}, k_j>)
      vision[l, h, i] = sum_{j <= p_i, j vision} A_ij  (the row's share of Eq. 6)
    """
    n_layers, n_q_heads, n, _ = q.shape
    group = n_q_heads // n_kv_heads
    pos = np.asarray(text_pos, dtype=np.int64)
    is_vision = np.asarray(modality) == 1
    lse2 = np.zeros((n_layers, n_q_heads, pos.size))
    vision = np.zeros((n_layers, n_q_heads, pos.size))
    for l in range(n_layers):
        for h in range(n_q_heads):
            logits = scale * (q[l, h, pos] @ k[l, h // group].T)
            logits = np.where(np.arange(n)[None, :] <= pos[:, None], logits, -np.inf)
            top = logits.max(axis=1)
            e = np.exp(logits - top[:, None])
            z = e.sum(axis=1)
            lse2[l, h] = (top + np.log(z)) / math.log(2.0)
            vision[l, h] = e[:, is_vision].sum(axis=1) / z
    return lse2, vision


# --------------------------------------------------------------------------
# the whole step
# --------------------------------------------------------------------------
def evict(q_bits, k_bits, v_bits, modality, text_pos, w, ratio: float,
          n_kv_heads: int, scale: float | None = None, weights: str = "given",
          basis: str = "vision", keep_first: int = 0, keep_last: int = 0,
          budget_stat: str = "tv", head_budgets: bool = False):
    """Score, budget, select and compact, all in float64 on the host.

    weights: "given" uses ``w``; "eq7" derives w~ by Eq. 7 (``w`` is ignored).
    basis:   "vision" -- r counts vision KV and every text KV is kept (case
             b_l > N_t of Eq. 10 throughout); "all" -- r counts every KV and
             Eq. 10 applies per layer with the text scores of Eq. 9.
    budget_stat: the statistic the layer budgets follow: "tv" (the method),
             "tt" or "uniform" (Table 1a); the returned "stat" is the one split.
    head_budgets: split H_kv * B over the (layer, KV head) pairs by their own TV
             mass ("tv") or uniformly; budgets and stat are then [L, H_kv].
    """
    q = widen_bf16(q_bits)
    k = widen_bf16(k_bits)
    d = q.shape[-1]
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    modality = np.asarray(modality)
    n_layers = q.shape[0]
    n_tokens = modality.size
    n_vision = int(np.count_nonzero(modality == 1))
    t_scores = None
    if weights == "eq7" or basis == "all":
        t_scores, w_eq7 = text_scores_and_weights(q, k, modality, text_pos, scale, n_kv_heads)
        if weights == "eq7":
            w = w_eq7
    w = np.asarray(w, dtype=np.float64)
    scores, stat = twr_scores_tvb_stat(q, k, modality, text_pos, w, scale, n_kv_heads)
    if head_budgets:
        if budget_stat == "tt":
            raise ValueError("head budgets follow the TV mass or nothing")
        stat = (np.zeros((n_layers, n_kv_heads)) if budget_stat == "uniform" else
                tv_statistic_per_head(q, k, modality, text_pos, scale, n_kv_heads))
    elif budget_stat == "tt":
        stat = tt_statistic(q, k, modality, text_pos, scale, n_kv_heads)
    elif budget_stat == "uniform":
        stat = np.zeros(n_layers)

    def split(total, cap):
        if not head_budgets:
            return tvb_budgets(stat, total, cap)
        return np.asarray(tvb_budgets(stat.ravel(), n_kv_heads * total, cap)).reshape(
            n_layers, n_kv_heads)

    if basis == "vision":
        total = vision_budget_total(ratio, n_vision, n_layers)
        budgets = split(total, n_vision)
        if keep_first or keep_last:
            offsets, idx = tpr_select_general(scores, None, budgets, modality, keep_first,
                                              keep_last, vision_basis=True)
        else:
            offsets, idx = tpr_select(scores, budgets, modality)
    else:
        total = all_budget_total(ratio, n_tokens, n_layers)
        budgets = split(total, n_tokens)
        offsets, idx = tpr_select_general(scores, t_scores, budgets, modality, keep_first,
                                          keep_last)
    k_out, v_out = compact(k_bits, v_bits, offsets, idx)
    out = dict(scores=scores, stat=stat, budgets=np.asarray(budgets, np.int64),
               offsets=offsets, idx=idx, k_out=k_out, v_out=v_out, w=w)
    if t_scores is not None:
        out["text_scores"] = t_scores
    return out
