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
   paper slices A^(TV) "out of A_l"), not as a softmax restricted to vision
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
# TVB: per-layer budgets from the statistic (Eq. 5)
# --------------------------------------------------------------------------
def vision_budget_total(ratio: float, n_vision: int, n_layers: int) -> int:
    """B_V = floor(r * N_v * L + 1/2): vision KV kept over all layers."""
    return int(math.floor(ratio * float(n_vision * n_layers) + 0.5))


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
    budgets: [L] vision budget b_l of each layer.
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
            chosen = vision[order[:int(budgets[l])]]
            rows = np.sort(np.concatenate([text, chosen]))
            kept.append(rows)
            offsets.append(offsets[-1] + rows.size)
    idx = np.concatenate(kept).astype(np.int64) if kept else np.zeros(0, np.int64)
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
# the whole step
# --------------------------------------------------------------------------
def evict(q_bits, k_bits, v_bits, modality, text_pos, w, ratio: float,
          n_kv_heads: int, scale: float | None = None):
    """Score, budget, select and compact, all in float64 on the host."""
    q = widen_bf16(q_bits)
    k = widen_bf16(k_bits)
    d = q.shape[-1]
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    w = np.asarray(w, dtype=np.float64)
    scores, stat = twr_scores_tvb_stat(q, k, modality, text_pos, w, scale, n_kv_heads)
    n_layers = q.shape[0]
    n_vision = int(np.count_nonzero(np.asarray(modality) == 1))
    total = vision_budget_total(ratio, n_vision, n_layers)
    budgets = tvb_budgets(stat, total, n_vision)
    offsets, idx = tpr_select(scores, budgets, modality)
    k_out, v_out = compact(k_bits, v_bits, offsets, idx)
    return dict(scores=scores, stat=stat, budgets=np.asarray(budgets, np.int64),
                offsets=offsets, idx=idx, k_out=k_out, v_out=v_out)
