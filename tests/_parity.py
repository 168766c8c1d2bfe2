"""Shared GPU-vs-oracle comparison helpers for the parity tests.

The CUDA path is driven through the C ABI (via the ctypes binding); the oracle
is evaluated on the same seeded host inputs.  Tolerances:
  * scores and TVB statistic: |gpu - oracle| <= 1e-3 |oracle| + 1e-6 max|oracle|
    (fp32 accumulation against fp64; the 1e-6 floor covers entries that are
    ~0 against the head's largest score);
  * budgets, retained index sets and compacted rows: exact, given the GPU's own
    statistic / scores / indices as the oracle's input (the integer decisions
    are taken in the same precision on both sides);
  * retained sets from the oracle's own fp64 scores: equal wherever the gap
    between the k-th and (k+1)-th oracle score exceeds 1e-3 relative.
"""
import math

import numpy as np
import torch

import oracle

RTOL = 1e-3
FLOOR = 1e-6


def device_inputs(inp, device="cuda"):
    def bf16(a):
        return torch.from_numpy(np.ascontiguousarray(a)).to(device).view(torch.bfloat16)
    return dict(q=bf16(inp["q"]), k=bf16(inp["k"]), v=bf16(inp["v"]),
                modality=torch.from_numpy(inp["modality"]).to(device),
                text_pos=torch.from_numpy(inp["text_pos"].astype(np.int32)).to(device),
                w=torch.from_numpy(np.ascontiguousarray(inp["w"], dtype=np.float32)).to(device))


def run_evict(api, wl, inp, ratio, dev=None):
    desc = api.desc_for_workload(wl)
    dev = dev or device_inputs(inp)
    ws = api.new_workspace(desc)
    out = api.alloc_outputs(desc, ratio)
    api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"],
                    dev["w"], ratio, out, ws)
    status = api.tgvkv_status(ws)
    rows = api.tgvkv_retained_rows(desc, ratio)
    res = dict(scores=out.scores.cpu().numpy(), stat=out.tvb_stat.cpu().numpy(),
               budgets=out.budgets.cpu().numpy().astype(np.int64),
               offsets=out.offsets.cpu().numpy(), idx=out.idx[:rows].cpu().numpy().astype(np.int64),
               k_out=out.k_out[:rows].view(torch.int16).cpu().numpy(),
               v_out=out.v_out[:rows].view(torch.int16).cpu().numpy(), status=status)
    return res


def assert_close(gpu, ref, what, rtol=RTOL, floor=FLOOR):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    if ref.size == 0:
        return
    scale = np.abs(ref).max(axis=-1, keepdims=True) if ref.ndim else np.abs(ref)
    tol = rtol * np.abs(ref) + floor * scale
    err = np.abs(gpu - ref)
    bad = err > tol
    if bad.any():
        i = np.unravel_index(np.argmax(err - tol), err.shape)
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside tolerance; worst at {i}: "
                             f"gpu={gpu[i]!r} oracle={ref[i]!r}")


def oracle_scores(wl, inp, layers):
    """fp64 oracle scores/stat of the given layers: ([len(layers), H_kv, N_v], [len])."""
    scale = 1.0 / math.sqrt(wl.d)
    sc, st = [], []
    for l in layers:
        s, t = oracle.twr_scores_tvb_stat(
            oracle.widen_bf16(inp["q"][l:l + 1]), oracle.widen_bf16(inp["k"][l:l + 1]),
            inp["modality"], inp["text_pos"], inp["w"][l:l + 1].astype(np.float64), scale, wl.H_kv)
        sc.append(s[0])
        st.append(t[0])
    return np.stack(sc), np.array(st)


def check_selection_and_compaction(wl, inp, g, layers, ref_scores=None):
    """Exact checks of select/compact for the given layers, given the GPU's
    scores and budgets; plus the gap rule against the oracle's fp64 scores."""
    H = wl.H_kv
    for n, l in enumerate(layers):
        lo, hi = g["offsets"][l * H], g["offsets"][(l + 1) * H]
        o_off, o_idx = oracle.tpr_select(g["scores"][l:l + 1], g["budgets"][l:l + 1],
                                         inp["modality"])
        assert hi - lo == o_off[-1]
        np.testing.assert_array_equal(g["offsets"][l * H:(l + 1) * H + 1] - lo, o_off)
        np.testing.assert_array_equal(g["idx"][lo:hi], o_idx)
        ko, vo = oracle.compact(inp["k"][l:l + 1], inp["v"][l:l + 1], o_off, o_idx)
        np.testing.assert_array_equal(g["k_out"][lo:hi], ko)
        np.testing.assert_array_equal(g["v_out"][lo:hi], vo)
        if ref_scores is not None:
            gap_rule(ref_scores[n], int(g["budgets"][l]), g["idx"][lo:hi], g["offsets"][l * H:(l + 1) * H + 1] - lo,
                     inp["modality"], g["scores"][l])


def gap_rule(ref, b, idx, off, modality, gpu_scores):
    """Where the oracle's k-th and (k+1)-th scores are separated by more than
    1e-3 relative, the kept vision set must equal the oracle's; otherwise every
    disagreeing key must lie within 1e-3 of the k-th oracle score."""
    vision = np.flatnonzero(modality == 1)
    rank = np.full(modality.size, -1)
    rank[vision] = np.arange(vision.size)
    for g in range(ref.shape[0]):
        rows = idx[off[g]:off[g + 1]]
        kept = set(int(rank[p]) for p in rows if modality[p] == 1)
        order = np.lexsort((np.arange(vision.size), -ref[g]))
        want = set(order[:b].tolist())
        if kept == want:
            continue
        kth = ref[g][order[b - 1]]
        nxt = ref[g][order[b]] if b < vision.size else -np.inf
        assert not (kth - nxt > RTOL * abs(kth)), (
            f"head {g}: retained set differs though the oracle's k-th/k+1-th gap is "
            f"{kth - nxt!r} (k-th {kth!r})")
        for v in kept ^ want:
            assert abs(ref[g][v] - kth) <= RTOL * abs(kth) + 1e-12, (g, v, ref[g][v], kth)


# ---------------------------------------------------------------- every layer
_STAT_CACHE = {}


def oracle_stat_all_layers(wl, inp, seed_key=None):
    """fp64 oracle statistic S_l of every layer, [L]; one spawned process per
    core (never forked: the test process has used the GPU).  Cached per
    workload and seed key."""
    key = (wl.name, seed_key)
    if key in _STAT_CACHE:
        return _STAT_CACHE[key]
    import concurrent.futures as cf
    import multiprocessing as mp
    import os
    scale = 1.0 / math.sqrt(wl.d)
    jobs = [(inp["q"][l], inp["k"][l], inp["modality"], inp["text_pos"], inp["w"][l], scale,
             wl.H_kv) for l in range(wl.L)]
    workers = max(1, min(wl.L, os.cpu_count() or 1))
    import _oracle_workers
    one = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")
    saved = {k: os.environ.get(k) for k in one}
    os.environ.update({k: "1" for k in one})     # one BLAS thread per worker process
    try:
        with cf.ProcessPoolExecutor(workers, mp_context=mp.get_context("spawn")) as ex:
            stat = np.array(list(ex.map(_oracle_workers.layer_stat, jobs)))
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    _STAT_CACHE[key] = stat
    return stat


def budgets_match(gpu_budgets, ref_stat, total, cap, rtol=RTOL):
    """The GPU's budgets against oracle.tvb_budgets on the oracle's fp64
    statistic.  They must be equal, except for layers whose quota (Eq. 5) sits
    within the tolerance of a rounding boundary: a statistic within rtol of the
    oracle's moves each quota by at most about 2 rtol of itself, so a layer may
    differ (by one unit) only where its fractional part is that close to an
    integer or to another layer's fractional part (the largest-remainder cut).
    Returns the layers that differ."""
    gpu = np.asarray(gpu_budgets, np.int64)
    want = np.asarray(oracle.tvb_budgets(ref_stat, total, cap), np.int64)
    assert gpu.sum() == want.sum() == total
    diff = np.flatnonzero(gpu != want)
    if diff.size == 0:
        return []
    stat = np.asarray(ref_stat, np.float64)
    quota = total * stat / stat.sum()
    frac = quota - np.floor(quota)
    tol = 2 * rtol * quota
    for l in diff:
        assert abs(int(gpu[l]) - int(want[l])) == 1, (l, gpu[l], want[l])
        near_int = min(frac[l], 1.0 - frac[l]) <= tol[l]
        near_other = np.any(np.abs(np.delete(frac, l) - frac[l]) <= np.delete(tol, l) + tol[l])
        assert near_int or near_other, (
            f"layer {l}: budget {gpu[l]} != oracle {want[l]} though its quota {quota[l]!r} "
            f"is not within tolerance of a rounding boundary")
    return diff.tolist()
