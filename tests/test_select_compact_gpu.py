"""tgvkv_select_compact: Eq. 10 selection and the compaction in one call, for
scores and budgets the caller holds.  Every kernel form -- warp per head, CTA
per head, the general form (sinks, the all-token basis) and select-then-compact
for sets too large for shared memory -- against the oracle's sets
(oracle.tpr_select_general, Eq. 10) and gathered rows (oracle.compact), on
continuous and on heavily tied scores; and the capacity check: a set that
would end past the caller's rows writes none of its indices or rows."""
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


# (L, H_kv, d, segments): text runs at both ends and between vision runs
SHAPES = {
    # 512 heads of 265 keys: the warp-per-head kernel
    "warp": (16, 32, 64, [("text", 20), ("vision", 150), ("text", 5), ("vision", 60), ("text", 30)]),
    # 12 heads: the CTA-per-head kernel, both vector widths
    "cta": (3, 4, 128, [("text", 13), ("vision", 150), ("text", 7), ("vision", 61), ("text", 40)]),
    "cta_d64": (2, 3, 64, [("vision", 5), ("text", 9), ("vision", 130), ("text", 3)]),
    # sets too large for one CTA's shared memory: select, then compact
    "split": (2, 2, 64, [("text", 40), ("vision", 23000), ("text", 960)]),
}


def _inputs(name, seed, tied, basis="vision"):
    L, H, d, segs = SHAPES[name]
    modality = np.concatenate([np.full(c, 1 if kind == "vision" else 0, np.uint8) for kind, c in segs])
    N = modality.size
    N_v = int(modality.sum())
    N_t = N - N_v
    rng = np.random.default_rng(seed)
    if tied:   # few distinct values: many keys equal to the threshold
        sc = (rng.integers(1, 9, (L, H, N_v)) / 8.0).astype(np.float32)
        ts = (rng.integers(1, 9, (L, H, N_t)) / 8.0).astype(np.float32)
    else:      # positive, no zeros (so no sign-of-zero question)
        sc = (rng.random((L, H, N_v)) + 1e-3).astype(np.float32)
        ts = (rng.random((L, H, N_t)) + 1e-3).astype(np.float32)
    cap = N if basis == "all" else N_v
    budgets = rng.integers(0, cap + 1, L).astype(np.int32)
    budgets[0] = min(cap, 3)           # a small set and, for L > 1, others of any size
    k = rng.integers(-2 ** 15, 2 ** 15, (L, H, N, d)).astype(np.int16)
    v = rng.integers(-2 ** 15, 2 ** 15, (L, H, N, d)).astype(np.int16)
    return dict(L=L, H=H, d=d, N=N, N_v=N_v, N_t=N_t, modality=modality, sc=sc, ts=ts,
                budgets=budgets, k=k, v=v)


def _oracle(x, basis, keep):
    off, idx = oracle.tpr_select_general(x["sc"].astype(np.float64), x["ts"].astype(np.float64),
                                         x["budgets"], x["modality"], keep[0], keep[1],
                                         vision_basis=(basis == "vision"))
    ko, vo = oracle.compact(x["k"], x["v"], off, idx)
    return off, idx, ko, vo


def _run(api, x, basis, keep, capacity, guard=16):
    desc = api.make_desc(x["L"], x["H"], x["H"], x["d"], x["N"], x["N_v"], 1, basis=basis,
                         keep_first=keep[0], keep_last=keep[1])
    ws = api.new_workspace(desc)
    LH = x["L"] * x["H"]
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    off = torch.full((LH + 1,), -7, dtype=torch.int64, device="cuda")
    idx = torch.full((capacity + guard,), -5, dtype=torch.int32, device="cuda")
    ko = torch.full((capacity + guard, x["d"]), 0x5A5A, dtype=torch.int16, device="cuda")
    vo = torch.full((capacity + guard, x["d"]), 0x5A5A, dtype=torch.int16, device="cuda")
    api.tgvkv_select_compact(desc, dev(x["sc"]), dev(x["ts"]), dev(x["budgets"]),
                             dev(x["modality"]), dev(x["k"]).view(torch.bfloat16),
                             dev(x["v"]).view(torch.bfloat16), off, idx[:capacity],
                             ko[:capacity].view(torch.bfloat16), vo[:capacity].view(torch.bfloat16), ws)
    return (desc, api.tgvkv_status(ws), off.cpu().numpy(), idx.cpu().numpy(), ko.cpu().numpy(),
            vo.cpu().numpy())


CASES = [("warp", "vision", (0, 0)), ("cta", "vision", (0, 0)), ("cta_d64", "vision", (0, 0)),
         ("split", "vision", (0, 0)), ("warp", "vision", (4, 1)), ("cta", "all", (4, 1)),
         ("cta_d64", "all", (0, 0)), ("split", "all", (8, 5))]


@pytest.mark.parametrize("tied", [False, True])
@pytest.mark.parametrize("name,basis,keep", CASES)
def test_select_compact_matches_oracle(api, name, basis, keep, tied):
    x = _inputs(name, 11, tied, basis)
    r_off, r_idx, r_ko, r_vo = _oracle(x, basis, keep)
    total = int(r_off[-1])
    desc, status, off, idx, ko, vo = _run(api, x, basis, keep, capacity=total)
    assert status == 0
    np.testing.assert_array_equal(off, r_off)
    np.testing.assert_array_equal(idx[:total], r_idx)
    np.testing.assert_array_equal(ko[:total], r_ko)
    np.testing.assert_array_equal(vo[:total], r_vo)
    # nothing written past the capacity
    assert np.all(idx[total:] == -5) and np.all(ko[total:] == 0x5A5A) and np.all(vo[total:] == 0x5A5A)
    general = basis == "all" or keep != (0, 0)
    want = 2 if name == "split" else 1
    assert api.tgvkv_select_compact_launches(desc) == want, (name, general)


@pytest.mark.parametrize("name,basis,keep", [("warp", "vision", (0, 0)), ("cta", "vision", (0, 0)),
                                             ("cta", "all", (4, 1)), ("split", "vision", (0, 0))])
def test_select_compact_capacity(api, name, basis, keep):
    """Capacity short of the sets: TGVKV_STATUS_INDEX; offsets in full; the
    sets that end within the capacity exact; no index or row of a set that
    does not fit, and nothing past the capacity."""
    x = _inputs(name, 12, False, basis)
    r_off, r_idx, r_ko, r_vo = _oracle(x, basis, keep)
    LH = x["L"] * x["H"]
    # cut inside the middle set, so that sets on both sides of the cut exist
    mid = LH // 2
    capacity = int(r_off[mid] + (r_off[mid + 1] - r_off[mid]) // 2)
    if r_off[mid + 1] == r_off[mid]:
        capacity = int(r_off[mid])
    _, status, off, idx, ko, vo = _run(api, x, basis, keep, capacity=capacity)
    assert status & 0x08
    np.testing.assert_array_equal(off, r_off)
    fit = int(np.searchsorted(r_off, capacity, side="right")) - 1   # sets [0, fit) end within
    end = int(r_off[fit])
    assert end <= capacity
    np.testing.assert_array_equal(idx[:end], r_idx[:end])
    np.testing.assert_array_equal(ko[:end], r_ko[:end])
    np.testing.assert_array_equal(vo[:end], r_vo[:end])
    assert np.all(idx[end:] == -5)
    assert np.all(ko[end:] == 0x5A5A) and np.all(vo[end:] == 0x5A5A)


def test_select_compact_matches_evict_tail(api):
    """On a full evict's own scores and budgets the call reproduces the
    evict's sets and rows (the same kernels, the same inputs)."""
    wl = synth.WORKLOADS["llava15"]
    wl = synth.custom("mini_llava", 4, 8, 8, 128, list(wl.segments), ratios=(0.05,))
    inp = synth.generate(wl, seed=3)
    desc = api.desc_for_workload(wl)
    ws = api.new_workspace(desc)
    dev = P.device_inputs(inp)
    out = api.alloc_outputs(desc, 0.05)
    api.tgvkv_evict(desc, dev["q"], dev["k"], dev["v"], dev["modality"], dev["text_pos"],
                    dev["w"], 0.05, out, ws)
    rows = api.tgvkv_retained_rows(desc, 0.05)
    off = torch.empty_like(out.offsets)
    idx = torch.empty_like(out.idx)
    ko = torch.empty_like(out.k_out)
    vo = torch.empty_like(out.v_out)
    api.tgvkv_select_compact(desc, out.scores, None, out.budgets, dev["modality"], dev["k"],
                             dev["v"], off, idx, ko, vo, ws)
    assert api.tgvkv_status(ws) == 0
    n = int(out.offsets[-1].item())
    assert n <= rows
    assert torch.equal(off, out.offsets)
    assert torch.equal(idx[:n], out.idx[:n])
    assert torch.equal(ko[:n].view(torch.int16), out.k_out[:n].view(torch.int16))
    assert torch.equal(vo[:n].view(torch.int16), out.v_out[:n].view(torch.int16))


@pytest.mark.parametrize("name", ["cta", "cta_d64", "warp"])
@pytest.mark.parametrize("extra", [0, -1, 1])
def test_select_ties_at_the_threshold(api, name, extra):
    """Scores of three values in known counts.  With b = #(score >= 2) every
    key equal to the threshold is kept (the kernels' no-tie emission); with
    b - 1 or b + 1 the keys equal to the threshold (2, or 1) must be broken by
    position (the tie-breaking emission).  Against the oracle's Eq. 10 sets."""
    x = _inputs(name, 13, False)
    rng = np.random.default_rng(14)
    L, H, N_v = x["L"], x["H"], x["N_v"]
    sc = rng.choice(np.array([1.0, 2.0, 3.0], np.float32), size=(L, H, N_v), p=[0.6, 0.3, 0.1])
    sc[:, :, 0] = 2.0                          # at least one key at the threshold in every head
    x["sc"] = sc.astype(np.float32)
    # one budget per layer, from the head with the fewest keys >= 2 (every head can fill it)
    ge2 = (sc >= 2.0).sum(axis=2).min(axis=1)
    x["budgets"] = np.clip(ge2 + extra, 0, N_v).astype(np.int32)
    r_off, r_idx, r_ko, r_vo = _oracle(x, "vision", (0, 0))
    total = int(r_off[-1])
    _, status, off, idx, ko, vo = _run(api, x, "vision", (0, 0), capacity=total)
    assert status == 0
    np.testing.assert_array_equal(off, r_off)
    np.testing.assert_array_equal(idx[:total], r_idx)
    np.testing.assert_array_equal(ko[:total], r_ko)
    np.testing.assert_array_equal(vo[:total], r_vo)


@pytest.mark.parametrize("name", ["cta", "warp", "split"])
def test_select_compact_head_budgets(api, name):
    """One budget per (layer, KV head) (the head-adaptive option): the sets of
    Eq. 10 with each head's own b, against the oracle."""
    x = _inputs(name, 15, False)
    rng = np.random.default_rng(16)
    L, H, N_v = x["L"], x["H"], x["N_v"]
    hb = rng.integers(0, N_v + 1, (L, H)).astype(np.int32)
    hb[0, 0] = 0
    hb[-1, -1] = N_v
    off_r, idx_r = oracle.tpr_select_general(x["sc"].astype(np.float64), x["ts"].astype(np.float64),
                                             hb, x["modality"], 0, 0, vision_basis=True)
    ko_r, vo_r = oracle.compact(x["k"], x["v"], off_r, idx_r)
    total = int(off_r[-1])
    desc = api.make_desc(L, H, H, x["d"], x["N"], N_v, 1, head_budgets=True)
    ws = api.new_workspace(desc)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    off = torch.empty(L * H + 1, dtype=torch.int64, device="cuda")
    idx = torch.empty(total, dtype=torch.int32, device="cuda")
    ko = torch.empty((total, x["d"]), dtype=torch.int16, device="cuda")
    vo = torch.empty_like(ko)
    api.tgvkv_select_compact(desc, dev(x["sc"]), None, dev(hb.reshape(-1)), dev(x["modality"]),
                             dev(x["k"]).view(torch.bfloat16), dev(x["v"]).view(torch.bfloat16),
                             off, idx, ko.view(torch.bfloat16), vo.view(torch.bfloat16), ws)
    assert api.tgvkv_status(ws) == 0
    np.testing.assert_array_equal(off.cpu().numpy(), off_r)
    np.testing.assert_array_equal(idx.cpu().numpy(), idx_r)
    np.testing.assert_array_equal(ko.cpu().numpy(), ko_r)
    np.testing.assert_array_equal(vo.cpu().numpy(), vo_r)
