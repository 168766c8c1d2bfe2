"""C-ABI surface checks that need no GPU: the library builds and loads, every
function declared in include/tgvkv.h is exported, host-side validation rejects
bad arguments before any launch, and the host-side budget arithmetic agrees
with the oracle."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2606_03075_gb300 import synth


@pytest.fixture(scope="module")
def lib(repo_root):
    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import _lib
    return _lib.load()


def _declared(repo_root):
    src = open(os.path.join(repo_root, "include", "tgvkv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tgvkv_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib, repo_root):
    from paper_2606_03075_gb300 import _lib
    names = _declared(repo_root)
    assert len(names) >= 11
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(_lib.SIGNATURES) == names


def _desc(**kw):
    from paper_2606_03075_gb300 import _lib
    base = dict(L=2, H_q=4, H_kv=2, d=128, N=100, N_v=60, n_win=8, softmax_scale=0.0,
                w_layer_stride=8)
    base.update(kw)
    return _lib.Desc(**base)


def test_validation_rejects_before_launch(lib):
    P = ctypes.c_void_p
    fake = P(0x1000)        # never dereferenced: every call below fails validation
    odd = P(0x1008)         # 8-byte aligned only
    d = _desc()
    ref = ctypes.byref

    def score(desc, q=fake, k=fake, ws=fake):
        return lib.tgvkv_score(desc, q, k, fake, fake, fake, fake, fake, ws, None)

    assert score(None) == 1
    assert score(ref(_desc(d=96))) == 2
    assert score(ref(_desc(H_q=3))) == 1
    assert score(ref(_desc(N_v=101))) == 1
    assert score(ref(_desc(N=70000, N_v=10))) == 2
    assert score(ref(d), q=P(0)) == 1
    assert score(ref(d), k=odd) == 1
    assert score(ref(d), ws=odd) == 1
    assert b"16-byte" in lib.tgvkv_last_error()
    assert lib.tgvkv_budget(ref(d), fake, 1.5, fake, fake, None) == 1
    assert lib.tgvkv_budget(ref(d), fake, -0.1, fake, fake, None) == 1
    assert lib.tgvkv_budget(ref(d), fake, float("nan"), fake, fake, None) == 1
    assert lib.tgvkv_select(ref(d), fake, fake, fake, fake, P(0), fake, None) == 1
    assert lib.tgvkv_compact(ref(d), fake, fake, fake, fake, odd, fake, 10, fake, None) == 1
    assert lib.tgvkv_compact(ref(d), fake, fake, fake, fake, fake, fake, -1, fake, None) == 1
    assert lib.tgvkv_evict(ref(d), fake, fake, fake, fake, fake, fake, 2.0, fake, fake, fake,
                           fake, fake, fake, fake, fake, None) == 1
    assert lib.tgvkv_workspace_size(ref(_desc(d=32))) == 0
    assert lib.tgvkv_retained_rows(ref(d), 1.01) == -1
    assert lib.tgvkv_status(None, None) < 0


def test_descriptor_limits(lib):
    """The size limits include/tgvkv.h states, at and just past each bound
    (tgvkv_workspace_size is 0 exactly when a descriptor is rejected)."""
    def ws(**kw):
        return lib.tgvkv_workspace_size(ctypes.byref(_desc(**kw)))

    assert ws(N=32768, N_v=32600) > 0
    assert ws(N=32769, N_v=32600) == 0
    assert ws(L=1024) > 0
    assert ws(L=1025) == 0
    assert ws(H_q=256, H_kv=1, n_win=128, w_layer_stride=128) > 0      # G * n_win = 32768
    assert ws(H_q=257, H_kv=1, n_win=128, w_layer_stride=128) == 0
    assert ws(L=255, H_q=257, H_kv=257) > 0                            # L * H_kv = 65535
    assert ws(L=256, H_q=256, H_kv=256) == 0
    assert ws(L=32, H_q=32, H_kv=32, head_budgets=1) > 0               # 1024 heads
    assert ws(L=33, H_q=32, H_kv=32, head_budgets=1) == 0
    assert ws(d=64) > 0 and ws(d=128) > 0
    for bad in (dict(d=32), dict(d=256), dict(L=0), dict(H_kv=0), dict(N=0), dict(N_v=-1),
                dict(N_v=101), dict(n_win=-1), dict(H_q=6, H_kv=4), dict(budget_basis=2),
                dict(weight_mode=2), dict(budget_stat=3), dict(head_budgets=2),
                dict(keep_first=-1), dict(head_budgets=1, budget_stat=1)):
        assert ws(**bad) == 0, bad
    assert ws(n_win=0) > 0 and ws(N_v=0) > 0 and ws(N_v=100) > 0


def test_descriptor_edges_accepted_and_bad_scales_rejected(lib):
    """The smallest valid shapes, a shared weight row and a cache of more than
    2^30 key rows pass validation; a negative weight stride and a softmax scale
    that is not finite are rejected (a scale <= 0 means 1/sqrt(d))."""
    def ws(**kw):
        return lib.tgvkv_workspace_size(ctypes.byref(_desc(**kw)))

    assert ws(H_q=1, H_kv=1) > 0
    assert ws(N=1, N_v=0) > 0 and ws(N=1, N_v=1) > 0
    assert ws(w_layer_stride=0) > 0
    assert ws(w_layer_stride=-1) == 0
    assert ws(L=255, H_q=257, H_kv=257, N=32768, N_v=100) > 0   # 2147450880 K rows
    assert ws(L=255, H_q=257, H_kv=257, n_win=32768, w_layer_stride=32768) > 0   # Q rows alike
    for bad in (float("nan"), float("inf"), float("-inf")):
        assert ws(softmax_scale=bad) == 0, bad
    assert ws(softmax_scale=-1.0) > 0 and ws(softmax_scale=0.0) > 0


def test_host_budget_arithmetic_matches_oracle(lib):
    ref = ctypes.byref
    for name, wl in synth.WORKLOADS.items():
        d = _desc(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                  w_layer_stride=wl.n_win)
        for r in (0.0, 0.05, 0.1, 0.2, 0.25, 0.5, 1.0) + tuple(wl.ratios):
            bv = oracle.vision_budget_total(r, wl.N_v, wl.L)
            assert lib.tgvkv_vision_budget_total(ref(d), r) == bv
            assert lib.tgvkv_retained_rows(ref(d), r) == wl.H_kv * (wl.L * wl.N_t + bv)
        assert lib.tgvkv_workspace_size(ref(d)) > 0
    rng = np.random.default_rng(3)
    for _ in range(300):
        L, nv = int(rng.integers(1, 64)), int(rng.integers(0, 5000))
        r = float(rng.random())
        d = _desc(L=L, N=nv + 5, N_v=nv)
        assert lib.tgvkv_vision_budget_total(ref(d), r) == oracle.vision_budget_total(r, nv, L)


def test_evict_launch_count(lib):
    """tgvkv_evict launches the score kernel (which also derives the layer
    budgets) and one fused select/gather kernel; select and compact run
    separately when the fused kernel's tables would not fit shared memory;
    without query rows the budget kernel replaces the score kernel."""
    ref = ctypes.byref
    for wl in synth.WORKLOADS.values():
        d = _desc(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                  w_layer_stride=wl.n_win)
        assert lib.tgvkv_evict_launches(ref(d)) == 2, wl.name
    assert lib.tgvkv_evict_launches(ref(_desc(N=32000, N_v=31000))) == 3
    assert lib.tgvkv_evict_launches(ref(_desc(n_win=0))) == 2
    assert lib.tgvkv_evict_launches(ref(_desc(d=32))) == -1
    assert lib.tgvkv_evict_launches(None) == -1


def test_all_basis_and_sink_arithmetic_matches_oracle(lib):
    """The all-token basis shares out floor(r * N * L + 1/2) rows; sinks add at
    most one row per sink to each (layer, head) set."""
    ref = ctypes.byref
    for wl in synth.WORKLOADS.values():
        base = dict(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                    w_layer_stride=wl.n_win)
        d_all = _desc(**base, budget_basis=1)
        d_snk = _desc(**base, keep_first=4, keep_last=1)
        for r in (0.0, 0.05, 0.2, 1.0):
            b = oracle.all_budget_total(r, wl.N, wl.L)
            assert lib.tgvkv_budget_total(ref(d_all), r) == b
            assert lib.tgvkv_retained_rows(ref(d_all), r) == wl.H_kv * b
            bv = oracle.vision_budget_total(r, wl.N_v, wl.L)
            assert lib.tgvkv_budget_total(ref(d_snk), r) == bv
            assert lib.tgvkv_retained_rows(ref(d_snk), r) == wl.H_kv * (wl.L * (wl.N_t + 5) + bv)
    assert lib.tgvkv_budget_total(ref(_desc(budget_basis=2)), 0.1) == -1
    assert lib.tgvkv_budget_total(ref(_desc(weight_mode=3)), 0.1) == -1
    assert lib.tgvkv_budget_total(ref(_desc(keep_first=-1)), 0.1) == -1


def test_evict_launch_count_with_text_pass(lib):
    """Eq. 7 weights add the text-key score pass and the weights kernel; the
    all-token basis adds the text-key pass (its Eq. 9 scores feed Eq. 10)."""
    ref = ctypes.byref
    for wl in synth.WORKLOADS.values():
        base = dict(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                    w_layer_stride=wl.n_win)
        assert lib.tgvkv_evict_launches(ref(_desc(**base, weight_mode=1))) == 4, wl.name
        assert lib.tgvkv_evict_launches(ref(_desc(**base, budget_basis=1))) == 3, wl.name
        assert lib.tgvkv_evict_launches(ref(_desc(**base, budget_basis=1, weight_mode=1))) == 4
        assert lib.tgvkv_evict_launches(ref(_desc(**base, keep_first=4, keep_last=1))) == 2


def test_select_compact_launch_count_and_validation(lib):
    """tgvkv_select_compact: the one fused kernel wherever tgvkv_evict uses it
    (select then compact for sets too large for shared memory), and host-side
    rejection of a negative capacity and of missing or misaligned buffers."""
    ref = ctypes.byref
    for wl in synth.WORKLOADS.values():
        d = _desc(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                  w_layer_stride=wl.n_win)
        assert lib.tgvkv_select_compact_launches(ref(d)) == 1, wl.name
        assert lib.tgvkv_select_compact_launches(ref(_desc(**{**dict(
            L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
            w_layer_stride=wl.n_win), "keep_first": 4, "keep_last": 1}))) == 1, wl.name
    assert lib.tgvkv_select_compact_launches(ref(_desc(N=32000, N_v=31000))) == 2
    assert lib.tgvkv_select_compact_launches(ref(_desc(d=32))) == -1
    assert lib.tgvkv_select_compact_launches(None) == -1
    P = ctypes.c_void_p
    fake, odd = P(0x1000), P(0x1008)   # never dereferenced: each call fails validation

    def call(cap=16, k=fake, k_out=fake, ws=fake, scores=fake):
        return lib.tgvkv_select_compact(ref(_desc()), scores, None, fake, fake, k, fake, fake,
                                        fake, k_out, fake, cap, ws, None)

    assert call(cap=-1) == 1
    assert call(k=odd) == 1 and call(k_out=odd) == 1
    assert call(ws=None) == 1 and call(scores=None) == 1


def test_decode_launch_count(lib):
    """Two decode kernels for every shape: the row streams, then the merge of
    the sets they split (launched as a programmatic dependent)."""
    ref = ctypes.byref
    for name, wl in synth.WORKLOADS.items():
        d = _desc(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                  w_layer_stride=wl.n_win)
        assert lib.tgvkv_decode_launches(ref(d)) == 2, name
    assert lib.tgvkv_decode_launches(ref(_desc(d=48))) == -1


def test_budget_statistic_modes(lib):
    """TT budgeting runs the text-key pass (one more launch); uniform does not;
    an unknown statistic is rejected."""
    ref = ctypes.byref
    wl = synth.WORKLOADS["llava15"]
    base = dict(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                w_layer_stride=wl.n_win)
    assert lib.tgvkv_evict_launches(ref(_desc(**base, budget_stat=1))) == 3
    assert lib.tgvkv_evict_launches(ref(_desc(**base, budget_stat=2))) == 2
    assert lib.tgvkv_evict_launches(ref(_desc(**base, budget_stat=3))) == -1


def test_head_budget_options(lib):
    ref = ctypes.byref
    wl = synth.WORKLOADS["llava15"]
    base = dict(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                w_layer_stride=wl.n_win)
    # same capacity as per-layer budgets: H_kv * B rows are shared out either way
    for r in (0.05, 0.2):
        assert (lib.tgvkv_retained_rows(ref(_desc(**base, head_budgets=1)), r) ==
                lib.tgvkv_retained_rows(ref(_desc(**base)), r))
    assert lib.tgvkv_evict_launches(ref(_desc(**base, head_budgets=1))) == 2
    assert lib.tgvkv_evict_launches(ref(_desc(**base, head_budgets=1, budget_stat=1))) == -1
    assert lib.tgvkv_evict_launches(ref(_desc(**base, head_budgets=2))) == -1
    big = dict(base, L=64, H_q=32, H_kv=32)            # 2048 heads
    assert lib.tgvkv_evict_launches(ref(_desc(**big, head_budgets=1))) == -1


def test_prefill_and_given_statistics_validation(lib):
    """tgvkv_prefill / tgvkv_evict_with_stats reject bad arguments on the host:
    null or misaligned buffers, an unsupported head size, a bad ratio."""
    P = ctypes.c_void_p
    fake = P(0x1000)
    odd = P(0x1008)
    d = _desc()
    ref = ctypes.byref

    def prefill(desc, q=fake, o=fake, q_text=fake, stats=fake, text_pos=fake):
        return lib.tgvkv_prefill(desc, q, fake, fake, fake, text_pos, o, q_text, stats, fake, None)

    assert prefill(None) == 1
    assert prefill(ref(_desc(d=96))) == 2
    assert prefill(ref(d), q=P(0)) == 1
    assert prefill(ref(d), o=odd) == 1
    assert prefill(ref(d), q_text=odd) == 1
    assert prefill(ref(d), stats=P(0)) == 1
    assert prefill(ref(d), text_pos=P(0)) == 1
    assert b"text_pos" in lib.tgvkv_last_error()

    def evict_stats(desc, stats=fake, ratio=0.1):
        return lib.tgvkv_evict_with_stats(desc, fake, fake, fake, fake, fake, fake, ratio, stats,
                                          fake, fake, fake, fake, fake, fake, fake, fake, None)

    assert evict_stats(ref(d), stats=P(0)) == 1
    assert b"row_stats" in lib.tgvkv_last_error()
    assert evict_stats(ref(d), ratio=1.5) == 1


def test_binding_host_side(lib):
    """The Python binding's host-only parts: descriptors from workloads and
    options, output shapes and dtypes as the header states them (on the meta
    device: no memory, no GPU), the retained-row capacity, errors raised."""
    import torch
    from paper_2606_03075_gb300 import api
    wl = synth.WORKLOADS["qwen25"]
    d = api.desc_for_workload(wl)
    assert (d.L, d.H_q, d.H_kv, d.d, d.N, d.N_v, d.n_win) == (
        wl.L, wl.H_q, wl.H_kv, wl.d, wl.N, wl.N_v, wl.n_win)
    assert d.w_layer_stride == wl.n_win and d.softmax_scale == 0.0
    assert (d.budget_basis, d.weight_mode, d.keep_first, d.keep_last, d.budget_stat,
            d.head_budgets) == (0, 0, 0, 0, 0, 0)
    o = api.desc_for_workload(wl, 0.125, basis="all", weights="eq7", keep_first=4, keep_last=1,
                              stat="uniform", head_budgets=True, w_layer_stride=0)
    assert (o.budget_basis, o.weight_mode, o.keep_first, o.keep_last, o.budget_stat,
            o.head_budgets, o.w_layer_stride) == (1, 1, 4, 1, 2, 1, 0)
    assert o.softmax_scale == 0.125
    assert api.budget_units(d) == wl.L and api.budget_units(o) == wl.L * wl.H_kv
    r = 0.05
    rows = wl.H_kv * (wl.L * wl.N_t + oracle.vision_budget_total(r, wl.N_v, wl.L))
    assert api.tgvkv_retained_rows(d, r) == rows
    out = api.alloc_outputs(d, r, device="meta")
    assert tuple(out.scores.shape) == (wl.L, wl.H_kv, wl.N_v) and out.scores.dtype == torch.float32
    assert tuple(out.tvb_stat.shape) == (wl.L,) and out.budgets.dtype == torch.int32
    assert tuple(out.offsets.shape) == (wl.L * wl.H_kv + 1,) and out.offsets.dtype == torch.int64
    assert tuple(out.idx.shape) == (rows,) and out.idx.dtype == torch.int32
    assert tuple(out.k_out.shape) == (rows, wl.d) == tuple(out.v_out.shape)
    assert out.k_out.dtype == torch.bfloat16
    heads = api.alloc_outputs(api.desc_for_workload(wl, head_budgets=True), r, device="meta")
    assert tuple(heads.budgets.shape) == (wl.L * wl.H_kv,) == tuple(heads.tvb_stat.shape)
    with pytest.raises(api.TgvkvError):
        api.tgvkv_retained_rows(d, 1.5)
    with pytest.raises(api.TgvkvError):
        api.tgvkv_workspace_size(api.make_desc(1, 2, 2, 96, 10, 5, 2))
    with pytest.raises(KeyError):
        api.make_desc(1, 2, 2, 64, 10, 5, 2, basis="text")
