"""Sharded eviction on CPU ranks (gloo, world size 2 and 3): the host logic of
paper_2606_03075_gb300.shard -- layer ranges, the all-gather of the TVB
statistic, identical budgets on every rank -- driven with the fp64 oracle as
the compute backend, against the unsharded oracle."""
import math
import os
import socket
import tempfile

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2606_03075_gb300 import shard, synth
from paper_2606_03075_gb300._lib import Desc


class OracleBackend:
    """The oracle behind the backend interface of shard.sharded_evict (CPU tensors)."""

    def score(self, desc, q, k, modality, text_pos, w):
        s, st = oracle.twr_scores_tvb_stat(
            oracle.widen_bf16(q.numpy()), oracle.widen_bf16(k.numpy()), modality.numpy(),
            text_pos.numpy(), w.numpy().astype(np.float64), 1.0 / math.sqrt(desc.d), desc.H_kv)
        return torch.from_numpy(s), torch.from_numpy(np.asarray(st, np.float64))

    def budget(self, desc_full, tvb_stat, ratio):
        total = oracle.vision_budget_total(ratio, desc_full.N_v, desc_full.L)
        return torch.tensor(oracle.tvb_budgets(tvb_stat.numpy(), total, desc_full.N_v),
                            dtype=torch.int32)

    def select_compact(self, desc, scores, budgets, modality, k, v):
        off, idx = oracle.tpr_select(scores.numpy(), budgets.numpy().tolist(), modality.numpy())
        ko, vo = oracle.compact(k.numpy(), v.numpy(), off, idx)
        return (torch.from_numpy(np.asarray(off, np.int64)), torch.from_numpy(np.asarray(idx)),
                torch.from_numpy(ko), torch.from_numpy(vo))


WL = synth.custom("shard5", 5, 4, 2, 64, [("text", 9), ("vision", 70), ("text", 6), ("vision", 30),
                                          ("text", 12)], weights="dirichlet", ratios=(0.2,))


def _desc(wl):
    return Desc(L=wl.L, H_q=wl.H_q, H_kv=wl.H_kv, d=wl.d, N=wl.N, N_v=wl.N_v, n_win=wl.n_win,
                softmax_scale=0.0, w_layer_stride=wl.n_win)


def _rank_main(rank, world, port, outdir):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        inp = synth.generate(WL, seed=7)
        l0, l1 = shard.layer_range(WL.L, rank, world)
        local = {k: torch.from_numpy(np.ascontiguousarray(inp[k][l0:l1])) for k in ("q", "k", "v", "w")}
        local["modality"] = torch.from_numpy(inp["modality"])
        local["text_pos"] = torch.from_numpy(inp["text_pos"].astype(np.int32))
        res = shard.sharded_evict(_desc(WL), local, 0.2, rank, world, OracleBackend())
        np.savez(os.path.join(outdir, f"r{rank}.npz"), l0=l0, l1=l1, budgets=res.budgets.numpy(),
                 stat=res.tvb_stat.numpy(), scores=res.scores.numpy(), offsets=res.offsets.numpy(),
                 idx=res.idx.numpy(), k_out=res.k_out.numpy(), v_out=res.v_out.numpy())
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_layer_ranges_cover_every_layer_once():
    for L in (1, 2, 5, 28, 32, 33):
        for world in (1, 2, 3, 4, 8):
            spans = [shard.layer_range(L, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == L
            assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
            sizes = [b - a for a, b in spans]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard.layer_range(4, 2, 2)


@pytest.mark.parametrize("world", [2, 3])
def test_cpu_ranks_match_the_unsharded_oracle(world):
    """5 layers over 2 ranks (3 + 2) or 3 ranks (2 + 2 + 1): the statistic's
    slices differ in length, so the all-gather's padding is exercised."""
    with tempfile.TemporaryDirectory() as outdir:
        mp.spawn(_rank_main, args=(world, _free_port(), outdir), nprocs=world, join=True)
        parts = [dict(np.load(os.path.join(outdir, f"r{r}.npz"))) for r in range(world)]
    inp = synth.generate(WL, seed=7)
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], inp["w"],
                       0.2, WL.H_kv)
    # the exchange gave every rank the whole statistic, hence the same budgets
    for p in parts:
        np.testing.assert_array_equal(p["stat"], ref["stat"])
        np.testing.assert_array_equal(p["budgets"], ref["budgets"])
    # each rank's layers: scores, CSR, retained positions and rows as in the unsharded run
    H = WL.H_kv
    for p in parts:
        l0, l1 = int(p["l0"]), int(p["l1"])
        np.testing.assert_array_equal(p["scores"], ref["scores"][l0:l1])
        lo, hi = ref["offsets"][l0 * H], ref["offsets"][l1 * H]
        np.testing.assert_array_equal(p["offsets"], ref["offsets"][l0 * H:l1 * H + 1] - lo)
        np.testing.assert_array_equal(p["idx"], ref["idx"][lo:hi])
        np.testing.assert_array_equal(p["k_out"], ref["k_out"][lo:hi])
        np.testing.assert_array_equal(p["v_out"], ref["v_out"][lo:hi])
    assert sum(int(p["l1"]) - int(p["l0"]) for p in parts) == WL.L


def _rank_leaves(rank, world, port, outdir):
    """Rank 1 leaves between steps, without joining the statistic's exchange;
    rank 0's exchange must end with an error within the group's timeout
    instead of waiting for it forever."""
    import datetime
    import time
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world, timeout=datetime.timedelta(seconds=10))
    try:
        if rank == 1:
            open(os.path.join(outdir, "r1_left"), "w").close()
            return
        inp = synth.generate(WL, seed=7)
        l0, l1 = shard.layer_range(WL.L, rank, world)
        local = {k: torch.from_numpy(np.ascontiguousarray(inp[k][l0:l1])) for k in ("q", "k", "v", "w")}
        local["modality"] = torch.from_numpy(inp["modality"])
        local["text_pos"] = torch.from_numpy(inp["text_pos"].astype(np.int32))
        t0 = time.time()
        try:
            shard.sharded_evict(_desc(WL), local, 0.2, rank, world, OracleBackend())
            outcome = "completed"
        except Exception as exc:      # the failed exchange surfaces as an error
            outcome = f"error {time.time() - t0:.1f} {type(exc).__name__}"
        with open(os.path.join(outdir, "r0.txt"), "w") as f:
            f.write(outcome)
    finally:
        dist.destroy_process_group()


def test_a_rank_that_leaves_fails_the_exchange_instead_of_hanging():
    world = 2
    with tempfile.TemporaryDirectory() as outdir:
        mp.spawn(_rank_leaves, args=(world, _free_port(), outdir), nprocs=world, join=True)
        assert os.path.exists(os.path.join(outdir, "r1_left"))
        outcome = open(os.path.join(outdir, "r0.txt")).read().split()
        assert outcome[0] == "error", outcome
        assert float(outcome[1]) < 30.0


class OracleHeadBackend(OracleBackend):
    """The oracle with per-head TV masses (for sharding by KV head)."""

    def score_heads(self, desc, q, k, modality, text_pos, w):
        qd, kd = oracle.widen_bf16(q.numpy()), oracle.widen_bf16(k.numpy())
        scale = 1.0 / math.sqrt(desc.d)
        s, _ = oracle.twr_scores_tvb_stat(qd, kd, modality.numpy(), text_pos.numpy(),
                                          w.numpy().astype(np.float64), scale, desc.H_kv)
        m = oracle.tv_statistic_per_head(qd, kd, modality.numpy(), text_pos.numpy(), scale,
                                         desc.H_kv)
        return torch.from_numpy(s), torch.from_numpy(np.asarray(m, np.float64))


WLH = synth.custom("shard_heads", 3, 10, 5, 64, [("text", 9), ("vision", 70), ("text", 6),
                                                ("vision", 30), ("text", 12)],
                   weights="dirichlet", ratios=(0.2,))


def _rank_heads(rank, world, port, outdir):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        inp = synth.generate(WLH, seed=9)
        G = WLH.H_q // WLH.H_kv
        g0, g1 = shard.head_range(WLH.H_kv, rank, world)
        local = {"q": torch.from_numpy(np.ascontiguousarray(inp["q"][:, G * g0:G * g1])),
                 "k": torch.from_numpy(np.ascontiguousarray(inp["k"][:, g0:g1])),
                 "v": torch.from_numpy(np.ascontiguousarray(inp["v"][:, g0:g1])),
                 "w": torch.from_numpy(inp["w"]),
                 "modality": torch.from_numpy(inp["modality"]),
                 "text_pos": torch.from_numpy(inp["text_pos"].astype(np.int32))}
        res = shard.head_sharded_evict(_desc(WLH), local, 0.2, rank, world, OracleHeadBackend())
        np.savez(os.path.join(outdir, f"h{rank}.npz"), g0=g0, g1=g1, budgets=res.budgets.numpy(),
                 stat=res.tvb_stat.numpy(), offsets=res.offsets.numpy(), idx=res.idx.numpy(),
                 k_out=res.k_out.numpy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_cpu_ranks_sharded_by_kv_head_match_the_unsharded_oracle(world):
    """5 KV heads over 2 ranks (3 + 2) or 3 ranks (2 + 2 + 1): padded blocks in
    the all-gather of the per-head masses."""
    inp = synth.generate(WLH, seed=9)
    ref = oracle.evict(inp["q"], inp["k"], inp["v"], inp["modality"], inp["text_pos"], inp["w"],
                       0.2, WLH.H_kv)
    with tempfile.TemporaryDirectory() as outdir:
        mp.spawn(_rank_heads, args=(world, _free_port(), outdir), nprocs=world, join=True)
        H = WLH.H_kv
        for r in range(world):
            z = np.load(os.path.join(outdir, f"h{r}.npz"))
            np.testing.assert_array_equal(z["budgets"], ref["budgets"])
            assert np.allclose(z["stat"], ref["stat"], rtol=1e-12)
            g0, g1 = int(z["g0"]), int(z["g1"])
            h = g1 - g0
            for l in range(WLH.L):
                for gl in range(h):
                    g = g0 + gl
                    lo, hi = z["offsets"][l * h + gl], z["offsets"][l * h + gl + 1]
                    rlo, rhi = ref["offsets"][l * H + g], ref["offsets"][l * H + g + 1]
                    np.testing.assert_array_equal(z["idx"][lo:hi], ref["idx"][rlo:rhi])
                    np.testing.assert_array_equal(z["k_out"][lo:hi], ref["k_out"][rlo:rhi])
