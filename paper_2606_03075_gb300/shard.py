"""Sharded eviction across ranks (one process per GPU), by layer or by KV head.

The eviction step shards by layer: scores, selection and gathering are
independent per (layer, KV head), and the TVB budget split (Eq. 5) is the one
step that needs every layer -- it divides the request's vision budget in
proportion to the per-layer statistic S_l.  Each rank therefore

  1. scores its own contiguous range of layers (tgvkv_score),
  2. all-gathers the L-vector of statistics (the only exchange: L floats),
  3. splits the budget over all L layers -- the same deterministic integers on
     every rank (tgvkv_budget on the full vector),
  4. selects and gathers its own layers with their budgets (tgvkv_select,
     tgvkv_compact), keeping a compacted cache of its layers.

Sharding by KV head (a tensor-parallel cache: every rank holds some KV heads of
every layer) exchanges the per-head TV masses instead: each rank scores its heads
of all layers, the L x H_kv masses are all-gathered, and every rank adds each
layer's masses in head order -- the order the single-device kernel adds them in,
so S_l and the budgets are bit-identical to one device's -- then selects and
gathers its own heads.

The compute calls go through a backend object, so that the host logic (layer
ranges, exchange, budget consistency) is the same whether the backend is the
CUDA library or, in tests on CPU ranks, another implementation.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch


def layer_range(L: int, rank: int, world: int) -> tuple:
    """Contiguous layers [l0, l1) of `rank`: the first L % world ranks get one more."""
    if not (0 <= rank < world):
        raise ValueError(f"rank {rank} outside a world of {world}")
    base, extra = divmod(L, world)
    l0 = rank * base + min(rank, extra)
    return l0, l0 + base + (1 if rank < extra else 0)


def gather_stat(local_stat: torch.Tensor, L: int, rank: int, world: int, group=None) -> torch.Tensor:
    """All-gather the per-rank slices of the L-vector of TVB statistics.

    Slices may differ in length by one; they are padded to the longest, gathered
    and concatenated in rank order.  Returns a tensor of L entries with the
    dtype and device of `local_stat`."""
    if world == 1:
        return local_stat.clone()
    import torch.distributed as dist
    width = math.ceil(L / world)
    buf = torch.zeros(width, dtype=local_stat.dtype, device=local_stat.device)
    buf[:local_stat.numel()] = local_stat
    parts = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(parts, buf, group=group)
    out = []
    for r in range(world):
        l0, l1 = layer_range(L, r, world)
        out.append(parts[r][:l1 - l0])
    full = torch.cat(out)
    assert full.numel() == L
    return full


def gather_head_masses(local: torch.Tensor, H_kv: int, rank: int, world: int,
                       group=None) -> torch.Tensor:
    """All-gather the per-rank [L, h] blocks of per-head TV masses (h = the
    rank's KV heads, head_range) into [L, H_kv] in global head order."""
    if world == 1:
        return local.clone()
    import torch.distributed as dist
    L = local.shape[0]
    width = math.ceil(H_kv / world)
    buf = torch.zeros((L, width), dtype=local.dtype, device=local.device)
    buf[:, :local.shape[1]] = local
    parts = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(parts, buf, group=group)
    cols = []
    for r in range(world):
        g0, g1 = layer_range(H_kv, r, world)
        cols.append(parts[r][:, :g1 - g0])
    full = torch.cat(cols, dim=1)
    assert full.shape == (L, H_kv)
    return full


def layer_stat_from_heads(masses: torch.Tensor) -> torch.Tensor:
    """S_l = the sum of layer l's per-head masses, added in head order from zero
    (one add per head: the order the score kernel uses, so the same bits)."""
    stat = torch.zeros(masses.shape[0], dtype=masses.dtype, device=masses.device)
    for g in range(masses.shape[1]):
        stat = stat + masses[:, g]
    return stat


@dataclass
class ShardResult:
    span: tuple            # (l0, l1) layers, or (g0, g1) KV heads, of this rank
    budgets: torch.Tensor  # int32 [L], identical on every rank
    scores: torch.Tensor   # float32 [layers][KV heads][N_v] of this rank
    tvb_stat: torch.Tensor  # float32 [L] (from every rank's part)
    offsets: torch.Tensor  # int64, CSR over this rank's (layer, KV head) sets
    idx: torch.Tensor      # int32 retained positions of this rank's heads
    k_out: torch.Tensor
    v_out: torch.Tensor


class CudaBackend:
    """The CUDA library through the Python binding; tensors on one device."""

    def __init__(self, device=None):
        from . import api
        self.api = api
        self.device = device

    def score_heads(self, desc, q, k, modality, text_pos, w):
        """Scores and the per-head TV masses [L, H_kv] (the score kernel with
        one statistic per (layer, KV head))."""
        d = self.api.make_desc(desc.L, desc.H_q, desc.H_kv, desc.d, desc.N, desc.N_v,
                               desc.n_win, desc.softmax_scale, desc.w_layer_stride,
                               head_budgets=True)
        out_s = torch.empty(desc.L * desc.H_kv * desc.N_v, dtype=torch.float32, device=self.device)
        out_t = torch.empty(desc.L * desc.H_kv, dtype=torch.float32, device=self.device)
        ws = self.api.new_workspace(d, self.device)
        self.api.tgvkv_score(d, q, k, modality, text_pos, w, out_s, out_t, ws)
        if self.api.tgvkv_status(ws) != 0:
            raise RuntimeError("device status bits set by tgvkv_score")
        return out_s.view(desc.L, desc.H_kv, desc.N_v), out_t.view(desc.L, desc.H_kv)

    def score(self, desc, q, k, modality, text_pos, w):
        out_s = torch.empty(desc.L * desc.H_kv * desc.N_v, dtype=torch.float32, device=self.device)
        out_t = torch.empty(desc.L, dtype=torch.float32, device=self.device)
        ws = self.api.new_workspace(desc, self.device)
        self.api.tgvkv_score(desc, q, k, modality, text_pos, w, out_s, out_t, ws)
        if self.api.tgvkv_status(ws) != 0:
            raise RuntimeError("device status bits set by tgvkv_score")
        return out_s.view(desc.L, desc.H_kv, desc.N_v), out_t

    def budget(self, desc_full, tvb_stat, ratio):
        budgets = torch.empty(desc_full.L, dtype=torch.int32, device=self.device)
        ws = self.api.new_workspace(desc_full, self.device)
        self.api.tgvkv_budget(desc_full, tvb_stat, ratio, budgets, ws)
        return budgets

    def select_compact(self, desc, scores, budgets, modality, k, v):
        ws = self.api.new_workspace(desc, self.device)
        heads = desc.L * desc.H_kv
        offsets = torch.empty(heads + 1, dtype=torch.int64, device=self.device)
        rows = int(desc.H_kv * (desc.L * (desc.N - desc.N_v)) + int(budgets.sum().item()) * desc.H_kv)
        idx = torch.empty(max(rows, 1), dtype=torch.int32, device=self.device)
        k_out = torch.empty((max(rows, 1), desc.d), dtype=torch.bfloat16, device=self.device)
        v_out = torch.empty_like(k_out)
        self.api.tgvkv_select(desc, scores.reshape(-1), budgets, modality, offsets, idx, ws)
        self.api.tgvkv_compact(desc, k, v, offsets, idx, k_out, v_out, ws)
        if self.api.tgvkv_status(ws) != 0:
            raise RuntimeError("device status bits set by tgvkv_select / tgvkv_compact")
        return offsets, idx[:rows], k_out[:rows], v_out[:rows]


def sharded_evict(desc_full, local: dict, ratio: float, rank: int, world: int, backend,
                  group=None) -> ShardResult:
    """Evict this rank's layers of one request.

    desc_full: the descriptor of the whole request (all L layers).
    local:     this rank's inputs -- q, k, v of its layers (leading dimension
               l1 - l0), and modality, text_pos, w (w with its own layers' rows).
    """
    from .api import make_desc
    L = desc_full.L
    l0, l1 = layer_range(L, rank, world)
    desc = make_desc(l1 - l0, desc_full.H_q, desc_full.H_kv, desc_full.d, desc_full.N,
                     desc_full.N_v, desc_full.n_win, desc_full.softmax_scale,
                     desc_full.w_layer_stride)
    scores, stat = backend.score(desc, local["q"], local["k"], local["modality"],
                                 local["text_pos"], local["w"])
    full_stat = gather_stat(stat, L, rank, world, group)            # the one exchange
    budgets = backend.budget(desc_full, full_stat, ratio)           # same integers on every rank
    offsets, idx, k_out, v_out = backend.select_compact(desc, scores, budgets[l0:l1].contiguous(),
                                                        local["modality"], local["k"], local["v"])
    return ShardResult((l0, l1), budgets, scores, full_stat, offsets, idx, k_out, v_out)


def head_sharded_evict(desc_full, local: dict, ratio: float, rank: int, world: int, backend,
                       group=None) -> ShardResult:
    """Evict this rank's KV heads (head_range) of every layer of one request.

    desc_full: the descriptor of the whole request (all H_kv heads).
    local:     this rank's inputs -- q of its query heads [L][G h][n_win][d], k, v of
               its KV heads [L][h][N][d], and modality, text_pos, w (all layers).
    The result's CSR runs over (layer, local head); tvb_stat is the full S_l.
    """
    from .api import make_desc
    H = desc_full.H_kv
    G = desc_full.H_q // H
    g0, g1 = head_range(H, rank, world)
    desc = make_desc(desc_full.L, G * (g1 - g0), g1 - g0, desc_full.d, desc_full.N,
                     desc_full.N_v, desc_full.n_win, desc_full.softmax_scale,
                     desc_full.w_layer_stride)
    scores, masses = backend.score_heads(desc, local["q"], local["k"], local["modality"],
                                         local["text_pos"], local["w"])
    full_masses = gather_head_masses(masses, H, rank, world, group)   # the one exchange
    stat = layer_stat_from_heads(full_masses)
    budgets = backend.budget(desc_full, stat, ratio)                   # same integers everywhere
    offsets, idx, k_out, v_out = backend.select_compact(desc, scores, budgets, local["modality"],
                                                        local["k"], local["v"])
    return ShardResult((g0, g1), budgets, scores, stat, offsets, idx, k_out, v_out)


def head_range(H_kv: int, rank: int, world: int) -> tuple:
    """Contiguous KV heads [g0, g1) of `rank`: the first H_kv % world ranks get one more."""
    return layer_range(H_kv, rank, world)
