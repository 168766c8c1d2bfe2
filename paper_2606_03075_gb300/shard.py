"""Layer-sharded eviction across ranks (one process per GPU).

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


@dataclass
class ShardResult:
    layers: tuple          # (l0, l1)
    budgets: torch.Tensor  # int32 [L], identical on every rank
    scores: torch.Tensor   # float32 [l1 - l0][H_kv][N_v]
    tvb_stat: torch.Tensor  # float32 [L] (gathered)
    offsets: torch.Tensor  # int64 [(l1 - l0) * H_kv + 1], CSR of this rank's heads
    idx: torch.Tensor      # int32 retained positions of this rank's heads
    k_out: torch.Tensor
    v_out: torch.Tensor


class CudaBackend:
    """The CUDA library through the Python binding; tensors on one device."""

    def __init__(self, device=None):
        from . import api
        self.api = api
        self.device = device

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
