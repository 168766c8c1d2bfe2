"""Seeded synthetic workloads for the eviction step.

This module draws random inputs only: bf16 text queries, K/V caches, the
modality layout, the query-row positions and the text weights.  It holds none
of the method's arithmetic, so both the CUDA path and the CPU oracle may take
their inputs from it.

Shapes follow five reference workloads (no model weights or datasets exist
here, so the values are synthetic):

* ``tiny``    - 1 layer, 8/8 heads, d=64, 16 text + 64 vision + 32 question
  tokens, iid N(0,1) keys, uniform weights, 25% vision budget.
* ``llava15`` - LLaVA-1.5-7B shape: 32 layers, 32/32 heads, d=128,
  35 text + 576 vision + 64 question tokens, budgets 5% and 20%.
* ``next``    - LLaVA-NeXT-7B shape: 32 layers, 32/32 heads, d=128,
  32 text + 2880 vision (5 tiles x 576) + 96 question tokens.
* ``qwen25``  - Qwen2.5-VL-7B shape, grouped-query: 28 layers, 28/4 heads,
  d=128, 32 text + 4096 vision + 224 question tokens.
* ``video``   - long video, grouped-query: 28 layers, 28/4 heads, d=128,
  32 text + 32 x (8 timestamp text + 256 vision) + 224 question tokens; every
  text token is a query row and the text weights are Dirichlet(1) per layer.

Key distribution of the non-tiny workloads, per (layer, KV head): text keys
iid N(0, I); vision keys sqrt(0.8) c + sqrt(0.2) e with one shared centre c,
so two vision keys have cosine ~0.8 (vision tokens are mutually similar, text
tokens diverse); then 4 channels of every key are scaled by 8 (outlier
channels).  Queries and values are iid N(0, 1).  Everything is rounded to bf16
(round to nearest even) and returned as int16 bit patterns.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

_TAG_Q, _TAG_K, _TAG_V, _TAG_W, _TAG_QALL = 1, 2, 3, 4, 5


@dataclass(frozen=True)
class Workload:
    name: str
    L: int
    H_q: int
    H_kv: int
    d: int
    segments: tuple            # ((kind, count), ...) with kind "text" | "vision"
    window: object = "last_text_segment"   # | "all_text" | int = last n text tokens
    weights: str = "uniform"   # | "dirichlet"
    keys: str = "clustered"    # | "iid"
    ratios: tuple = (0.05,)
    outlier_channels: int = 4
    outlier_scale: float = 8.0
    vision_cosine: float = 0.8
    extra: dict = field(default_factory=dict, compare=False)

    # ---- layout -------------------------------------------------------
    @property
    def modality(self) -> np.ndarray:
        parts = [np.full(c, 1 if kind == "vision" else 0, np.uint8)
                 for kind, c in self.segments]
        return np.concatenate(parts) if parts else np.zeros(0, np.uint8)

    @property
    def N(self) -> int:
        return int(sum(c for _, c in self.segments))

    @property
    def N_v(self) -> int:
        return int(sum(c for kind, c in self.segments if kind == "vision"))

    @property
    def N_t(self) -> int:
        return self.N - self.N_v

    @property
    def text_pos(self) -> np.ndarray:
        text = np.flatnonzero(self.modality == 0).astype(np.int32)
        if self.window == "all_text":
            return text
        if self.window == "last_text_segment":
            kind, count = self.segments[-1]
            assert kind == "text"
            return np.arange(self.N - count, self.N, dtype=np.int32)
        return text[-int(self.window):]

    @property
    def n_win(self) -> int:
        return int(self.text_pos.size)

    @property
    def G(self) -> int:
        return self.H_q // self.H_kv

    def input_bytes(self) -> dict:
        """Bytes of each device input of one step."""
        return dict(q=self.L * self.H_q * self.n_win * self.d * 2,
                    k=self.L * self.H_kv * self.N * self.d * 2,
                    v=self.L * self.H_kv * self.N * self.d * 2,
                    modality=self.N, text_pos=4 * self.n_win,
                    w=4 * self.L * self.n_win)


def _video_segments(frames=32, stamp=8, per_frame=256, head=32, tail=224):
    seg = [("text", head)]
    for _ in range(frames):
        seg += [("text", stamp), ("vision", per_frame)]
    seg.append(("text", tail))
    return tuple(seg)


WORKLOADS = {
    "tiny": Workload("tiny", 1, 8, 8, 64,
                     (("text", 16), ("vision", 64), ("text", 32)),
                     keys="iid", ratios=(0.25,), outlier_channels=0),
    "llava15": Workload("llava15", 32, 32, 32, 128,
                        (("text", 35), ("vision", 576), ("text", 64)),
                        ratios=(0.05, 0.20)),
    "next": Workload("next", 32, 32, 32, 128,
                     (("text", 32), ("vision", 2880), ("text", 96)),
                     ratios=(0.05, 0.10, 0.20)),
    "qwen25": Workload("qwen25", 28, 28, 4, 128,
                       (("text", 32), ("vision", 4096), ("text", 224)),
                       ratios=(0.05,)),
    "video": Workload("video", 28, 28, 4, 128, _video_segments(),
                      window="all_text", weights="dirichlet", ratios=(0.05,)),
}


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (round to nearest even), as int16."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    u = (u + (((u >> 16) & 1) + np.uint32(0x7FFF))) >> 16
    return u.astype(np.uint16).view(np.int16)


def _rng(seed: int, tag: int, layer: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), tag, int(layer)])


def draw_layer(wl: Workload, seed: int, layer: int):
    """Inputs of one layer: (q [H_q,n_win,d], k, v [H_kv,N,d] int16, w [n_win] f32)."""
    n, d, n_win = wl.N, wl.d, wl.n_win
    rq = _rng(seed, _TAG_Q, layer)
    q = rq.standard_normal((wl.H_q, n_win, d), dtype=np.float32)

    rk = _rng(seed, _TAG_K, layer)
    vis = wl.modality == 1
    k = np.empty((wl.H_kv, n, d), np.float32)
    for g in range(wl.H_kv):
        x = rk.standard_normal((n, d), dtype=np.float32)
        if wl.keys == "clustered":
            centre = rk.standard_normal(d, dtype=np.float32)
            a = np.float32(np.sqrt(wl.vision_cosine))
            b = np.float32(np.sqrt(1.0 - wl.vision_cosine))
            x[vis] = a * centre[None, :] + b * x[vis]
        if wl.outlier_channels:
            ch = rk.choice(d, wl.outlier_channels, replace=False)
            x[:, ch] *= np.float32(wl.outlier_scale)
        k[g] = x

    rv = _rng(seed, _TAG_V, layer)
    v = rv.standard_normal((wl.H_kv, n, d), dtype=np.float32)

    rw = _rng(seed, _TAG_W, layer)
    if wl.weights == "dirichlet":
        w = rw.dirichlet(np.ones(n_win)).astype(np.float32)
    else:
        w = np.full(n_win, 1.0 / n_win, np.float32)
    return to_bf16_bits(q), to_bf16_bits(k), to_bf16_bits(v), w


def _each_layer(fn, n_layers):
    """fn(l) for every layer on a few threads (every layer draws from its own
    seeded streams, so the result does not depend on the order)."""
    workers = max(1, min(n_layers, os.cpu_count() or 1, 16))
    if workers == 1:
        for l in range(n_layers):
            fn(l)
        return
    with ThreadPoolExecutor(workers) as ex:
        list(ex.map(fn, range(n_layers)))


def generate(wl: Workload, seed: int = 0) -> dict:
    """All inputs of one eviction step as host numpy arrays."""
    L, n, d, n_win = wl.L, wl.N, wl.d, wl.n_win
    q = np.empty((L, wl.H_q, n_win, d), np.int16)
    k = np.empty((L, wl.H_kv, n, d), np.int16)
    v = np.empty((L, wl.H_kv, n, d), np.int16)
    w = np.empty((L, n_win), np.float32)

    def one(l):
        q[l], k[l], v[l], w[l] = draw_layer(wl, seed, l)

    _each_layer(one, L)
    return dict(q=q, k=k, v=v, w=w, modality=wl.modality,
                text_pos=wl.text_pos.astype(np.int32))


def draw_prefill_queries(wl: Workload, seed: int, layer: int, q_rows: np.ndarray) -> np.ndarray:
    """Queries of every token of one layer, [H_q, N, d] int16 bf16 bits: the
    query-row positions (text_pos) hold q_rows, that layer's q of draw_layer;
    every other position holds a fresh N(0, 1) draw."""
    r = _rng(seed, _TAG_QALL, layer)
    q = to_bf16_bits(r.standard_normal((wl.H_q, wl.N, wl.d), dtype=np.float32))
    q[:, wl.text_pos] = q_rows
    return q


def generate_prefill(wl: Workload, seed: int = 0, inp: dict | None = None) -> dict:
    """generate() plus q_all [L, H_q, N, d]: the queries of every token, whose
    rows at the query positions are generate()'s q."""
    inp = dict(inp if inp is not None else generate(wl, seed))
    q_all = np.empty((wl.L, wl.H_q, wl.N, wl.d), np.int16)

    def one(l):
        q_all[l] = draw_prefill_queries(wl, seed, l, inp["q"][l])

    _each_layer(one, wl.L)
    inp["q_all"] = q_all
    return inp


def custom(name, L, H_q, H_kv, d, segments, **kw) -> Workload:
    """A workload with an arbitrary layout (parity and edge-case tests)."""
    return Workload(name, L, H_q, H_kv, d, tuple(segments), **kw)
