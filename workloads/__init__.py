"""Seeded synthetic workloads for block-causal attention.

This module holds shapes, seeds and random draws only: no attention arithmetic.
Both the fp64 oracle (through the tests) and the CUDA path take their inputs
from here, so the two sides see the same bf16 tensors.

The paper trains and streams on VAE latents of DROID / RealEstate10K videos
(Sec. 4.1); those datasets are not available, so iid Gaussian tensors with
the paper's shapes stand in for the post-RoPE Q/K/V of one attention layer:
head dims from the model table (Sec. 4.1, model configurations), a chunk of two
latent frames (Sec. 4.1, training details) at 880 tokens per chunk, and the
cache / in-flight window sizes of the ablations (Sec. 4.3).

Draw order (fixed, part of the recipe): a fresh ``torch.Generator('cpu')``
seeded with the config seed; ``randn`` in fp32 in the order listed per config;
gains / standard deviations drawn after the tensors; products in fp32; the
result rounded to bf16 (round-to-nearest-even, torch's ``.to``).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import torch

__all__ = [
    "TrainConfig", "CacheConfig", "TRAIN_CONFIGS", "CACHE_CONFIGS",
    "gen_train", "gen_cache", "ring_slice_rows",
]


@dataclasses.dataclass(frozen=True)
class TrainConfig:
    """Block-causal attention over ``n_chunks * T`` tokens (fwd, optionally bwd)."""
    name: str
    B: int
    H: int
    d: int
    n_chunks: int
    T: int
    seed: int
    gain_lo: float = 1.0   # per-head gain on Q and K, U[gain_lo, gain_hi]
    gain_hi: float = 1.0
    backward: bool = True

    @property
    def N(self) -> int:
        return self.n_chunks * self.T

    @property
    def scale(self) -> float:
        return 1.0 / (self.d ** 0.5)


@dataclasses.dataclass(frozen=True)
class CacheConfig:
    """In-flight query chunks against a FIFO ring of committed chunks.

    ``W`` in-flight chunks of ``T`` tokens; ring of ``cap`` tokens of which
    ``len`` are valid, the logically oldest at physical row ``head``.
    ``steps`` successive calls, each committing the oldest in-flight chunk's
    K/V into the ring (streaming, Sec. 3.5).
    """
    name: str
    B: int
    H: int
    d: int
    W: int
    T: int
    cap: int
    length: int
    head: int
    steps: int
    seed: int
    std_lo: float = 1.0    # per-chunk std on K and V, U[std_lo, std_hi]
    std_hi: float = 1.0
    sink: int = 0          # tokens of the sink anchor ahead of the ring (Sec. 3.5)

    @property
    def scale(self) -> float:
        return 1.0 / (self.d ** 0.5)


TRAIN_CONFIGS: Dict[str, TrainConfig] = {
    # 4 chunks x 64 tokens, forward only
    "tiny_fwd": TrainConfig("tiny_fwd", B=1, H=2, d=64, n_chunks=4, T=64, seed=0,
                            backward=False),
    # MiniWorld-B-like width 768 / 12 heads, 16 chunks of 880 tokens (two
    # latent frames of 440 tokens each)
    "train_b12_d64": TrainConfig("train_b12_d64", B=2, H=12, d=64, n_chunks=16,
                                 T=880, seed=1),
    # width 2048 / 16 heads, 21 chunks, peaky logits from per-head gains
    "train_h16_d128_peaky": TrainConfig("train_h16_d128_peaky", B=1, H=16, d=128,
                                        n_chunks=21, T=880, seed=2,
                                        gain_lo=1.0, gain_hi=4.0),
    # the paper's 32-chunk training window with 600-token chunks (15 x 20
    # latent positions x 2 frames) at the MiniWorld-1B head layout (1536 / 12)
    "train_1b_32x600": TrainConfig("train_1b_32x600", B=1, H=12, d=128, n_chunks=32,
                                   T=600, seed=6),
    # the MiniWorld-0.5B head layout (1152 / 16 = 72 channels per head)
    "train_05b_d72": TrainConfig("train_05b_d72", B=1, H=16, d=72, n_chunks=16, T=880,
                                 seed=7),
}

CACHE_CONFIGS: Dict[str, CacheConfig] = {
    # one query chunk against an 8-chunk ring whose head wraps mid-buffer
    "rolling_cache": CacheConfig("rolling_cache", B=1, H=16, d=128, W=1, T=880,
                                 cap=8 * 880, length=8 * 880, head=5 * 880,
                                 steps=64, seed=3),
    # 4 in-flight chunks against a 12-chunk ring, per-chunk K/V scales
    "pipelined": CacheConfig("pipelined", B=1, H=16, d=128, W=4, T=880,
                             cap=12 * 880, length=12 * 880, head=7 * 880,
                             steps=1, seed=4, std_lo=0.5, std_hi=1.5),
    # 8 in-flight chunks, a 12-chunk ring and a resident sink of one latent
    # frame (half a 2-frame chunk), the shape of the paper's cache ablation
    "sink_anchor": CacheConfig("sink_anchor", B=1, H=16, d=128, W=8, T=880,
                               cap=12 * 880, length=12 * 880, head=3 * 880,
                               steps=1, seed=5, sink=440),
}


def _bf16(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16)


def gen_train(cfg: TrainConfig, device: str = "cpu") -> Dict[str, torch.Tensor]:
    """Q, K, V (and dO when ``cfg.backward``) as bf16 ``[B, H, N, d]``.

    Draws: Q, K, V, [dO], then one gain per head g_h ~ U[lo, hi] applied to
    both Q and K.
    """
    g = torch.Generator("cpu").manual_seed(cfg.seed)
    shape = (cfg.B, cfg.H, cfg.N, cfg.d)
    q = torch.randn(shape, generator=g, dtype=torch.float32)
    k = torch.randn(shape, generator=g, dtype=torch.float32)
    v = torch.randn(shape, generator=g, dtype=torch.float32)
    do = torch.randn(shape, generator=g, dtype=torch.float32) if cfg.backward else None
    if cfg.gain_hi != 1.0 or cfg.gain_lo != 1.0:
        gain = cfg.gain_lo + (cfg.gain_hi - cfg.gain_lo) * torch.rand(
            (cfg.H,), generator=g, dtype=torch.float32)
        q = q * gain.view(1, cfg.H, 1, 1)
        k = k * gain.view(1, cfg.H, 1, 1)
    out = {"q": _bf16(q), "k": _bf16(k), "v": _bf16(v)}
    if do is not None:
        out["do"] = _bf16(do)
    return {n: t.to(device) for n, t in out.items()}


def ring_slice_rows(cap: int, start: int, rows: int) -> List[int]:
    """Physical ring rows written when ``rows`` tokens go to logical slot ``start``."""
    return [(start + r) % cap for r in range(rows)]


def gen_cache(cfg: CacheConfig, device: str = "cpu",
              steps: Optional[int] = None) -> Dict[str, torch.Tensor]:
    """Initial ring contents and the per-step in-flight Q/K/V.

    Draws: ring K ``[B,H,cap,d]``, ring V, then for each step s in order
    Q_s, K_s, V_s ``[B,H,W*T,d]``, then (when std_lo/std_hi differ from 1) one
    std per chunk ~ U[lo, hi] for the ``cap/T`` ring chunks in logical order
    followed by the ``W`` in-flight chunks, shared by K and V, B and H.
    Only the first ``steps`` (default ``cfg.steps``) steps are materialised; the
    draws of earlier steps never depend on how many are kept after them.
    The sink anchor (``cfg.sink`` > 0) comes from its own generator, seeded
    ``cfg.seed + 10000``: K then V ``[B,H,sink,d]``.
    """
    n_steps = cfg.steps if steps is None else steps
    g = torch.Generator("cpu").manual_seed(cfg.seed)
    rshape = (cfg.B, cfg.H, cfg.cap, cfg.d)
    qshape = (cfg.B, cfg.H, cfg.W * cfg.T, cfg.d)
    k_ring = torch.randn(rshape, generator=g, dtype=torch.float32)
    v_ring = torch.randn(rshape, generator=g, dtype=torch.float32)
    need_std = cfg.std_lo != 1.0 or cfg.std_hi != 1.0
    qs, ks, vs = [], [], []
    for s in range(cfg.steps):
        if s >= n_steps and not need_std:
            break  # later draws cannot influence the kept ones
        q = torch.randn(qshape, generator=g, dtype=torch.float32)
        k = torch.randn(qshape, generator=g, dtype=torch.float32)
        v = torch.randn(qshape, generator=g, dtype=torch.float32)
        if s < n_steps:
            qs.append(q)
            ks.append(k)
            vs.append(v)
    if need_std:
        n_ring_chunks = cfg.cap // cfg.T
        std = cfg.std_lo + (cfg.std_hi - cfg.std_lo) * torch.rand(
            (n_ring_chunks + cfg.W,), generator=g, dtype=torch.float32)
        # ring rows: physical row p holds logical token (p - head) mod cap
        logical = (torch.arange(cfg.cap) - cfg.head) % cfg.cap
        ring_std = std[logical // cfg.T].view(1, 1, cfg.cap, 1)
        k_ring = k_ring * ring_std
        v_ring = v_ring * ring_std
        new_std = std[n_ring_chunks + torch.arange(cfg.W * cfg.T) // cfg.T]
        new_std = new_std.view(1, 1, cfg.W * cfg.T, 1)
        ks = [k * new_std for k in ks]
        vs = [v * new_std for v in vs]
    out = {}
    if cfg.sink > 0:
        gs = torch.Generator("cpu").manual_seed(cfg.seed + 10000)
        sshape = (cfg.B, cfg.H, cfg.sink, cfg.d)
        out["k_sink"] = _bf16(torch.randn(sshape, generator=gs, dtype=torch.float32))
        out["v_sink"] = _bf16(torch.randn(sshape, generator=gs, dtype=torch.float32))
    out.update({
        "k_ring": _bf16(k_ring), "v_ring": _bf16(v_ring),
        "q": torch.stack([_bf16(x) for x in qs]),
        "k_new": torch.stack([_bf16(x) for x in ks]),
        "v_new": torch.stack([_bf16(x) for x in vs]),
    })
    return {n: t.to(device) for n, t in out.items()}
