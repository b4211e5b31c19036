"""The bench's work accounting against the oracle (CPU only).

The bench counts FLOPs over unmasked (query, key) pairs in closed form.  With
all queries zero every visible key scores the same, so the oracle's LSE of a
row is ln(number of keys that row sees): summing exp(LSE) over the rows
counts the unmasked pairs through the oracle's own visibility rules, with no
formula shared with the bench.
"""
import math
import os
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import oracle  # noqa: E402
from workloads import CacheConfig, TrainConfig  # noqa: E402


def _visible_pairs(lse: torch.Tensor) -> int:
    counts = torch.exp(lse.double())
    assert torch.allclose(counts, counts.round(), atol=1e-6)
    return int(counts.round().sum().item())


@pytest.mark.parametrize("B,H,n,T", [(1, 1, 1, 8), (2, 3, 4, 5), (1, 2, 7, 3), (1, 1, 12, 1)])
def test_training_pairs_match_the_oracle(B, H, n, T):
    cfg = TrainConfig("t", B=B, H=H, d=8, n_chunks=n, T=T, seed=0)
    q = torch.zeros(B, H, n * T, 8)
    k = torch.randn(B, H, n * T, 8)
    _, lse = oracle.fwd(q, k, k, T, 1.0)
    assert bench.train_pairs(cfg) == _visible_pairs(lse)


@pytest.mark.parametrize("B,H,W,T,cap,length,head,sink", [
    (1, 1, 1, 4, 16, 16, 5, 0),
    (2, 2, 3, 4, 20, 12, 17, 0),
    (1, 2, 2, 5, 15, 0, 0, 0),
    (1, 1, 4, 3, 12, 12, 11, 6),
])
def test_cache_pairs_match_the_oracle(B, H, W, T, cap, length, head, sink):
    cfg = CacheConfig("c", B=B, H=H, d=8, W=W, T=T, cap=cap, length=length, head=head, steps=1,
                      seed=0, sink=sink)
    d = 8
    q = torch.zeros(B, H, W * T, d)
    kn = torch.randn(B, H, W * T, d)
    kr = torch.randn(B, H, cap, d)
    ks = torch.randn(B, H, sink, d) if sink else None
    _, lse = oracle.cache_fwd(q, kn, kn, kr, kr, cap, head, length, T, 1.0, ks, ks)
    assert bench.cache_pairs(cfg) == _visible_pairs(lse)


def test_flop_conventions():
    """Forward: QK^T and PV, 2 FLOPs per multiply-add over d each (4 d per
    pair).  Backward: S recomputed, dP, dV, dK and dQ (10 d per pair)."""
    assert bench.fwd_flops(3, 64) == 4 * 64 * 3
    assert bench.bwd_flops(3, 64) == 10 * 64 * 3


def test_headline_workload_size():
    """train_b12_d64: 24 heads of 16 chunks x 880 tokens, 136 chunk pairs per
    head (2.53e9 unmasked pairs), 2.26 TFLOP per fwd+bwd step."""
    cfg = bench.TRAIN_CONFIGS[bench.WORKLOAD]
    pairs = bench.train_pairs(cfg)
    assert pairs == 24 * 880 * 880 * 136
    flops = bench.fwd_flops(pairs, cfg.d) + bench.bwd_flops(pairs, cfg.d)
    assert math.isclose(flops, 2264766873600.0)
