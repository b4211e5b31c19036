"""fp64 CPU oracle for block-causal attention: test infrastructure, not product.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline /
reference arm may import this package.  The CUDA path never calls it.
Every function is pinned by ``tests/test_oracle.py`` (worked examples, library
special cases, invariants, finite differences, brute force).
"""
from .bca import (  # noqa: F401
    F64, block_causal_mask, bwd, bwd_dense, cache_commit, cache_fwd, cache_fwd_reshift, chunk_of, dkv_rows, dq_rows,
    fwd, fwd_dense, fwd_loops, fwd_rows, probs_dense, qkv_split_rope, ring_advance,
    ring_logical, rope_rotate,
)
