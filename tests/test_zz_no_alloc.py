"""The allocation-free ring-cache forward, mw_bca_cache_fwd_noalloc.

Some callers cannot allocate device memory: hosts that only hand the library
their own input/output buffers, and real-time streaming loops that must not
call cudaMalloc/cudaFree (those can synchronise the device).  For them the
library keeps its split-KV scratch in a fixed static device array.  These
tests call the new entry point through the C ABI and check its results
against the fp64 oracle (and bit for bit against the workspace-taking
mw_bca_cache_fwd, which runs the same kernels and split plan) on consecutive
calls that share the one scratch array, on a request that fills the array to
within 4 KB, and that requests beyond it are refused before anything runs.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process.
"""
import math

import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_REL, LSE_REL = 2e-2, 5e-3, 1e-3
MW_NOALLOC_SCRATCH_BYTES = 64 << 20  # include/mw_bca.h


@pytest.fixture(scope="module")
def mw():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2608_01127_gb300 as pkg
    pkg.library()
    torch.cuda.set_device(0)
    pkg.mw_set_option("cache_splits", 0)
    return pkg


def _case(B, H, W, T, cap, d, seed):
    g = torch.Generator().manual_seed(seed)
    q, kn, vn = (torch.randn(B, H, W * T, d, generator=g).to(torch.bfloat16).cuda()
                 for _ in range(3))
    kr, vr = (torch.randn(B, H, cap, d, generator=g).to(torch.bfloat16).cuda() for _ in range(2))
    return q, kn, vn, kr, vr


def _noalloc(mw, q, kn, vn, kr, vr, head, length, T, scale):
    B, H, M, d = q.shape
    cap = kr.shape[2]
    o = torch.full_like(q, float("nan"))
    lse = torch.full((B, H, M), float("nan"), dtype=torch.float32, device=q.device)
    code = mw.library().mw_bca_cache_fwd_noalloc(
        q.data_ptr(), kn.data_ptr(), vn.data_ptr(), kr.data_ptr(), vr.data_ptr(), cap, head,
        length, o.data_ptr(), lse.data_ptr(), B, H, M // T, T, d, scale,
        torch.cuda.current_stream().cuda_stream)
    return code, o, lse


def _close(o, lse, o_ref, lse_ref):
    a, b = o.double().cpu(), o_ref.double()
    assert torch.isfinite(a).all() and torch.isfinite(lse).all()
    assert float((a - b).abs().max()) <= O_MAX_ABS
    assert float((a - b).norm() / b.norm()) <= O_REL
    err = (lse.double().cpu() - lse_ref).abs() / lse_ref.abs().clamp_min(1.0)
    assert float(err.max()) <= LSE_REL


def _check(mw, case, inputs, heads):
    """One allocation-free call: bit-identical to the workspace entry point,
    and within the tolerances of the oracle on the sampled heads."""
    B, H, W, T, cap, length, head, d = case
    q, kn, vn, kr, vr = inputs
    scale = 1.0 / math.sqrt(d)
    code, o, lse = _noalloc(mw, q, kn, vn, kr, vr, head, length, T, scale)
    assert code == 0, mw.library().mw_last_error().decode()
    o_ws, lse_ws = mw.mw_bca_cache_fwd(q, kn, vn, kr, vr, head, length, T, scale)
    torch.cuda.synchronize()
    assert torch.equal(o, o_ws) and torch.equal(lse, lse_ws)
    for h in heads:
        sl = (slice(None), slice(h, h + 1))
        o_ref, lse_ref = oracle.cache_fwd(q[sl].cpu(), kn[sl].cpu(), vn[sl].cpu(), kr[sl].cpu(),
                                          vr[sl].cpu(), cap, head, length, T, scale)
        _close(o[sl], lse[sl], o_ref, lse_ref)


def test_noalloc_matches_the_oracle_on_consecutive_calls(mw):
    # two different workloads back to back: the second call reuses the scratch
    # the first one left behind; then the first workload again
    cases = [
        # B, H, W, T, cap, length, head, d   (both use split-KV partials)
        (1, 16, 1, 880, 7040, 7040, 4400, 128),
        (1, 4, 3, 200, 3000, 2600, 2900, 64),
    ]
    inputs = [_case(*c[:5], c[7], seed=21 + i) for i, c in enumerate(cases)]
    for i in (0, 1, 0):
        B, H, W, T, cap, length, head, d = cases[i]
        assert mw.mw_bca_cache_workspace_size(B, H, W, T, d, length) > 0
        _check(mw, cases[i], inputs[i], heads=(0, H - 1))
    assert mw.mw_device_status() == 0


def test_noalloc_fills_the_scratch_to_the_limit(mw):
    # 16 forced splits of 16 heads x 508 rows at d = 128: the partials take
    # 4 KB less than the whole array
    case = (1, 16, 2, 254, 2048, 2048, 1000, 128)
    B, H, W, T, cap, length, head, d = case
    try:
        mw.mw_set_option("cache_splits", 16)
        need = mw.mw_bca_cache_workspace_size(B, H, W, T, d, length)
        assert MW_NOALLOC_SCRATCH_BYTES - 4096 <= need <= MW_NOALLOC_SCRATCH_BYTES
        _check(mw, case, _case(B, H, W, T, cap, d, seed=31), heads=(0, 7, H - 1))
    finally:
        mw.mw_set_option("cache_splits", 0)
    assert mw.mw_device_status() == 0


@pytest.mark.parametrize("splits,B,H,W,T,cap,d", [
    (16, 1, 16, 4, 880, 10560, 128),   # far beyond: 16 partials of a 16-head window
    (2, 1, 4, 1, 32265, 512, 64),      # 2560 bytes beyond
])
def test_noalloc_refuses_sizes_beyond_the_scratch(mw, splits, B, H, W, T, cap, d):
    # real buffers of the full sizes, so that even a broken size check could
    # only read and write memory that belongs to this test
    lib = mw.library()
    q, kn, vn, kr, vr = (torch.zeros(B, H, r, d, dtype=torch.bfloat16, device="cuda")
                         for r in (W * T, W * T, W * T, cap, cap))
    o = torch.zeros_like(q)
    lse = torch.zeros(B, H, W * T, dtype=torch.float32, device="cuda")
    try:
        mw.mw_set_option("cache_splits", splits)
        need = lib.mw_bca_cache_workspace_size(B, H, W, T, d, cap)
        assert need > MW_NOALLOC_SCRATCH_BYTES
        code = lib.mw_bca_cache_fwd_noalloc(q.data_ptr(), kn.data_ptr(), vn.data_ptr(),
                                            kr.data_ptr(), vr.data_ptr(), cap, 0, cap,
                                            o.data_ptr(), lse.data_ptr(), B, H, W, T, d,
                                            1.0 / math.sqrt(d),
                                            torch.cuda.current_stream().cuda_stream)
        assert code == 5  # MW_ERR_WORKSPACE, before anything is enqueued
        assert str(need) in lib.mw_last_error().decode()
        torch.cuda.synchronize()
        assert not o.any() and not lse.any()  # nothing ran
    finally:
        mw.mw_set_option("cache_splits", 0)
