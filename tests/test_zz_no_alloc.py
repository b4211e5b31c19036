"""The allocation-free ring-cache forward, mw_bca_cache_fwd_noalloc.

Some callers cannot allocate device memory: hosts that only hand the library
their own input/output buffers, and real-time streaming loops that must not
call cudaMalloc/cudaFree (those can synchronise the device).  For them the
library keeps its split-KV scratch in a fixed static device array.  These
tests call the new entry point through the C ABI and check that it returns
what the workspace-taking mw_bca_cache_fwd returns, on consecutive calls that
share the one scratch array, and that oversized requests are refused.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process.
"""
import ctypes
import math

import pytest
import torch

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_REL, LSE_REL = 2e-2, 5e-3, 1e-3


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
    a, b = o.double(), o_ref.double()
    assert torch.isfinite(a).all() and torch.isfinite(lse).all()
    assert float((a - b).abs().max()) <= O_MAX_ABS
    assert float((a - b).norm() / b.norm()) <= O_REL
    assert float(((lse - lse_ref).abs() / lse_ref.abs().clamp_min(1.0)).max()) <= LSE_REL


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(mw):
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
        q, kn, vn, kr, vr = inputs[i]
        scale = 1.0 / math.sqrt(d)
        o_ref, lse_ref = mw.mw_bca_cache_fwd(q, kn, vn, kr, vr, head, length, T, scale)
        code, o, lse = _noalloc(mw, q, kn, vn, kr, vr, head, length, T, scale)
        assert code == 0, mw.library().mw_last_error().decode()
        torch.cuda.synchronize()
        _close(o, lse, o_ref, lse_ref)
    assert mw.mw_device_status() == 0


def test_noalloc_refuses_sizes_beyond_the_scratch(mw):
    lib = mw.library()
    try:
        mw.mw_set_option("cache_splits", 16)   # 16 partials of a 3520-row, 16-head window
        need = lib.mw_bca_cache_workspace_size(1, 16, 4, 880, 128, 10560)
        assert need > (64 << 20)
        fake = ctypes.c_void_p(0x10000)
        code = lib.mw_bca_cache_fwd_noalloc(fake, fake, fake, fake, fake, 10560, 0, 10560, fake,
                                            None, 1, 16, 4, 880, 128, 0.088, None)
        assert code == 5  # MW_ERR_WORKSPACE, before anything is enqueued
        assert str(need) in lib.mw_last_error().decode()
    finally:
        mw.mw_set_option("cache_splits", 0)
