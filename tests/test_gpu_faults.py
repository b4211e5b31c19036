"""Failure detection without a GPU fault.

Every wait inside the kernels is bounded.  A test-only option makes the
forward kernel skip its Q load, so the MMA warp's wait for Q can never
complete: after the (short) budget it records a timeout in the device status
word, releases the other roles of its CTA through a shared abort flag, lets
in-flight copies land, frees its tensor memory and returns.  Nothing traps or
hangs; the host reads MW_ERR_TIMEOUT and the context stays usable.
"""
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

MW_OK, MW_ERR_TIMEOUT = 0, 4


@pytest.fixture(scope="module")
def mw():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2608_01127_gb300 as pkg
    pkg.library()
    torch.cuda.set_device(0)
    assert pkg.mw_device_status(clear=True) == MW_OK
    return pkg


def _small():
    g = torch.Generator().manual_seed(5)
    return [torch.randn(1, 1, 256, 64, generator=g).to(torch.bfloat16) for _ in range(3)]


def test_expired_wait_is_reported_and_the_context_survives(mw):
    q, k, v = _small()
    qc, kc, vc = (t.cuda() for t in (q, k, v))
    mw.mw_set_option("wait_budget_ms", 100)
    mw.mw_set_option("debug_skip_q_load", 1)
    try:
        mw.mw_bca_fwd(qc, kc, vc, 64)        # one CTA; enqueues and returns
        status = mw.mw_device_status(clear=True)
        message = mw.library().mw_last_error().decode()
    finally:
        mw.mw_set_option("debug_skip_q_load", 0)
        mw.mw_set_option("wait_budget_ms", 2000)
    assert status == MW_ERR_TIMEOUT
    assert "expired" in message
    # the same context keeps working, and the status word was cleared
    o, lse = mw.mw_bca_fwd(qc, kc, vc, 64)
    torch.cuda.synchronize()
    assert mw.mw_device_status() == MW_OK
    o_ref, _ = oracle.fwd(q, k, v, 64, 0.125)
    assert float((o.double().cpu() - o_ref).abs().max()) <= 2e-2
