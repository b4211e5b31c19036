"""Failure detection without a GPU fault.

Every wait inside the kernels is bounded.  A test-only option makes the
forward and backward kernels skip their Q loads, so the MMA warp's wait for
Q can never complete: after the (short) budget it records a timeout in the
device status word, releases the other roles of its CTA through a shared
abort flag, lets in-flight copies land, gives its outputs a defined value
(O = 0 and LSE = -inf; dK = dV = 0), frees its tensor memory and returns.
Nothing traps or hangs; the host reads MW_ERR_TIMEOUT and the context stays
usable.
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
        o_bad, lse_bad = mw.mw_bca_fwd(qc, kc, vc, 64)   # one CTA; enqueues and returns
        status = mw.mw_device_status(clear=True)
        message = mw.library().mw_last_error().decode()
    finally:
        mw.mw_set_option("debug_skip_q_load", 0)
        mw.mw_set_option("wait_budget_ms", 2000)
    assert status == MW_ERR_TIMEOUT
    assert "expired" in message
    assert torch.count_nonzero(o_bad) == 0
    assert bool((lse_bad == float("-inf")).all())
    # the same context keeps working, and the status word was cleared
    o, lse = mw.mw_bca_fwd(qc, kc, vc, 64)
    torch.cuda.synchronize()
    assert mw.mw_device_status() == MW_OK
    o_ref, _ = oracle.fwd(q, k, v, 64, 0.125)
    assert float((o.double().cpu() - o_ref).abs().max()) <= 2e-2


def test_expired_backward_wait_leaves_zero_key_gradients(mw):
    q, k, v = _small()
    do = torch.randn(q.shape, generator=torch.Generator().manual_seed(6)).to(torch.bfloat16)
    qc, kc, vc, doc = (t.cuda() for t in (q, k, v, do))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, 64)
    outs = tuple(torch.full_like(qc, float("nan")) for _ in range(3))
    mw.mw_set_option("wait_budget_ms", 100)
    mw.mw_set_option("debug_skip_q_load", 1)
    try:
        mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, 64, out=outs)   # two key-tile CTAs
        status = mw.mw_device_status(clear=True)
    finally:
        mw.mw_set_option("debug_skip_q_load", 0)
        mw.mw_set_option("wait_budget_ms", 2000)
    assert status == MW_ERR_TIMEOUT
    # no CTA got past its first wait: nothing reduced into dQ, and every
    # key row's dK and dV came out as zeros rather than the NaN fill
    for t in outs:
        assert torch.count_nonzero(t) == 0
    dq, dk, dv = mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, 64)
    torch.cuda.synchronize()
    assert mw.mw_device_status() == MW_OK
    refs = oracle.bwd(q, k, v, do, 64, 0.125)
    for g, r in zip((dq, dk, dv), refs):
        assert float((g.double().cpu() - r).norm() / r.norm()) <= 1e-2
