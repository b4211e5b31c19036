"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded bf16 inputs.

Tolerances (whole-tensor): O max-abs <= 2e-2 and rel-L2 <= 5e-3;
dQ/dK/dV rel-L2 <= 1e-2; LSE |err| <= 1e-3 * max(1, |LSE|).
"""
import math

import pytest
import torch

import oracle
from workloads import CACHE_CONFIGS, TRAIN_CONFIGS, gen_cache, gen_train

pytestmark = pytest.mark.gpu

O_MAX_ABS, O_REL, G_REL, LSE_REL = 2e-2, 5e-3, 1e-2, 1e-3


@pytest.fixture(scope="module")
def mw():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2608_01127_gb300 as pkg
    pkg.library()
    torch.cuda.set_device(0)
    # every in-kernel wait is bounded; keep the bound short so that a broken
    # pipeline fails fast instead of stalling each CTA for the default 2 s
    pkg.mw_set_option("wait_budget_ms", 250)
    assert pkg.mw_device_status(clear=True) == 0
    return pkg


def _rel(a, ref):
    a = a.double().cpu()
    return float((a - ref).norm() / ref.norm().clamp_min(1e-300))


def check_o(o, ref, what=""):
    a = o.double().cpu()
    max_abs = float((a - ref).abs().max())
    rel = _rel(o, ref)
    assert torch.isfinite(a).all(), what
    assert max_abs <= O_MAX_ABS and rel <= O_REL, f"{what} O max-abs {max_abs:.3e} rel-L2 {rel:.3e}"


def check_lse(lse, ref, what=""):
    a = lse.double().cpu()
    err = float(((a - ref).abs() / ref.abs().clamp_min(1.0)).max())
    assert err <= LSE_REL, f"{what} LSE rel err {err:.3e}"


def check_grad(g, ref, what=""):
    assert torch.isfinite(g.double()).all(), what
    rel = _rel(g, ref)
    assert rel <= G_REL, f"{what} rel-L2 {rel:.3e}"


def _inputs(B, H, n, T, d, seed, gain=1.0):
    g = torch.Generator().manual_seed(seed)
    shape = (B, H, n * T, d)
    q, k, v, do = (torch.randn(shape, generator=g) for _ in range(4))
    return [(t * s).to(torch.bfloat16) for t, s in ((q, gain), (k, gain), (v, 1.0), (do, 1.0))]


# ------------------------------------------------------------------ training path

def test_tiny_config_forward(mw):
    cfg = TRAIN_CONFIGS["tiny_fwd"]
    x = gen_train(cfg)
    o, lse = mw.mw_bca_fwd(*(x[n].cuda() for n in ("q", "k", "v")), cfg.T, cfg.scale)
    o_ref, lse_ref = oracle.fwd(x["q"], x["k"], x["v"], cfg.T, cfg.scale)
    check_o(o, o_ref, "tiny")
    check_lse(lse, lse_ref, "tiny")


SMALL = [
    # B, H, n_chunks, T, d, gain
    (1, 1, 1, 16, 64, 1.0),      # fewer rows than one tile
    (1, 2, 3, 100, 64, 1.0),     # chunk edges inside tiles, ragged tail
    (2, 1, 4, 64, 128, 1.0),
    (1, 1, 300, 1, 64, 1.0),     # token-causal
    (1, 2, 20, 16, 128, 2.0),
    (1, 1, 2, 880, 128, 4.0),    # one latent frame per chunk, peaky logits
    (1, 3, 5, 200, 64, 1.0),
    (1, 2, 4, 160, 64, 4.0),     # peaky logits at d = 64 (the running max jumps: O rescaled)
    (2, 2, 1, 600, 128, 1.0),    # a single chunk: full bidirectional attention
    (1, 20, 3, 96, 128, 1.0),    # the 3B head layout (20 heads of 128)
    (1, 2, 3, 100, 72, 1.0),     # the 0.5B head dim (72: 80-wide MMAs on 128-wide tiles)
    (1, 2, 3, 100, 80, 2.0),     # the widest head dim on 80-wide MMAs (ones from column 80)
    (1, 1, 2, 150, 88, 1.0),     # the narrowest on 128-wide MMAs
    (2, 1, 2, 130, 96, 2.0),     # another padded head dim
]


@pytest.mark.parametrize("B,H,n,T,d,gain", SMALL)
def test_small_shapes_forward_backward(mw, B, H, n, T, d, gain):
    q, k, v, do = _inputs(B, H, n, T, d, seed=1000 + n * T + d, gain=gain)
    sc = 1.0 / math.sqrt(d)
    qc, kc, vc, doc = (t.cuda() for t in (q, k, v, do))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, T, sc)
    dq, dk, dv = mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, T, sc)
    o_ref, lse_ref = oracle.fwd(q, k, v, T, sc)
    dq_r, dk_r, dv_r = oracle.bwd(q, k, v, do, T, sc)
    tag = f"B{B} H{H} n{n} T{T} d{d}"
    check_o(o, o_ref, tag)
    check_lse(lse, lse_ref, tag)
    check_grad(dq, dq_r, tag + " dQ")
    check_grad(dk, dk_r, tag + " dK")
    check_grad(dv, dv_r, tag + " dV")


@pytest.mark.parametrize("name", ["train_b12_d64", "train_h16_d128_peaky", "train_1b_32x600",
                                  "train_05b_d72"])
def test_full_size_training_configs(mw, name):
    """Full-size launch; the oracle recomputes two sampled (b, h) heads in full."""
    cfg = TRAIN_CONFIGS[name]
    x = gen_train(cfg)
    qc, kc, vc, doc = (x[n].cuda() for n in ("q", "k", "v", "do"))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, cfg.T, cfg.scale)
    dq, dk, dv = mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, cfg.T, cfg.scale)
    torch.cuda.synchronize()
    for b, h in ((0, 0), (cfg.B - 1, cfg.H - 1)):
        sl = (slice(b, b + 1), slice(h, h + 1))
        q, k, v, do = (x[n][sl] for n in ("q", "k", "v", "do"))
        o_ref, lse_ref = oracle.fwd(q, k, v, cfg.T, cfg.scale)
        dq_r, dk_r, dv_r = oracle.bwd(q, k, v, do, cfg.T, cfg.scale)
        tag = f"{name} b{b} h{h}"
        check_o(o[sl], o_ref, tag)
        check_lse(lse[sl], lse_ref, tag)
        check_grad(dq[sl], dq_r, tag + " dQ")
        check_grad(dk[sl], dk_r, tag + " dK")
        check_grad(dv[sl], dv_r, tag + " dV")
    assert mw.mw_device_status() == 0


@pytest.mark.parametrize("d,N,T", [(64, 65536, 4096), (128, 32768, 2048)])
def test_long_sequence_sampled_rows_and_invariants(mw, d, N, T):
    """A long sequence (16 chunks): O, LSE and dQ on sampled query rows and dK,
    dV on sampled key rows (from the second half, so that the oracle only
    needs the later queries) against the oracle's row-by-row forms; plus two
    identities that hold at any size: sum_j dK_j = 0 (each row of dS sums to
    zero) and sum_j dV_j = sum_i dO_i (each row of P sums to one)."""
    q, k, v, do = _inputs(1, 1, N // T, T, d, seed=55)
    sc = 1.0 / math.sqrt(d)
    qc, kc, vc, doc = (t.cuda() for t in (q, k, v, do))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, T, sc)
    dq, dk, dv = mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, T, sc)
    torch.cuda.synchronize()
    g = torch.Generator().manual_seed(9)
    rows = sorted(set([0, T - 1, T, N // 2, N - T, N - 1] +
                      torch.randint(0, N, (26,), generator=g).tolist()))
    q1, k1, v1, do1 = (t[0, 0] for t in (q, k, v, do))
    o_ref, lse_ref = oracle.fwd_rows(q1, k1, v1, T, sc, rows)
    check_o(o[0, 0, rows], o_ref, f"long d{d} sampled O")
    check_lse(lse[0, 0, rows], lse_ref, f"long d{d} sampled LSE")
    check_grad(dq[0, 0, rows], oracle.dq_rows(q1, k1, v1, do1, T, sc, rows), f"long d{d} sampled dQ")
    krows = sorted(set([N // 2, N // 2 + T - 1, N - T - 1, N - T, N - 1] +
                       torch.randint(N // 2, N, (11,), generator=g).tolist()))
    dk_ref, dv_ref = oracle.dkv_rows(q1, k1, v1, do1, T, sc, krows)
    check_grad(dk[0, 0, krows], dk_ref, f"long d{d} sampled dK")
    check_grad(dv[0, 0, krows], dv_ref, f"long d{d} sampled dV")
    dk64, dv64 = dk[0, 0].double().cpu(), dv[0, 0].double().cpu()
    assert float(dk64.sum(0).norm() / dk64.norm()) < 2e-2
    sum_do = do1.double().sum(0)
    assert float((dv64.sum(0) - sum_do).norm() / sum_do.norm()) < 2e-2


def test_head_groups_of_unequal_size(mw):
    """Seven heads of 64K tokens: the forward schedules its query blocks in
    head groups of about three waves of CTAs (here 2 + 2 + 2 + 1 heads),
    the larger groups first; every head's rows come out as the oracle's
    (sampled rows of a head from each group)."""
    B, H, N, T, d = 1, 7, 65536, 4096, 64
    q, k, v, _ = _inputs(B, H, N // T, T, d, seed=61)
    sc = 1.0 / math.sqrt(d)
    o, lse = mw.mw_bca_fwd(q.cuda(), k.cuda(), v.cuda(), T, sc)
    torch.cuda.synchronize()
    g = torch.Generator().manual_seed(13)
    rows = sorted(set([0, T - 1, N // 2, N - 1] + torch.randint(0, N, (8,), generator=g).tolist()))
    for h in (0, 3, 4, 6):
        o_ref, lse_ref = oracle.fwd_rows(q[0, h], k[0, h], v[0, h], T, sc, rows)
        check_o(o[0, h, rows], o_ref, f"head {h}")
        check_lse(lse[0, h, rows], lse_ref, f"head {h}")
    assert mw.mw_device_status() == 0


def test_backward_head_groups_of_unequal_size(mw):
    """Eleven heads of 16K tokens: head by head, the last head's longest key
    tiles would start near the end of the backward launch, so the key tiles
    run in head groups (here 4 + 4 + 3 heads), those of a group's heads side
    by side, the first (longest) ones first.  Sampled dQ rows and dK, dV key
    rows of a head from each group against the oracle's row-by-row forms,
    and sum_j dV_j = sum_i dO_i on every head."""
    B, H, N, T, d = 1, 11, 16384, 2048, 64
    q, k, v, do = _inputs(B, H, N // T, T, d, seed=67)
    sc = 1.0 / math.sqrt(d)
    qc, kc, vc, doc = (t.cuda() for t in (q, k, v, do))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, T, sc)
    dq, dk, dv = mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, T, sc)
    torch.cuda.synchronize()
    g = torch.Generator().manual_seed(17)
    rows = sorted(set([0, N // 2, N - 1] + torch.randint(0, N, (5,), generator=g).tolist()))
    krows = sorted(set([0, 127, 128, N - T, N - 1] + torch.randint(0, N, (3,), generator=g).tolist()))
    for h in (0, 5, 10):
        q1, k1, v1, do1 = (t[0, h] for t in (q, k, v, do))
        check_grad(dq[0, h, rows], oracle.dq_rows(q1, k1, v1, do1, T, sc, rows), f"head {h} dQ")
        dk_ref, dv_ref = oracle.dkv_rows(q1, k1, v1, do1, T, sc, krows)
        check_grad(dk[0, h, krows], dk_ref, f"head {h} dK")
        check_grad(dv[0, h, krows], dv_ref, f"head {h} dV")
    sum_do = do[0].double().sum(1)
    err = (dv[0].double().cpu().sum(1) - sum_do).norm(dim=-1) / sum_do.norm(dim=-1)
    assert float(err.max()) < 2e-2, err
    assert mw.mw_device_status() == 0


@pytest.mark.parametrize("d", [64, 72])
def test_backward_cta_order_does_not_change_the_gradients(mw, d):
    """The backward's CTA order (head by head, or head groups of any size)
    only changes when each key tile runs: dK and dV (each key tile's own)
    come out bit for bit the same, and dQ (fp32 sums in another order)
    within rounding."""
    B, H, n, T = 1, 5, 6, 256
    q, k, v, do = _inputs(B, H, n, T, d, seed=71)
    sc = 1.0 / math.sqrt(d)
    qc, kc, vc, doc = (t.cuda() for t in (q, k, v, do))
    o, lse = mw.mw_bca_fwd(qc, kc, vc, T, sc)
    results = []
    try:
        for g in (1, 2, 3, 5):
            mw.mw_set_option("bwd_group_heads", g)
            results.append(mw.mw_bca_bwd(qc, kc, vc, o, lse, doc, T, sc))
    finally:
        mw.mw_set_option("bwd_group_heads", 0)
    dq0, dk0, dv0 = results[0]
    for dq, dk, dv in results[1:]:
        assert torch.equal(dk, dk0) and torch.equal(dv, dv0)
        assert float((dq.float() - dq0.float()).norm() / dq0.float().norm()) < 1e-3
    dq_r, dk_r, dv_r = oracle.bwd(q, k, v, do, T, sc)
    check_grad(dk0, dk_r, "dK")
    check_grad(dv0, dv_r, "dV")
    check_grad(dq0, dq_r, "dQ")
    assert mw.mw_device_status() == 0


def test_forward_is_deterministic_and_stays_in_bounds(mw):
    B, H, n, T, d = 1, 2, 3, 100, 64
    q, k, v, _ = _inputs(B, H, n, T, d, seed=7)
    N = n * T
    qc, kc, vc = (t.cuda() for t in (q, k, v))
    # outputs carved out of NaN-filled buffers: the guard bands must survive
    numel = B * H * N * d
    buf = torch.full((numel + 4096,), float("nan"), dtype=torch.bfloat16, device="cuda")
    o = buf[2048:2048 + numel].view(B, H, N, d)
    lbuf = torch.full((B * H * N + 512,), float("nan"), dtype=torch.float32, device="cuda")
    lse = lbuf[256:256 + B * H * N].view(B, H, N)
    lib = mw.library()
    s = torch.cuda.current_stream().cuda_stream
    assert lib.mw_bca_fwd(qc.data_ptr(), kc.data_ptr(), vc.data_ptr(), o.data_ptr(),
                          lse.data_ptr(), B, H, n, T, d, 0.125, s) == 0
    torch.cuda.synchronize()
    assert torch.isnan(buf[:2048]).all() and torch.isnan(buf[2048 + numel:]).all()
    assert torch.isnan(lbuf[:256]).all() and torch.isnan(lbuf[256 + B * H * N:]).all()
    o2, lse2 = mw.mw_bca_fwd(qc, kc, vc, T, 0.125)
    assert torch.equal(o, o2) and torch.equal(lse, lse2)


def test_autograd_wrapper(mw):
    q, k, v, do = _inputs(1, 2, 3, 64, 64, seed=11)
    qc, kc, vc = (t.cuda().requires_grad_(True) for t in (q, k, v))
    o = mw.BlockCausalAttention.apply(qc, kc, vc, 64, None)
    o.backward(do.cuda())
    dq_r, dk_r, dv_r = oracle.bwd(q, k, v, do, 64, 0.125)
    check_grad(qc.grad, dq_r, "autograd dQ")
    check_grad(kc.grad, dk_r, "autograd dK")
    check_grad(vc.grad, dv_r, "autograd dV")


# ------------------------------------------------------------------ rolling cache

def _ring_case(B, H, W, T, cap, d, seed, std=1.0):
    g = torch.Generator().manual_seed(seed)
    q, kn, vn = (torch.randn(B, H, W * T, d, generator=g).to(torch.bfloat16) for _ in range(3))
    kr, vr = ((std * torch.randn(B, H, cap, d, generator=g)).to(torch.bfloat16) for _ in range(2))
    return q, kn, vn, kr, vr


CACHE_SMALL = [
    # B, H, W, T, cap, length, head, d, splits (0 = automatic)
    (1, 2, 1, 64, 512, 512, 100, 128, 0),
    (1, 2, 3, 100, 1000, 300, 900, 64, 0),     # partially filled ring that wraps
    (2, 1, 2, 64, 640, 0, 0, 128, 0),          # empty ring: training form
    (1, 1, 1, 880, 1760, 1760, 1759, 128, 0),  # head at cap - 1
    (1, 2, 4, 96, 1152, 1152, 576, 64, 5),     # forced split-KV
    (1, 2, 2, 130, 780, 780, 390, 128, 1),     # forced single pass
    (1, 1, 1, 16, 48, 40, 30, 64, 3),          # tiny ring, more splits than needed
    (1, 2, 2, 64, 640, 640, 320, 72, 3),       # padded head dim with split-KV
    (1, 2, 2, 200, 1200, 1000, 900, 80, 2),    # 80-wide MMAs, wrapped ring, split-KV
]


@pytest.mark.parametrize("B,H,W,T,cap,length,head,d,splits", CACHE_SMALL)
def test_cache_forward_small(mw, B, H, W, T, cap, length, head, d, splits):
    q, kn, vn, kr, vr = _ring_case(B, H, W, T, cap, d, seed=cap + head + W)
    sc = 1.0 / math.sqrt(d)
    mw.mw_set_option("cache_splits", splits)
    try:
        o, lse = mw.mw_bca_cache_fwd(q.cuda(), kn.cuda(), vn.cuda(), kr.cuda(), vr.cuda(),
                                     head, length, T, sc)
    finally:
        mw.mw_set_option("cache_splits", 0)
    o_ref, lse_ref = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, length, T, sc)
    tag = f"W{W} T{T} cap{cap} len{length} head{head} splits{splits}"
    check_o(o, o_ref, tag)
    check_lse(lse, lse_ref, tag)


def test_cache_split_count_does_not_change_the_result(mw):
    """Split-KV partials merged by the combine kernel give the unsplit result:
    every split count matches the oracle, and the runs agree with each other
    to within the oracle tolerance (their bf16 P roundings differ slightly
    because each split keeps its own running maximum)."""
    cpu = _ring_case(1, 4, 2, 200, 2400, 128, seed=5)
    q, kn, vn, kr, vr = (t.cuda() for t in cpu)
    o_ref, lse_ref = oracle.cache_fwd(*cpu, 2400, 1700, 2400, 200, 0.09)
    outs = []
    for s in (1, 2, 7, 8, 12):
        mw.mw_set_option("cache_splits", s)
        try:
            outs.append(mw.mw_bca_cache_fwd(q, kn, vn, kr, vr, 1700, 2400, 200, 0.09))
        finally:
            mw.mw_set_option("cache_splits", 0)
        check_o(outs[-1][0], o_ref, f"splits {s}")
        check_lse(outs[-1][1], lse_ref, f"splits {s}")
    for o, lse in outs[1:]:
        assert float((o.float() - outs[0][0].float()).abs().max()) <= O_MAX_ABS
        assert float(((lse - outs[0][1]).abs() / outs[0][1].abs().clamp_min(1)).max()) <= LSE_REL


def test_ring_rotation_matches(mw):
    """Rotating the physical ring while moving the head by the same amount is
    invisible (the logical key order is unchanged)."""
    cap, T = 1024, 128
    q, kn, vn, kr, vr = _ring_case(1, 2, 1, T, cap, 128, seed=9)
    o_ref, lse_ref = oracle.cache_fwd(q, kn, vn, kr, vr, cap, 0, cap, T, 128 ** -0.5)
    for r in (0, 1, 300, 1023):
        krr, vrr = torch.roll(kr, r, 2), torch.roll(vr, r, 2)
        o, lse = mw.mw_bca_cache_fwd(q.cuda(), kn.cuda(), vn.cuda(), krr.cuda(), vrr.cuda(), r,
                                     cap, T)
        check_o(o, o_ref, f"rotation {r}")
        check_lse(lse, lse_ref, f"rotation {r}")


@pytest.mark.parametrize("d", [128, 72])
def test_commit_is_bit_exact(mw, d):
    B, H, cap, rows = 2, 3, 1000, 300
    g = torch.Generator().manual_seed(3)
    kr, vr, ks, vs = (torch.randn(B, H, n, d, generator=g).to(torch.bfloat16)
                      for n in (cap, cap, rows, rows))
    for slot in (0, 650, 999):
        kg, vg = kr.cuda(), vr.cuda()
        mw.mw_bca_cache_commit(kg, vg, slot, ks.cuda(), vs.cuda())
        k_ref, v_ref = oracle.cache_commit(kr, vr, cap, slot, ks, vs)
        assert torch.equal(kg.cpu(), k_ref) and torch.equal(vg.cpu(), v_ref)


def _check_qkv(qkv, rope_dims, base, per_frame, first, got):
    """Rotated channels of Q and K within one bf16 ulp of the fp64 oracle (the
    kernel turns them in fp32 and rounds once, so near a rounding tie it may
    land on the other neighbour) plus 2^-16 absolute (the fast sine and cosine
    are good to about 2^-21 on the reduced angle, which matters where x cos
    and y sin nearly cancel), and nearly all of them rounded exactly like the
    oracle; everything else, and all of V, bit for bit."""
    ref = oracle.qkv_split_rope(qkv, rope_dims, base, per_frame, first)
    for name, g, r in zip("QKV", got, ref):
        g = g.cpu()
        rot = rope_dims if name != "V" else 0
        assert torch.equal(g[..., rot:].double(), r[..., rot:]), f"{name} unrotated channels"
        if rot:
            gr, rr = g[..., :rot].double(), r[..., :rot]
            err = (gr - rr).abs()
            assert bool((err <= rr.abs() * 2.0 ** -7 + 2.0 ** -16).all()), \
                f"{name} max err {float(err.max()):.3e}"
            same = float((g[..., :rot] == rr.to(torch.bfloat16)).double().mean())
            assert same >= 0.99, f"{name}: only {same:.4f} of rotated values round like the oracle"


@pytest.mark.parametrize("B,N,H,d,rope_dims,base,per_frame,first", [
    (2, 100, 3, 64, 32, 1e4, 7, 3),          # ragged token block, several frames per block
    (1, 77, 2, 72, 20, 500.0, 1, 0),         # d = 72; rope_dims ends inside a 16-byte piece
    (1, 64, 4, 128, 128, 1e4, 440, 1000),    # every channel turns
    (1, 50, 2, 64, 0, 1e4, 1, 0),            # plain split
    (1, 40, 1, 64, 64, 1e4, 1, (1 << 24) - 39),  # the largest positions
])
def test_qkv_split_rope(mw, B, N, H, d, rope_dims, base, per_frame, first):
    g = torch.Generator().manual_seed(17)
    qkv = torch.randn(B, N, 3, H, d, generator=g).to(torch.bfloat16)
    got = mw.mw_qkv_rope_split(qkv.cuda(), rope_dims, base, per_frame, first)
    torch.cuda.synchronize()
    _check_qkv(qkv, rope_dims, base, per_frame, first, got)
    assert mw.mw_device_status() == 0


def test_qkv_split_rope_training_shape(mw):
    """The d=64 training layout (B2 H12, 16 chunks of 880 tokens, 440 tokens
    per latent frame, 32 rotated channels): V everywhere, Q and K on two token
    ranges that start on frame boundaries (the oracle restarts there)."""
    B, N, H, d, P = 2, 16 * 880, 12, 64, 440
    g = torch.Generator().manual_seed(18)
    qkv = torch.randn(B, N, 3, H, d, generator=g).to(torch.bfloat16)
    q, k, v = mw.mw_qkv_rope_split(qkv.cuda(), 32, 1e4, P, 0)
    torch.cuda.synchronize()
    assert torch.equal(v.cpu(), qkv[:, :, 2].permute(0, 2, 1, 3))
    for t0, n in ((0, 1000), (N - 2 * P, 2 * P)):
        sl = slice(t0, t0 + n)
        part = tuple(x[:, :, sl] for x in (q, k, v))
        _check_qkv(qkv[:, sl].contiguous(), 32, 1e4, P, t0 // P, part)


@pytest.mark.parametrize("d", [64, 128])
def test_qkv_split_rope_matches_the_fused_sink_rotation(mw, d):
    """Sink keys turned by the split kernel and stored rotated give bit for bit
    the attention of the re-shift, which turns them as it reads them (both
    round the same fp32 rotation to bf16)."""
    B, H, T, cap, S, shift = 1, 2, 128, 1280, 300, 77
    g = torch.Generator().manual_seed(19)
    q, kn, vn = (torch.randn(B, H, T, d, generator=g).to(torch.bfloat16).cuda() for _ in range(3))
    kr, vr = (torch.randn(B, H, cap, d, generator=g).to(torch.bfloat16).cuda() for _ in range(2))
    ks, vs = (torch.randn(B, H, S, d, generator=g).to(torch.bfloat16).cuda() for _ in range(2))
    o1, l1 = mw.mw_bca_cache_fwd_rope(q, kn, vn, ks, vs, kr, vr, 100, cap, T, 32, 1e4, shift)
    qkv = torch.zeros(B, S, 3, H, d, dtype=torch.bfloat16, device="cuda")
    qkv[:, :, 1] = ks.permute(0, 2, 1, 3)
    _, ks_rot, _ = mw.mw_qkv_rope_split(qkv, 32, 1e4, S, shift)  # every sink token at frame `shift`
    o2, l2 = mw.mw_bca_cache_fwd_sink(q, kn, vn, ks_rot, vs, kr, vr, 100, cap, T)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


@pytest.mark.parametrize("W,T,cap,length,head,d,splits", [
    (2, 100, 1000, 1000, 700, 64, 3),    # split-KV: the commit shares the combine's launch
    (2, 100, 1000, 1000, 700, 64, 1),    # single pass: the commit runs on its own
    (1, 128, 640, 512, 88, 128, 2),      # ring not yet full; the commit wraps past its end
])
def test_cache_step_equals_forward_then_commit(mw, W, T, cap, length, head, d, splits):
    """mw_bca_cache_step gives bit for bit what mw_bca_cache_fwd followed by
    mw_bca_cache_commit of the oldest in-flight chunk gives (Sec. 3.5)."""
    q, kn, vn, kr, vr = (t.cuda() for t in _ring_case(1, 2, W, T, cap, d, seed=cap + d))
    slot = (head + length) % cap  # append position (evicts nothing until the ring is full)
    mw.mw_set_option("cache_splits", splits)
    try:
        k1, v1 = kr.clone(), vr.clone()
        o1, l1 = mw.mw_bca_cache_fwd(q, kn, vn, k1, v1, head, length, T)
        mw.mw_bca_cache_commit(k1, v1, slot, kn[:, :, :T].contiguous(), vn[:, :, :T].contiguous())
        k2, v2 = kr.clone(), vr.clone()
        o2, l2 = mw.mw_bca_cache_step(q, kn, vn, k2, v2, head, length, slot, T, T)
        torch.cuda.synchronize()
    finally:
        mw.mw_set_option("cache_splits", 0)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)
    assert mw.mw_device_status() == 0


def test_programmatic_launch_changes_nothing(mw):
    """Forward, streaming step and backward give the same bits with the
    programmatic dependent launch on and off (only the launch overlaps)."""
    q, kn, vn, kr, vr = (t.cuda() for t in _ring_case(1, 2, 2, 100, 1000, 64, seed=23))
    g = torch.Generator().manual_seed(24)
    do = torch.randn(1, 2, 200, 64, generator=g).to(torch.bfloat16).cuda()
    runs = []
    try:
        for pdl in (1, 0):
            mw.mw_set_option("pdl", pdl)
            mw.mw_set_option("cache_splits", 3)
            k1, v1 = kr.clone(), vr.clone()
            o_c, l_c = mw.mw_bca_cache_step(q, kn, vn, k1, v1, 700, 1000, 700, 100, 100)
            o, lse = mw.mw_bca_fwd(q, kn, vn, 100)
            grads = mw.mw_bca_bwd(q, kn, vn, o, lse, do, 100)
            torch.cuda.synchronize()
            runs.append((o_c, l_c, k1, v1, o, lse))
            runs[-1] += tuple(grads)
    finally:
        mw.mw_set_option("pdl", 1)
        mw.mw_set_option("cache_splits", 0)
    # dQ accumulates with floating-point atomics in no fixed order: compare it
    # to within rounding, everything else bit for bit
    for a, b in zip(runs[0][:-3], runs[1][:-3]):
        assert torch.equal(a, b)
    dq0, dq1 = runs[0][-3].double(), runs[1][-3].double()
    assert float((dq0 - dq1).norm() / dq0.norm()) < 1e-3
    for a, b in zip(runs[0][-2:], runs[1][-2:]):
        assert torch.equal(a, b)
    assert mw.mw_device_status() == 0


def test_rolling_cache_config_steps(mw):
    """The streaming workload over its full length: one 880-token chunk
    against an 8-chunk ring whose head wraps mid-buffer, 64 steps, each
    committing the chunk (FIFO eviction), so the head laps the ring eight
    times.  Every step's O and LSE are checked on two sampled heads (the
    first and the last) against the oracle run on the oracle's own ring; the
    full O of the first three steps, and the whole ring at the end (bit-exact)."""
    cfg = CACHE_CONFIGS["rolling_cache"]
    x = gen_cache(cfg)
    steps = cfg.steps
    assert steps == 64
    kr, vr = x["k_ring"].clone(), x["v_ring"].clone()
    krg, vrg = kr.cuda(), vr.cuda()
    head, length = cfg.head, cfg.length
    heads = (slice(0, 1), slice(cfg.H - 1, cfg.H))
    for s in range(steps):
        q, kn, vn = x["q"][s], x["k_new"][s], x["v_new"][s]
        o, lse = mw.mw_bca_cache_fwd(q.cuda(), kn.cuda(), vn.cuda(), krg, vrg, head, length,
                                     cfg.T, cfg.scale)
        for hs in ((slice(None),) if s < 3 else heads):
            sl = (slice(None), hs)
            o_ref, lse_ref = oracle.cache_fwd(q[sl], kn[sl], vn[sl], kr[sl], vr[sl], cfg.cap,
                                              head, length, cfg.T, cfg.scale)
            check_o(o[sl], o_ref, f"step {s} heads {hs}")
            check_lse(lse[sl], lse_ref, f"step {s} heads {hs}")
        slot, head, length = oracle.ring_advance(cfg.cap, head, length, cfg.T)
        mw.mw_bca_cache_commit(krg, vrg, slot, kn.cuda(), vn.cuda())
        kr, vr = oracle.cache_commit(kr, vr, cfg.cap, slot, kn, vn)
    assert (head, length) == ((cfg.head + steps * cfg.T) % cfg.cap, cfg.cap)
    assert torch.equal(krg.cpu(), kr) and torch.equal(vrg.cpu(), vr)
    assert mw.mw_device_status() == 0


def test_pipelined_config(mw):
    """Four in-flight chunks, block-causal among themselves, against a wrapped
    12-chunk ring with per-chunk K/V scales."""
    cfg = CACHE_CONFIGS["pipelined"]
    x = gen_cache(cfg)
    q, kn, vn = x["q"][0], x["k_new"][0], x["v_new"][0]
    o, lse = mw.mw_bca_cache_fwd(q.cuda(), kn.cuda(), vn.cuda(), x["k_ring"].cuda(),
                                 x["v_ring"].cuda(), cfg.head, cfg.length, cfg.T, cfg.scale)
    o_ref, lse_ref = oracle.cache_fwd(q, kn, vn, x["k_ring"], x["v_ring"], cfg.cap, cfg.head,
                                      cfg.length, cfg.T, cfg.scale)
    check_o(o, o_ref, "pipelined")
    check_lse(lse, lse_ref, "pipelined")


SINK_SMALL = [
    # B, H, W, T, cap, length, head, sink, d, splits (0 = automatic)
    (1, 2, 1, 64, 512, 512, 100, 32, 128, 0),     # half-chunk sink, wrapped ring
    (1, 2, 3, 100, 1000, 300, 900, 1, 64, 0),     # one sink token, partial ring
    (2, 1, 2, 64, 640, 0, 0, 200, 128, 0),        # sink only (empty ring), ragged tile
    (1, 2, 2, 96, 960, 960, 480, 128, 64, 4),     # sink of exactly one tile, forced splits
    (1, 1, 1, 880, 1760, 1760, 1759, 440, 128, 1),  # one latent frame, single pass
]


@pytest.mark.parametrize("B,H,W,T,cap,length,head,sink,d,splits", SINK_SMALL)
def test_cache_forward_with_sink(mw, B, H, W, T, cap, length, head, sink, d, splits):
    q, kn, vn, kr, vr = _ring_case(B, H, W, T, cap, d, seed=cap + head + sink)
    g = torch.Generator().manual_seed(sink + 7)
    ks, vs = (torch.randn(B, H, sink, d, generator=g).to(torch.bfloat16) for _ in range(2))
    sc = 1.0 / math.sqrt(d)
    mw.mw_set_option("cache_splits", splits)
    try:
        o, lse = mw.mw_bca_cache_fwd_sink(q.cuda(), kn.cuda(), vn.cuda(), ks.cuda(), vs.cuda(),
                                          kr.cuda(), vr.cuda(), head, length, T, sc)
    finally:
        mw.mw_set_option("cache_splits", 0)
    o_ref, lse_ref = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, length, T, sc, ks, vs)
    tag = f"sink{sink} W{W} T{T} cap{cap} len{length} head{head} splits{splits}"
    check_o(o, o_ref, tag)
    check_lse(lse, lse_ref, tag)


def test_empty_sink_is_the_plain_cache_path(mw):
    """sink_len = 0 is exactly mw_bca_cache_fwd (same kernels, same bits)."""
    q, kn, vn, kr, vr = (t.cuda() for t in _ring_case(1, 2, 2, 128, 1024, 128, seed=31))
    o0, l0 = mw.mw_bca_cache_fwd(q, kn, vn, kr, vr, 300, 1024, 128)
    empty = torch.empty(1, 2, 0, 128, dtype=torch.bfloat16, device="cuda")
    o1, l1 = mw.mw_bca_cache_fwd_sink(q, kn, vn, empty, empty, kr, vr, 300, 1024, 128)
    assert torch.equal(o0, o1) and torch.equal(l0, l1)


def test_sink_anchor_config(mw):
    """Eight in-flight chunks against a wrapped 12-chunk ring behind a one-frame
    (440-token) sink anchor; the oracle checks two of the 16 heads."""
    cfg = CACHE_CONFIGS["sink_anchor"]
    x = gen_cache(cfg)
    q, kn, vn = x["q"][0], x["k_new"][0], x["v_new"][0]
    o, lse = mw.mw_bca_cache_fwd_sink(q.cuda(), kn.cuda(), vn.cuda(), x["k_sink"].cuda(),
                                      x["v_sink"].cuda(), x["k_ring"].cuda(), x["v_ring"].cuda(),
                                      cfg.head, cfg.length, cfg.T, cfg.scale)
    heads = [0, 11]
    sel = lambda t: t[:, heads]
    o_ref, lse_ref = oracle.cache_fwd(sel(q), sel(kn), sel(vn), sel(x["k_ring"]), sel(x["v_ring"]),
                                      cfg.cap, cfg.head, cfg.length, cfg.T, cfg.scale,
                                      sel(x["k_sink"]), sel(x["v_sink"]))
    check_o(o[:, heads], o_ref, "sink_anchor")
    check_lse(lse[:, heads], lse_ref, "sink_anchor")


ROPE_SMALL = [
    # B, H, W, T, cap, length, head, sink, d, rope_dims, shift, splits (0 = automatic)
    (1, 2, 1, 64, 512, 512, 100, 32, 128, 32, 8, 0),          # a quarter-tile sink
    (1, 2, 2, 100, 1000, 300, 900, 32, 64, 64, 1000, 0),      # every channel, a large shift
    (1, 1, 1, 880, 1760, 1760, 1759, 440, 128, 16, 4, 3),     # one-frame sink, forced splits
    (2, 1, 2, 64, 640, 640, 0, 200, 64, 2, 1, 0),             # sink over two tiles, one pair
    (1, 2, 1, 64, 512, 512, 200, 16, 72, 24, 7, 2),           # padded head dim, splits
    (1, 2, 1, 64, 512, 512, 300, 130, 64, 64, (1 << 24) - 5, 0),  # the largest shifts
    (1, 2, 1, 64, 512, 512, 300, 0, 64, 32, 50, 0),           # no sink: nothing turns
    (1, 2, 1, 64, 512, 512, 300, 64, 64, 32, 0, 0),           # nothing evicted yet
]


@pytest.mark.parametrize("B,H,W,T,cap,length,head,sink,d,rope_dims,shift,splits", ROPE_SMALL)
def test_cache_forward_rope_reshift(mw, B, H, W, T, cap, length, head, sink, d, rope_dims, shift,
                                    splits):
    """Queries, in-flight and ring keys stand for keys rotated at stream
    positions (any bf16 values are), the sink for keys at its own position;
    the oracle re-indexes the window by the shift as Sec. 3.5 describes."""
    q, kn, vn, kr, vr = _ring_case(B, H, W, T, cap, d, seed=cap + rope_dims + sink)
    g = torch.Generator().manual_seed(sink + 11)
    ks, vs = (torch.randn(B, H, sink, d, generator=g).to(torch.bfloat16) for _ in range(2))
    sc, base = 1.0 / math.sqrt(d), 10000.0
    mw.mw_set_option("cache_splits", splits)
    try:
        o, lse = mw.mw_bca_cache_fwd_rope(q.cuda(), kn.cuda(), vn.cuda(),
                                          ks.cuda() if sink else None, vs.cuda() if sink else None,
                                          kr.cuda(), vr.cuda(), head, length, T, rope_dims, base,
                                          shift, sc)
    finally:
        mw.mw_set_option("cache_splits", 0)
    o_ref, lse_ref = oracle.cache_fwd_reshift(q, kn, vn, kr, vr, cap, head, length, T, sc, ks, vs,
                                              rope_dims, base, shift)
    tag = f"rope{rope_dims} shift{shift} sink{sink} len{length} splits{splits}"
    check_o(o, o_ref, tag)
    check_lse(lse, lse_ref, tag)


def test_rope_reshift_streaming(mw):
    """Streaming with a one-frame sink and a FIFO ring: every chunk's queries
    and keys are rotated once, at their stream frames (frame 0 is the sink's,
    the stream's tokens follow from frame 1), and the keys are committed as
    they are; after evictions the window is re-indexed by the evicted frames,
    which here only turns the sink as it is read."""
    B, H, T, d, P, cap, sink = 1, 2, 64, 128, 32, 256, 32
    rope_dims, base, sc = 32, 10000.0, 1.0 / math.sqrt(d)
    g = torch.Generator().manual_seed(41)
    ks, vs = (torch.randn(B, H, sink, d, generator=g).to(torch.bfloat16) for _ in range(2))
    ks = oracle.rope_rotate(ks, torch.zeros(sink, dtype=torch.long), rope_dims, base).to(torch.bfloat16)
    kr = torch.zeros(B, H, cap, d, dtype=torch.bfloat16)
    vr = torch.zeros(B, H, cap, d, dtype=torch.bfloat16)
    ring = mw.RingState(cap, 0, 0)
    kr_g, vr_g = kr.cuda(), vr.cuda()
    evicted = 0  # tokens that have left the ring
    for step in range(7):  # the ring fills after 4 steps, then evicts
        q_raw, k_raw, v_new = (torch.randn(B, H, T, d, generator=g).to(torch.bfloat16)
                               for _ in range(3))
        frames = 1 + (step * T + torch.arange(T)) // P
        q = oracle.rope_rotate(q_raw, frames, rope_dims, base).to(torch.bfloat16)
        k = oracle.rope_rotate(k_raw, frames, rope_dims, base).to(torch.bfloat16)
        shift = evicted // P
        o, lse = mw.mw_bca_cache_fwd_rope(q.cuda(), k.cuda(), v_new.cuda(), ks.cuda(), vs.cuda(),
                                          kr_g, vr_g, ring.head, ring.length, T, rope_dims, base,
                                          shift, sc)
        o_ref, lse_ref = oracle.cache_fwd_reshift(q, k, v_new, kr, vr, cap, ring.head, ring.length,
                                                  T, sc, ks, vs, rope_dims, base, shift)
        check_o(o, o_ref, f"stream step {step} shift {shift}")
        check_lse(lse, lse_ref, f"stream step {step}")
        before = ring.length
        slot = ring.commit(T)
        evicted += before + T - ring.length
        mw.mw_bca_cache_commit(kr_g, vr_g, slot, k.cuda(), v_new.cuda())
        kr, vr = oracle.cache_commit(kr, vr, cap, slot, k, v_new)
    assert evicted == 3 * T


def test_device_status_is_clean(mw):
    torch.cuda.synchronize()
    assert mw.mw_device_status() == 0


def test_cuda_graph_replay_matches_eager(mw):
    """A training step and a streaming step captured once as CUDA graphs and
    replayed give the eager results (the entry points only enqueue work on
    the caller's stream)."""
    B, H, n, T, d = 1, 2, 3, 128, 64
    q, k, v, do = (t.cuda() for t in _inputs(B, H, n, T, d, seed=21))
    o_e, lse_e = mw.mw_bca_fwd(q, k, v, T)
    dq_e, dk_e, dv_e = mw.mw_bca_bwd(q, k, v, o_e, lse_e, do, T)
    ws = torch.empty(mw.mw_bca_bwd_workspace_size(B, H, n, T, d), dtype=torch.uint8, device="cuda")
    cq, ckn, cvn, ckr, cvr = (t.cuda() for t in _ring_case(1, 2, 2, 64, 512, 128, seed=22))
    cws = torch.empty(max(1, mw.mw_bca_cache_workspace_size(1, 2, 2, 64, 128, 512)),
                      dtype=torch.uint8, device="cuda")
    co_e, clse_e = mw.mw_bca_cache_fwd(cq, ckn, cvn, ckr, cvr, 100, 512, 64, workspace=cws)
    kr_g, vr_g = ckr.clone(), cvr.clone()
    kr_e, vr_e = ckr.clone(), cvr.clone()
    mw.mw_bca_cache_commit(kr_e, vr_e, 100, ckn, cvn)
    out = {}
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            out["o"], out["lse"] = mw.mw_bca_fwd(q, k, v, T)
            out["grads"] = mw.mw_bca_bwd(q, k, v, out["o"], out["lse"], do, T, workspace=ws)
            out["co"], out["clse"] = mw.mw_bca_cache_fwd(cq, ckn, cvn, kr_g, vr_g, 100, 512, 64,
                                                         workspace=cws)
            mw.mw_bca_cache_commit(kr_g, vr_g, 100, ckn, cvn)
    torch.cuda.current_stream().wait_stream(side)
    graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(out["o"], o_e) and torch.equal(out["lse"], lse_e)
    for g_, e_ in zip(out["grads"], (dq_e, dk_e, dv_e)):
        assert float((g_.float() - e_.float()).abs().max()) <= 1e-2
    assert torch.equal(out["co"], co_e) and torch.equal(out["clse"], clse_e)
    assert torch.equal(kr_g, kr_e) and torch.equal(vr_g, vr_e)
    assert mw.mw_device_status() == 0
