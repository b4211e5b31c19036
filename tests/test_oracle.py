"""Pins of the fp64 oracle against things other than itself (CPU only).

Worked examples derived by hand, special cases that reduce to PyTorch's own
scaled-dot-product attention, invariants fixed by the definition of
block-causal attention (Sec. 3.2), central finite differences for the
gradients, and brute-force scalar loops.  The rolling-cache functions are
pinned to the training form over the unrolled key sequence and to ring
rotation (Sec. 3.5).
"""
import json
import math
import os

import pytest
import torch
import torch.nn.functional as F

import oracle

F64 = torch.float64


def _rand(*shape, seed=0, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return scale * torch.randn(*shape, generator=g, dtype=F64)


def _kron_mask(n, T):
    """Block-causal mask built independently: lower-triangular chunk matrix
    (chunk c sees chunks <= c) expanded by an all-ones T x T block."""
    return torch.kron(torch.tril(torch.ones(n, n)), torch.ones(T, T)).bool()


# ---------------------------------------------------------------- worked examples

def _golden(golden_dir):
    with open(os.path.join(golden_dir, "worked_examples.json")) as f:
        return json.load(f)["cases"]


def test_worked_examples_all_forms(golden_dir):
    for case in _golden(golden_dir):
        T, sc = case["T"], case["scale"]
        q = torch.tensor(case["q"], dtype=F64)
        k = torch.tensor(case["k"], dtype=F64)
        v = torch.tensor(case["v"], dtype=F64)
        do = torch.tensor(case["do"], dtype=F64)
        exp_o = torch.tensor(case["o"], dtype=F64)
        exp_lse = torch.tensor(case["lse"], dtype=F64)
        # scalar loops
        o_l, lse_l = oracle.fwd_loops(case["q"], case["k"], case["v"], T, sc)
        assert torch.allclose(torch.tensor(o_l, dtype=F64), exp_o, atol=1e-14, rtol=0)
        assert torch.allclose(torch.tensor(lse_l, dtype=F64), exp_lse, atol=1e-14, rtol=0)
        # dense and row-block, as [1,1,N,d]
        q4, k4, v4, do4 = (t[None, None] for t in (q, k, v, do))
        for o, lse in (oracle.fwd_dense(q4, k4, v4, T, sc), oracle.fwd(q4, k4, v4, T, sc)):
            assert torch.allclose(o[0, 0], exp_o, atol=1e-14, rtol=0), case["name"]
            assert torch.allclose(lse[0, 0], exp_lse, atol=1e-14, rtol=0), case["name"]
        p = oracle.probs_dense(q4, k4, T, sc)[0, 0]
        assert torch.allclose(p, torch.tensor(case["p"], dtype=F64), atol=1e-15, rtol=0)
        for dq, dk, dv in (oracle.bwd(q4, k4, v4, do4, T, sc),
                           oracle.bwd_dense(q4, k4, v4, do4, T, sc)):
            assert torch.allclose(dq[0, 0], torch.tensor(case["dq"], dtype=F64), atol=1e-14, rtol=0)
            assert torch.allclose(dk[0, 0], torch.tensor(case["dk"], dtype=F64), atol=1e-14, rtol=0)
            assert torch.allclose(dv[0, 0], torch.tensor(case["dv"], dtype=F64), atol=1e-14, rtol=0)


# ---------------------------------------------------------------- library special cases

@pytest.mark.parametrize("T,d", [(16, 8), (37, 16), (64, 64)])
def test_one_chunk_is_full_attention(T, d):
    q, k, v = (_rand(2, 3, T, d, seed=s) for s in (1, 2, 3))
    sc = 1.0 / math.sqrt(d)
    o, lse = oracle.fwd(q, k, v, T, sc)
    ref = F.scaled_dot_product_attention(q, k, v, scale=sc)
    assert torch.allclose(o, ref, atol=1e-12, rtol=0)
    ref_lse = torch.logsumexp(sc * q @ k.transpose(-1, -2), dim=-1)
    assert torch.allclose(lse, ref_lse, atol=1e-12, rtol=0)


@pytest.mark.parametrize("N,d", [(7, 4), (40, 16), (96, 32)])
def test_token_chunks_are_causal_attention(N, d):
    q, k, v = (_rand(1, 2, N, d, seed=s) for s in (4, 5, 6))
    sc = 0.3
    o, lse = oracle.fwd(q, k, v, 1, sc)
    ref = F.scaled_dot_product_attention(q, k, v, is_causal=True, scale=sc)
    assert torch.allclose(o, ref, atol=1e-12, rtol=0)
    causal = torch.ones(N, N).tril().bool()
    s = (sc * q @ k.transpose(-1, -2)).masked_fill(~causal, float("-inf"))
    assert torch.allclose(lse, torch.logsumexp(s, dim=-1), atol=1e-12, rtol=0)


@pytest.mark.parametrize("n,T,d", [(3, 5, 8), (4, 16, 16), (6, 11, 32)])
def test_general_mask_vs_library_with_kron_mask(n, T, d):
    N = n * T
    q, k, v = (_rand(2, 2, N, d, seed=s) for s in (7, 8, 9))
    sc = 1.0 / math.sqrt(d)
    mask = _kron_mask(n, T)
    ref = F.scaled_dot_product_attention(q, k, v, attn_mask=mask, scale=sc)
    for o, _ in (oracle.fwd(q, k, v, T, sc), oracle.fwd_dense(q, k, v, T, sc)):
        assert torch.allclose(o, ref, atol=1e-12, rtol=0)
    assert torch.equal(oracle.block_causal_mask(N, T), mask)
    # library autograd of the library routine pins the analytic backward
    qa, ka, va = (t.clone().requires_grad_(True) for t in (q, k, v))
    do = _rand(2, 2, N, d, seed=10)
    F.scaled_dot_product_attention(qa, ka, va, attn_mask=mask, scale=sc).backward(do)
    for dq, dk, dv in (oracle.bwd(q, k, v, do, T, sc), oracle.bwd_dense(q, k, v, do, T, sc)):
        assert torch.allclose(dq, qa.grad, atol=1e-11, rtol=0)
        assert torch.allclose(dk, ka.grad, atol=1e-11, rtol=0)
        assert torch.allclose(dv, va.grad, atol=1e-11, rtol=0)


# ---------------------------------------------------------------- brute force

@pytest.mark.parametrize("n,T,d", [(1, 3, 2), (3, 2, 3), (4, 3, 5), (2, 7, 4)])
def test_loops_dense_rowblock_agree(n, T, d):
    N = n * T
    q, k, v = (_rand(N, d, seed=s) for s in (11, 12, 13))
    sc = 0.7
    o_l, lse_l = oracle.fwd_loops(q.tolist(), k.tolist(), v.tolist(), T, sc)
    o_l, lse_l = torch.tensor(o_l, dtype=F64), torch.tensor(lse_l, dtype=F64)
    o_d, lse_d = oracle.fwd_dense(q, k, v, T, sc)
    o_r, lse_r = oracle.fwd(q[None, None], k[None, None], v[None, None], T, sc)
    o_s, lse_s = oracle.fwd_rows(q, k, v, T, sc, range(N))
    for o, lse in ((o_d, lse_d), (o_r[0, 0], lse_r[0, 0]), (o_s, lse_s)):
        assert torch.allclose(o, o_l, atol=1e-13, rtol=0)
        assert torch.allclose(lse, lse_l, atol=1e-13, rtol=0)


# ---------------------------------------------------------------- invariants

def test_probability_rows_sum_to_one_and_mask_is_zero():
    n, T, d = 5, 6, 8
    q, k = _rand(1, 2, n * T, d, seed=14, scale=3.0), _rand(1, 2, n * T, d, seed=15, scale=3.0)
    p = oracle.probs_dense(q, k, T, 0.5)
    assert torch.allclose(p.sum(-1), torch.ones(1, 2, n * T, dtype=F64), atol=1e-12, rtol=0)
    assert torch.all(p[..., ~_kron_mask(n, T)] == 0)
    assert torch.all(p[..., _kron_mask(n, T)] > 0)


def test_permutation_within_a_chunk():
    n, T, d = 4, 8, 16
    N = n * T
    q, k, v = (_rand(1, 1, N, d, seed=s) for s in (16, 17, 18))
    sc = 0.25
    o, lse = oracle.fwd(q, k, v, T, sc)
    g = torch.Generator().manual_seed(19)
    for c in range(n):
        perm = torch.arange(N)
        perm[c * T:(c + 1) * T] = c * T + torch.randperm(T, generator=g)
        # permuting queries permutes output rows
        o_q, lse_q = oracle.fwd(q[:, :, perm], k, v, T, sc)
        assert torch.allclose(o_q, o[:, :, perm], atol=1e-13, rtol=0)
        assert torch.allclose(lse_q, lse[:, :, perm], atol=1e-13, rtol=0)
        # permuting keys and values together leaves every output unchanged
        o_kv, lse_kv = oracle.fwd(q, k[:, :, perm], v[:, :, perm], T, sc)
        assert torch.allclose(o_kv, o, atol=1e-13, rtol=0)
        assert torch.allclose(lse_kv, lse, atol=1e-13, rtol=0)


def test_permutation_across_chunks_changes_output():
    """Moving a key to an earlier chunk must change the result (guards an
    all-visible mask)."""
    n, T, d = 3, 4, 8
    q, k, v = (_rand(1, 1, n * T, d, seed=s) for s in (20, 21, 22))
    o, _ = oracle.fwd(q, k, v, T, 0.5)
    perm = torch.arange(n * T)
    perm[0], perm[n * T - 1] = n * T - 1, 0
    o2, _ = oracle.fwd(q, k[:, :, perm], v[:, :, perm], T, 0.5)
    assert not torch.allclose(o[:, :, :T], o2[:, :, :T])


@pytest.mark.parametrize("form", ["rowblock", "dense"])
def test_causality_later_chunks_do_not_leak(form):
    n, T, d = 5, 4, 8
    N = n * T
    q, k, v = (_rand(1, 2, N, d, seed=s) for s in (23, 24, 25))
    f = oracle.fwd if form == "rowblock" else oracle.fwd_dense
    o, lse = f(q, k, v, T, 0.4)
    for c in range(1, n):
        q2, k2, v2 = q.clone(), k.clone(), v.clone()
        for t in (q2, k2, v2):
            t[:, :, c * T:] += _rand(1, 2, N - c * T, d, seed=26 + c)
        o2, lse2 = f(q2, k2, v2, T, 0.4)
        assert torch.equal(o2[:, :, :c * T], o[:, :, :c * T])
        assert torch.equal(lse2[:, :, :c * T], lse[:, :, :c * T])
        assert not torch.allclose(o2[:, :, c * T:], o[:, :, c * T:])


def test_gradients_flow_only_backwards_in_time():
    """dO on chunks < c only: keys of chunks >= c get exactly zero dK, dV."""
    n, T, d = 4, 3, 5
    N = n * T
    q, k, v = (_rand(1, 1, N, d, seed=s) for s in (30, 31, 32))
    for c in range(1, n):
        do = _rand(1, 1, N, d, seed=33)
        do[:, :, c * T:] = 0
        dq, dk, dv = oracle.bwd(q, k, v, do, T, 0.5)
        assert torch.all(dk[:, :, c * T:] == 0) and torch.all(dv[:, :, c * T:] == 0)
        assert torch.all(dq[:, :, c * T:] == 0)
        assert dk[:, :, :c * T].abs().max() > 0


def test_gradient_sums():
    """sum_j dK_j = 0 (each dS row sums to zero) and sum_j dV_j = sum_i dO_i."""
    n, T, d = 6, 5, 8
    N = n * T
    q, k, v, do = (_rand(2, 2, N, d, seed=s) for s in (40, 41, 42, 43))
    dq, dk, dv = oracle.bwd(q, k, v, do, T, 0.35)
    assert torch.allclose(dk.sum(-2), torch.zeros(2, 2, d, dtype=F64), atol=1e-12, rtol=0)
    assert torch.allclose(dv.sum(-2), do.sum(-2), atol=1e-12, rtol=0)


def test_identical_keys_average_visible_values():
    n, T, d = 4, 3, 6
    N = n * T
    q, v = _rand(1, 1, N, d, seed=50), _rand(1, 1, N, d, seed=51)
    k = _rand(1, 1, 1, d, seed=52).expand(1, 1, N, d).contiguous()
    o, lse = oracle.fwd(q, k, v, T, 0.5)
    for i in range(N):
        end = (i // T + 1) * T
        assert torch.allclose(o[0, 0, i], v[0, 0, :end].mean(0), atol=1e-13, rtol=0)
        s = 0.5 * float(q[0, 0, i] @ k[0, 0, 0])
        assert abs(float(lse[0, 0, i]) - (s + math.log(end))) < 1e-12


def test_finite_differences():
    """Central differences of L = sum(O * G) match the analytic gradients."""
    n, T, d = 3, 2, 4
    N = n * T
    q, k, v, G = (_rand(1, 1, N, d, seed=s) for s in (60, 61, 62, 63))
    sc = 0.6
    dq, dk, dv = oracle.bwd(q, k, v, G, T, sc)
    h = 1e-6

    def loss(qq, kk, vv):
        return float((oracle.fwd(qq, kk, vv, T, sc)[0] * G).sum())

    for which, grad in ((0, dq), (1, dk), (2, dv)):
        num = torch.zeros_like(grad)
        for i in range(N):
            for x in range(d):
                args_p = [q.clone(), k.clone(), v.clone()]
                args_m = [q.clone(), k.clone(), v.clone()]
                args_p[which][0, 0, i, x] += h
                args_m[which][0, 0, i, x] -= h
                num[0, 0, i, x] = (loss(*args_p) - loss(*args_m)) / (2 * h)
        err = (num - grad).abs().max() / grad.abs().max()
        assert err < 1e-6, (which, float(err))


def test_dq_rows_matches_the_full_backward():
    """The row-by-row dQ (used for long sequences) equals the full backward's
    dQ rows, itself pinned by finite differences and autograd."""
    N, T, d = 25, 5, 6
    q, k, v, do = (_rand(1, 1, N, d, seed=s)[0, 0] for s in (120, 121, 122, 123))
    dq, _, _ = oracle.bwd(q.view(1, 1, N, d), k.view(1, 1, N, d), v.view(1, 1, N, d),
                          do.view(1, 1, N, d), T, 0.7)
    rows = [0, 3, 4, 5, 11, 19, 24]
    got = oracle.dq_rows(q, k, v, do, T, 0.7, rows)
    assert torch.allclose(got, dq[0, 0, rows], atol=1e-13, rtol=0)


def test_dkv_rows_matches_the_full_backward():
    """The row-by-row dK/dV (used for long sequences) equals the full
    backward's dK/dV rows, itself pinned by finite differences and autograd;
    small query blocks make several blocks per chunk and a ragged last one."""
    N, T, d = 28, 7, 5
    q, k, v, do = (_rand(1, 1, N, d, seed=s)[0, 0] for s in (130, 131, 132, 133))
    _, dk, dv = oracle.bwd(q.view(1, 1, N, d), k.view(1, 1, N, d), v.view(1, 1, N, d),
                           do.view(1, 1, N, d), T, 0.6)
    for rows in ([0, 6, 7, 13, 20, 27], [27, 21], [9]):
        gk, gv = oracle.dkv_rows(q, k, v, do, T, 0.6, rows, block=3)
        assert torch.allclose(gk, dk[0, 0, rows], atol=1e-13, rtol=0)
        assert torch.allclose(gv, dv[0, 0, rows], atol=1e-13, rtol=0)


# ---------------------------------------------------------------- rolling cache

def _cache_case(W, T, cap, length, head, d=8, seed=70, B=1, H=2):
    q = _rand(B, H, W * T, d, seed=seed)
    kn = _rand(B, H, W * T, d, seed=seed + 1)
    vn = _rand(B, H, W * T, d, seed=seed + 2)
    kr = _rand(B, H, cap, d, seed=seed + 3)
    vr = _rand(B, H, cap, d, seed=seed + 4)
    return q, kn, vn, kr, vr


@pytest.mark.parametrize("W,T,cap_chunks,head", [(1, 4, 5, 0), (1, 4, 5, 9), (3, 3, 4, 5),
                                                 (4, 5, 6, 29), (2, 2, 3, 1)])
def test_cache_equals_unrolled_training_form(W, T, cap_chunks, head):
    cap = cap_chunks * T
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5)
    # unrolled: cached tokens (logical order) then the in-flight chunks
    idx = torch.tensor([(head + t) % cap for t in range(cap)])
    keys = torch.cat([kr[:, :, idx], kn], dim=-2)
    vals = torch.cat([vr[:, :, idx], vn], dim=-2)
    qq = torch.cat([torch.zeros_like(kr), q], dim=-2)
    o_ref, lse_ref = oracle.fwd(qq, keys, vals, T, 0.5)
    assert torch.allclose(o, o_ref[:, :, cap:], atol=1e-13, rtol=0)
    assert torch.allclose(lse, lse_ref[:, :, cap:], atol=1e-13, rtol=0)
    # and through the library routine with its own mask
    mask = torch.zeros(W * T, cap + W * T, dtype=torch.bool)
    for j in range(W):
        mask[j * T:(j + 1) * T, :cap + (j + 1) * T] = True
    ref = F.scaled_dot_product_attention(q, keys, vals, attn_mask=mask, scale=0.5)
    assert torch.allclose(o, ref, atol=1e-12, rtol=0)


@pytest.mark.parametrize("S,W,T,cap_chunks,head", [(1, 1, 4, 5, 9), (2, 2, 4, 3, 5), (4, 2, 4, 3, 0),
                                                   (9, 3, 3, 4, 7)])
def test_sink_anchor_comes_first_and_is_always_visible(S, W, T, cap_chunks, head):
    """Sec. 3.5: the committed history is the sink anchor (never evicted, first
    position) followed by the FIFO ring; every in-flight chunk sees all of it."""
    cap = cap_chunks * T
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head)
    ks, vs = _rand(1, 2, S, 8, seed=91), _rand(1, 2, S, 8, seed=92)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks, vs)
    idx = torch.tensor([(head + t) % cap for t in range(cap)])
    keys = torch.cat([ks, kr[:, :, idx], kn], dim=-2)
    vals = torch.cat([vs, vr[:, :, idx], vn], dim=-2)
    mask = torch.zeros(W * T, S + cap + W * T, dtype=torch.bool)
    for j in range(W):
        mask[j * T:(j + 1) * T, :S + cap + (j + 1) * T] = True
    ref = F.scaled_dot_product_attention(q, keys, vals, attn_mask=mask, scale=0.5)
    assert torch.allclose(o, ref, atol=1e-12, rtol=0)
    # LSE from its definition over the visible keys
    s_all = 0.5 * q @ keys.transpose(-1, -2)
    lse_ref = torch.logsumexp(s_all.masked_fill(~mask, float("-inf")), dim=-1)
    assert torch.allclose(lse, lse_ref, atol=1e-12, rtol=0)
    # a sink of S tokens is the same as S more tokens at the ring's logical front
    ring2_k = torch.cat([ks, kr[:, :, idx]], dim=-2)
    ring2_v = torch.cat([vs, vr[:, :, idx]], dim=-2)
    o2, lse2 = oracle.cache_fwd(q, kn, vn, ring2_k, ring2_v, S + cap, 0, S + cap, T, 0.5)
    assert torch.equal(o2, o) and torch.equal(lse2, lse)


def test_sink_of_whole_chunks_is_training_form():
    """With a one-chunk sink the cache path equals the training form over
    [sink ; ring (logical) ; in-flight] (Sec. 3.2 block-causal mask)."""
    W, T, cap, head = 2, 4, 12, 5
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head)
    ks, vs = _rand(1, 2, T, 8, seed=93), _rand(1, 2, T, 8, seed=94)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks, vs)
    idx = torch.tensor([(head + t) % cap for t in range(cap)])
    keys = torch.cat([ks, kr[:, :, idx], kn], dim=-2)
    vals = torch.cat([vs, vr[:, :, idx], vn], dim=-2)
    qq = torch.cat([torch.zeros_like(ks), torch.zeros_like(kr), q], dim=-2)
    o_ref, lse_ref = oracle.fwd(qq, keys, vals, T, 0.5)
    assert torch.allclose(o, o_ref[:, :, T + cap:], atol=1e-13, rtol=0)
    assert torch.allclose(lse, lse_ref[:, :, T + cap:], atol=1e-13, rtol=0)


def test_rope_rotate_hand_values():
    """d = 4 with both pairs rotated, base 100: pair 0 turns by the frame index,
    pair 1 by frame / 10."""
    x = torch.tensor([[1.0, 0.0, 0.0, 1.0]], dtype=F64)
    y = oracle.rope_rotate(x, torch.tensor([2]), 4, 100.0)
    want = torch.tensor([[math.cos(2.0), math.sin(2.0), -math.sin(0.2), math.cos(0.2)]], dtype=F64)
    assert torch.allclose(y, want, atol=1e-15, rtol=0)
    # frame 0 and rope_dims 0 leave the rows unchanged; the last channels never move
    assert torch.equal(oracle.rope_rotate(x, torch.tensor([0]), 4, 100.0), x)
    assert torch.equal(oracle.rope_rotate(x, torch.tensor([5]), 0, 100.0), x)
    z = oracle.rope_rotate(torch.ones(1, 6, dtype=F64), torch.tensor([3]), 2, 10.0)
    assert torch.equal(z[:, 2:], torch.ones(1, 4, dtype=F64))


def test_rope_rotate_is_a_complex_phase():
    """Channel pairs as complex numbers: rotation multiplies pair i by
    exp(1j * frame * base^(-2i/rope_dims)) and keeps every pair's norm."""
    x = _rand(1, 2, 9, 12, seed=95).to(F64)
    frames = torch.tensor([0, 1, 1, 2, 3, 5, 8, 13, 21])
    y = oracle.rope_rotate(x, frames, 8, 500.0)
    zx = torch.view_as_complex(x[..., :8].reshape(1, 2, 9, 4, 2).contiguous())
    freq = 500.0 ** (-2.0 * torch.arange(4, dtype=F64) / 8)
    phase = torch.polar(torch.ones(9, 4, dtype=F64), frames.to(F64)[:, None] * freq[None, :])
    zy = torch.view_as_real(zx * phase).reshape(1, 2, 9, 8)
    assert torch.allclose(y[..., :8], zy, atol=1e-13, rtol=0)
    assert torch.equal(y[..., 8:], x[..., 8:])


def test_rope_reshift_keeps_relative_positions():
    """Scores of rotated queries and keys depend on frame differences only:
    moving every position (sink, ring, in-flight chunks) by the same offset
    changes nothing (the re-indexing of Sec. 3.5 is lossless)."""
    W, T, cap, head, P = 2, 4, 12, 5, 2
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head)
    ks, vs = _rand(1, 2, 2, 8, seed=96), _rand(1, 2, 2, 8, seed=97)

    def run(first):
        new_frames = first + cap // P + torch.arange(W * T) // P
        qr = oracle.rope_rotate(q, new_frames, 6, 50.0)
        knr = oracle.rope_rotate(kn, new_frames, 6, 50.0)
        ksr = oracle.rope_rotate(ks, torch.full((2,), first - 1), 6, 50.0)  # one frame ahead
        return oracle.cache_fwd(qr, knr, vn, kr, vr, cap, head, cap, T, 0.5, ksr, vs,
                                rope=(6, 50.0, P, first))

    o1, l1 = run(1)
    o2, l2 = run(7)
    assert torch.allclose(o1, o2, atol=1e-12, rtol=0) and torch.allclose(l1, l2, atol=1e-12, rtol=0)
    # and the rotation really is applied: other offsets between ring and queries differ
    new_frames = 1 + cap // P + torch.arange(W * T) // P
    qr = oracle.rope_rotate(q, new_frames, 6, 50.0)
    knr = oracle.rope_rotate(kn, new_frames, 6, 50.0)
    o3, _ = oracle.cache_fwd(qr, knr, vn, kr, vr, cap, head, cap, T, 0.5,
                             oracle.rope_rotate(ks, torch.zeros(2, dtype=torch.long), 6, 50.0),
                             vs, rope=(6, 50.0, P, 4))
    assert (o3 - o1).abs().max() > 1e-3


def test_rope_ring_equals_prerotated_ring():
    """Rotating the ring on read equals handing over the logically ordered,
    already rotated keys with no RoPE (the ring rewrite the fused read avoids)."""
    W, T, cap, head, P = 1, 4, 8, 3, 4
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, rope=(8, 1e4, P, 2))
    logical = oracle.ring_logical(kr.to(F64), cap, head, cap)
    rotated = oracle.rope_rotate(logical, 2 + torch.arange(cap) // P, 8, 1e4)
    o2, lse2 = oracle.cache_fwd(q, kn, vn, rotated, oracle.ring_logical(vr.to(F64), cap, head, cap),
                                cap, 0, cap, T, 0.5)
    assert torch.equal(o, o2) and torch.equal(lse, lse2)


def _reshift_case(seed=150, W=2, T=4, cap_chunks=3, head=5, S=3, d=8):
    cap = cap_chunks * T
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, head, d=d, seed=seed)
    ks, vs = _rand(1, 2, S, d, seed=seed + 7), _rand(1, 2, S, d, seed=seed + 8)
    return W, T, cap, head, q, kn, vn, kr, vr, ks, vs


def test_reshift_without_evictions_is_the_plain_sink_forward():
    W, T, cap, head, q, kn, vn, kr, vr, ks, vs = _reshift_case()
    o, lse = oracle.cache_fwd_reshift(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks, vs, 6, 50.0, 0)
    o2, lse2 = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks, vs)
    assert torch.equal(o, o2) and torch.equal(lse, lse2)


def test_reshift_only_moves_the_sink_relative_to_the_window():
    """Turning every non-sink row back by the same angle keeps their mutual
    scores; without a sink the shift therefore changes nothing, and with one
    it equals turning only the sink forward by the shift (the form the
    kernels use)."""
    W, T, cap, head, q, kn, vn, kr, vr, ks, vs = _reshift_case()
    empty = ks[:, :, :0]
    for shift in (1, 7, 1000):
        o, lse = oracle.cache_fwd_reshift(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, empty,
                                          vs[:, :, :0], 6, 50.0, shift)
        o2, lse2 = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5)
        assert torch.allclose(o, o2, atol=1e-12, rtol=0) and torch.allclose(lse, lse2, atol=1e-12, rtol=0)
        o, lse = oracle.cache_fwd_reshift(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks, vs, 6,
                                          50.0, shift)
        ks_fwd = oracle.rope_rotate(ks, torch.full((1,), shift), 6, 50.0)
        o3, lse3 = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks_fwd, vs)
        assert torch.allclose(o, o3, atol=1e-12, rtol=0) and torch.allclose(lse, lse3, atol=1e-12, rtol=0)
        # the direction matters: turning the sink back instead gives other scores
        ks_bad = oracle.rope_rotate(ks, torch.full((1,), -shift), 6, 50.0)
        o4, _ = oracle.cache_fwd(q, kn, vn, kr, vr, cap, head, cap, T, 0.5, ks_bad, vs)
        assert (o4 - o).abs().max() > 1e-6


def test_reshift_equals_window_positions():
    """Keys rotated at stream positions and re-shifted by the evicted frames
    give the attention of the same keys rotated at their window positions
    (ring token t at frame first + t // P, the window counted from the
    oldest retained chunk; the sink at frame 0)."""
    W, T, cap, head, q0, kn0, vn, kr0, vr, ks0, vs = _reshift_case(seed=170)
    P, first, shift, dims, base = 2, 1, 9, 6, 50.0
    logical = torch.arange(cap)
    ring_window = first + logical // P                    # logical order
    win_frames = first + cap // P + torch.arange(W * T) // P
    # stream-rotated inputs (what the caller holds): window frame + shift
    phys = torch.tensor([(head + t) % cap for t in range(cap)])
    inv = torch.empty_like(phys)
    inv[phys] = logical                                   # physical row -> logical index
    kr_stream = oracle.rope_rotate(kr0, ring_window[inv] + shift, dims, base)
    q_s = oracle.rope_rotate(q0, win_frames + shift, dims, base)
    kn_s = oracle.rope_rotate(kn0, win_frames + shift, dims, base)
    ks = oracle.rope_rotate(ks0, torch.zeros(ks0.shape[-2], dtype=torch.long), dims, base)
    o, lse = oracle.cache_fwd_reshift(q_s, kn_s, vn, kr_stream, vr, cap, head, cap, T, 0.5, ks, vs,
                                      dims, base, shift)
    # the window-position form: queries and in-flight keys at window frames,
    # the ring turned on read from its unrotated keys
    q_w = oracle.rope_rotate(q0, win_frames, dims, base)
    kn_w = oracle.rope_rotate(kn0, win_frames, dims, base)
    o2, lse2 = oracle.cache_fwd(q_w, kn_w, vn, kr0, vr, cap, head, cap, T, 0.5, ks, vs,
                                rope=(dims, base, P, first))
    assert torch.allclose(o, o2, atol=1e-12, rtol=0) and torch.allclose(lse, lse2, atol=1e-12, rtol=0)


def test_ring_rotation_is_invisible():
    W, T, cap = 2, 3, 12
    q, kn, vn, kr, vr = _cache_case(W, T, cap, cap, 4)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, cap, 4, cap, T, 0.5)
    for r in (1, 5, 11):
        kr2 = torch.roll(kr, shifts=r, dims=-2)
        vr2 = torch.roll(vr, shifts=r, dims=-2)
        o2, lse2 = oracle.cache_fwd(q, kn, vn, kr2, vr2, cap, (4 + r) % cap, cap, T, 0.5)
        assert torch.equal(o2, o) and torch.equal(lse2, lse)


def test_partially_filled_ring_ignores_unused_rows():
    W, T, cap, length, head = 2, 4, 20, 8, 15
    q, kn, vn, kr, vr = _cache_case(W, T, cap, length, head)
    used = [(head + t) % cap for t in range(length)]
    kr_nan, vr_nan = torch.full_like(kr, float("nan")), torch.full_like(vr, float("nan"))
    kr_nan[:, :, used], vr_nan[:, :, used] = kr[:, :, used], vr[:, :, used]
    o, lse = oracle.cache_fwd(q, kn, vn, kr_nan, vr_nan, cap, head, length, T, 0.5)
    assert torch.isfinite(o).all()
    o_ref, lse_ref = oracle.cache_fwd(q, kn, vn, kr[:, :, used], vr[:, :, used],
                                      length, 0, length, T, 0.5)
    assert torch.equal(o, o_ref) and torch.equal(lse, lse_ref)


def test_empty_ring_is_training_form():
    W, T = 3, 4
    q, kn, vn, kr, vr = _cache_case(W, T, 8, 0, 0)
    o, lse = oracle.cache_fwd(q, kn, vn, kr, vr, 8, 0, 0, T, 0.5)
    o_ref, lse_ref = oracle.fwd(q, kn, vn, T, 0.5)
    assert torch.allclose(o, o_ref, atol=1e-14, rtol=0)
    assert torch.allclose(lse, lse_ref, atol=1e-14, rtol=0)


def test_commit_is_fifo():
    """Committing a chunk into a full ring evicts exactly the oldest chunk and
    appends the new one at the logical end; committed rows never change."""
    T, cap = 3, 9
    ring = torch.arange(cap, dtype=F64).view(1, 1, cap, 1)
    head, length = 0, 0
    history = []
    for step in range(7):
        chunk = (100.0 * (step + 1) + torch.arange(T, dtype=F64)).view(1, 1, T, 1)
        slot, head, length = oracle.ring_advance(cap, head, length, T)
        ring, _ = oracle.cache_commit(ring, ring, cap, slot, chunk, chunk)
        history.append(chunk)
        logical = oracle.ring_logical(ring, cap, head, length)
        expect = torch.cat(history[-(cap // T):], dim=-2)
        assert torch.equal(logical, expect), step
    # wrap handling of a commit that straddles the end of the buffer
    ring = torch.zeros(1, 1, 5, 1, dtype=F64)
    src = torch.tensor([1.0, 2.0, 3.0], dtype=F64).view(1, 1, 3, 1)
    out, _ = oracle.cache_commit(ring, ring, 5, 3, src, src)
    assert out.flatten().tolist() == [3.0, 0.0, 0.0, 1.0, 2.0]


def test_product_ring_bookkeeping_matches_oracle():
    """The package's host-side FIFO plan agrees with the oracle's reading of
    the rolling cache (Sec. 3.5) over fills, wraps and evictions."""
    from paper_2608_01127_gb300 import RingState
    for cap, head, length, rows in ((9, 0, 0, 3), (7040, 4400, 7040, 880), (10, 7, 4, 3),
                                    (10, 9, 10, 10), (5, 2, 1, 5)):
        ring = RingState(cap, head, length)
        h, n = head, length
        for _ in range(6):
            slot, h, n = oracle.ring_advance(cap, h, n, rows)
            assert ring.commit(rows) == slot
            assert (ring.head, ring.length) == (h, n)


def test_qkv_split_moves_every_element_to_its_head():
    """Without rotation the split is a pure relabelling: written out element by
    element, Q[b,h,t,c] = qkv[b,t,0,h,c], K takes index 1 and V index 2."""
    B, N, H, d = 2, 3, 2, 8
    qkv = torch.arange(B * N * 3 * H * d, dtype=F64).reshape(B, N, 3, H, d)
    q, k, v = oracle.qkv_split_rope(qkv)
    for b in range(B):
        for t in range(N):
            for h in range(H):
                for c in range(d):
                    flat = (((b * N + t) * 3) * H + h) * d + c
                    assert q[b, h, t, c] == flat
                    assert k[b, h, t, c] == flat + H * d
                    assert v[b, h, t, c] == flat + 2 * H * d


def test_qkv_split_rope_hand_values():
    """Token 5 with two tokens per frame, first frame 1, sits at frame 3: its
    query and key pair i turn by 3 * base^(-2i/rope_dims); V never turns, and
    channels past rope_dims never move."""
    B, N, H, d = 1, 6, 1, 8
    qkv = torch.zeros(B, N, 3, H, d, dtype=F64)
    qkv[0, 5, 0, 0, :] = torch.tensor([1.0, 0.0, 0.0, 2.0, 1.0, 1.0, 5.0, 6.0])
    qkv[0, 5, 1, 0, :] = torch.tensor([0.0, 1.0, 3.0, 0.0, 2.0, 0.0, 7.0, 8.0])
    qkv[0, 5, 2, 0, :] = torch.tensor([1.0, 2.0, 3.0, 4.0, 5.0, 6.0, 7.0, 8.0])
    q, k, v = oracle.qkv_split_rope(qkv, rope_dims=6, base=64.0, tokens_per_frame=2,
                                    first_frame=1)
    a0, a1, a2 = 3.0, 3.0 * 64.0 ** (-2.0 / 6), 3.0 * 64.0 ** (-4.0 / 6)  # 3, 0.75, 0.1875
    c, s = math.cos, math.sin
    want_q = [c(a0), s(a0), -2 * s(a1), 2 * c(a1), c(a2) - s(a2), s(a2) + c(a2), 5.0, 6.0]
    want_k = [-s(a0), c(a0), 3 * c(a1), 3 * s(a1), 2 * c(a2), 2 * s(a2), 7.0, 8.0]
    assert torch.allclose(q[0, 0, 5], torch.tensor(want_q, dtype=F64), atol=1e-15, rtol=0)
    assert torch.allclose(k[0, 0, 5], torch.tensor(want_k, dtype=F64), atol=1e-15, rtol=0)
    assert torch.equal(v[0, 0, 5], qkv[0, 5, 2, 0])
    assert torch.equal(q[0, 0, :5], torch.zeros(5, d, dtype=F64))


def test_qkv_split_rope_scores_depend_on_frame_differences():
    """With every channel rotated, Q K^T is unchanged when all positions move
    by the same number of frames, and changes when the spacing changes."""
    B, N, H, d = 1, 12, 2, 8
    qkv = _rand(B, N, 3 * H, d, seed=98).to(F64).reshape(B, N, 3, H, d)
    q1, k1, _ = oracle.qkv_split_rope(qkv, d, 100.0, 3, 0)
    q2, k2, _ = oracle.qkv_split_rope(qkv, d, 100.0, 3, 11)
    q3, k3, _ = oracle.qkv_split_rope(qkv, d, 100.0, 2, 0)
    s1, s2, s3 = q1 @ k1.transpose(-1, -2), q2 @ k2.transpose(-1, -2), q3 @ k3.transpose(-1, -2)
    assert torch.allclose(s1, s2, atol=1e-12, rtol=0)
    assert (s3 - s1).abs().max() > 1e-3
