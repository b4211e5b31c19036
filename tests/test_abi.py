"""C-ABI checks that need no GPU: the library builds for sm_103a, loads,
exports every entry point the header declares, and rejects bad arguments
with the documented status codes before touching the device."""
import ctypes
import os
import re
import subprocess

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mw_bca.h")

OK, INVALID, UNSUPPORTED, CUDA, TIMEOUT, WORKSPACE = range(6)
FAKE = ctypes.c_void_p(0x10000)        # aligned, never dereferenced on these paths
MISALIGNED = ctypes.c_void_p(0x10008)


@pytest.fixture(scope="module")
def mw():
    from paper_2608_01127_gb300 import _build
    _build.build()
    import paper_2608_01127_gb300 as pkg
    pkg.library()
    return pkg


def _declared():
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mw_[a-z_]+)\s*\(", text)))


def test_header_declares_the_python_exports(mw):
    assert _declared() == sorted(mw.EXPORTED_SYMBOLS)


def test_library_exports_every_declared_symbol(mw):
    out = subprocess.run(["nm", "-D", "--defined-only", mw.lib_path], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r" T (mw_\w+)$", out, flags=re.M))
    for name in _declared():
        assert name in exported, name
        assert hasattr(mw.library(), name)


def test_status_strings(mw):
    lib = mw.library()
    for code, name in mw.STATUS.items():
        assert lib.mw_status_string(code).decode() == name


def test_fwd_rejects_bad_arguments(mw):
    lib = mw.library()
    args = dict(q=FAKE, k=FAKE, v=FAKE, o=FAKE, lse=None, B=1, H=1, n=2, T=64, d=64, s=0.125)

    def call(**kw):
        a = {**args, **kw}
        return lib.mw_bca_fwd(a["q"], a["k"], a["v"], a["o"], a["lse"], a["B"], a["H"], a["n"],
                              a["T"], a["d"], a["s"], None)

    assert call(q=None) == INVALID
    assert call(o=None) == INVALID
    assert call(k=MISALIGNED) == INVALID
    assert call(d=100) == UNSUPPORTED   # not a multiple of 8
    assert call(d=136) == UNSUPPORTED
    assert call(d=56) == UNSUPPORTED
    assert call(d=0) == UNSUPPORTED
    assert call(B=0) == INVALID
    assert call(T=0) == INVALID
    assert call(n=0) == INVALID
    assert call(n=1 << 15, T=1 << 10) == INVALID   # 2^25 tokens
    assert call(B=1 << 10, H=1 << 10, n=1, T=1 << 12) == INVALID   # 2^32 tokens over all heads
    assert call(s=0.0) == INVALID
    assert call(s=-1.0) == INVALID
    assert "scale" in lib.mw_last_error().decode()


def test_bwd_rejects_bad_arguments_and_workspace(mw):
    lib = mw.library()
    B, H, n, T, d = 1, 2, 3, 50, 64
    need = lib.mw_bca_bwd_workspace_size(B, H, n, T, d)
    # dQ accumulator (fp32, rows padded to 128) + two fp32 row vectors, 256-byte
    # aligned, + the d = 64 bias rows of the MMA-folded LSE and D terms (32 bytes a row)
    assert need == 2 * 256 * 64 * 4 + 2 * 256 * 4 + 2 * 256 * 4 + 2 * 256 * 32
    assert lib.mw_bca_bwd_workspace_size(B, H, n, T, 100) == 0
    # a padded head dim (72) keeps a 128-wide fp32 accumulator
    assert lib.mw_bca_bwd_workspace_size(B, H, n, T, 72) == 2 * 256 * 128 * 4 + 2 * 256 * 4 + 2 * 256 * 4

    def call(ws=FAKE, ws_bytes=need, lse=FAKE, d=d):
        return lib.mw_bca_bwd(FAKE, FAKE, FAKE, FAKE, lse, FAKE, FAKE, FAKE, FAKE, ws, ws_bytes,
                              B, H, n, T, d, 0.125, None)

    assert call(ws=None) == WORKSPACE
    assert call(ws_bytes=need - 1) == WORKSPACE
    assert call(ws=ctypes.c_void_p(0x10010)) == INVALID   # not 256-byte aligned
    assert call(lse=None) == INVALID
    assert call(d=32) == UNSUPPORTED


def test_cache_rejects_bad_ring_state(mw):
    lib = mw.library()

    def call(cap=1024, head=0, length=1024, kc=FAKE, B=1, H=2, W=1, T=64, d=128):
        return lib.mw_bca_cache_fwd(FAKE, FAKE, FAKE, kc, FAKE, cap, head, length, FAKE, None,
                                    None, 0, B, H, W, T, d, 0.1, None)

    assert call(head=1024) == INVALID
    assert call(head=-1) == INVALID
    assert call(length=1025) == INVALID
    assert call(length=-1) == INVALID
    assert call(cap=0, head=0, length=0) == INVALID
    assert call(kc=None) == INVALID
    assert call(d=84) == UNSUPPORTED
    assert call(T=0) == INVALID


def test_sink_entry_rejects_bad_sink(mw):
    lib = mw.library()

    def call(sink_len=440, ks=FAKE, vs=FAKE, head=0):
        return lib.mw_bca_cache_fwd_sink(FAKE, FAKE, FAKE, ks, vs, sink_len, FAKE, FAKE, 1024,
                                         head, 1024, FAKE, None, None, 0, 1, 2, 1, 64, 128, 0.1,
                                         None)

    assert call(sink_len=-1) == INVALID
    assert call(sink_len=(1 << 24) + 1) == INVALID
    assert call(ks=None) == INVALID
    assert call(vs=None) == INVALID
    assert call(head=1024) == INVALID  # the ring checks still apply


def test_rope_entry_rejects_bad_rope(mw):
    lib = mw.library()

    def call(dims=32, base=1e4, shift=3):
        return lib.mw_bca_cache_fwd_rope(FAKE, FAKE, FAKE, None, None, 0, FAKE, FAKE, 1024, 0,
                                         1024, dims, base, shift, FAKE, None, None, 0,
                                         1, 2, 1, 64, 128, 0.1, None)

    assert call(dims=-2) == INVALID
    assert call(dims=31) == INVALID       # odd
    assert call(dims=130) == INVALID      # more than d
    assert call(base=1.0) == INVALID
    assert call(base=float("nan")) == INVALID
    assert call(shift=-1) == INVALID
    assert call(shift=(1 << 24) + 1) == INVALID  # angles past 2^24 frames


def test_step_rejects_bad_commit(mw):
    lib = mw.library()

    def call(slot=100, rows=880, kc=FAKE):
        # one 880-token chunk against a full 7040-token ring
        return lib.mw_bca_cache_step(FAKE, FAKE, FAKE, kc, FAKE, 7040, 0, 7040, slot, rows, FAKE,
                                     None, None, 0, 1, 2, 1, 880, 64, 0.125, None)

    assert call(rows=-1) == INVALID
    assert call(rows=881) == INVALID        # more rows than the in-flight chunks hold
    assert call(slot=7040) == INVALID
    assert call(slot=-1) == INVALID
    assert call(kc=MISALIGNED) == INVALID
    assert call(kc=None) == INVALID


def test_commit_rejects_bad_slots(mw):
    lib = mw.library()

    def call(cap=100, slot=0, rows=10, src=FAKE):
        return lib.mw_bca_cache_commit(FAKE, FAKE, cap, slot, src, FAKE, rows, 1, 1, 64, None)

    assert call(slot=100) == INVALID
    assert call(slot=-3) == INVALID
    assert call(rows=0) == INVALID
    assert call(rows=101) == INVALID
    assert call(src=None) == INVALID
    assert call(src=MISALIGNED) == INVALID


def test_qkv_split_rejects_bad_arguments(mw):
    lib = mw.library()

    def call(qkv=FAKE, q=FAKE, B=2, N=100, H=3, d=64, dims=32, base=1e4, per_frame=7, first=0):
        return lib.mw_qkv_rope_split(qkv, q, FAKE, FAKE, B, N, H, d, dims, base, per_frame,
                                     first, None)

    assert call(qkv=None) == INVALID
    assert call(qkv=MISALIGNED) == INVALID
    assert call(q=MISALIGNED) == INVALID
    assert call(N=0) == INVALID
    assert call(B=0) == INVALID
    assert call(N=1 << 24, B=200) == INVALID        # more than 2^31 tokens
    assert call(d=100) == UNSUPPORTED
    assert call(d=136) == UNSUPPORTED
    assert call(dims=33) == INVALID                 # odd
    assert call(dims=66) == INVALID                 # more than d
    assert call(base=0.5) == INVALID
    assert call(per_frame=0) == INVALID
    assert call(first=-1) == INVALID
    assert call(first=(1 << 24) - 10, per_frame=1) == INVALID  # frame positions past 2^24


def test_options(mw):
    lib = mw.library()
    assert lib.mw_set_option(b"no_such_option", 1) == INVALID
    assert lib.mw_set_option(b"cache_splits", -1) == INVALID
    assert lib.mw_set_option(b"cache_splits", 99) == INVALID
    assert lib.mw_set_option(b"wait_budget_ms", 0) == INVALID
    assert lib.mw_set_option(b"cache_splits", 0) == OK
    assert lib.mw_set_option(b"pdl", 0) == OK
    assert lib.mw_set_option(b"pdl", 1) == OK


def test_workspace_follows_split_override(mw):
    lib = mw.library()
    try:
        assert lib.mw_set_option(b"cache_splits", 3) == OK
        size = lib.mw_bca_cache_workspace_size(1, 16, 1, 880, 128, 7040)
        assert size == 3 * 16 * 880 * 128 * 4 + ((3 * 16 * 880 * 4 + 255) // 256) * 256
        assert lib.mw_set_option(b"cache_splits", 1) == OK
        assert lib.mw_bca_cache_workspace_size(1, 16, 1, 880, 128, 7040) == 0
    finally:
        lib.mw_set_option(b"cache_splits", 0)


def _makespan(lengths, sms):
    """List scheduling: each CTA, in order, starts on the SM that frees first."""
    import heapq
    free = [0] * sms
    end = 0
    for w in lengths:
        t = heapq.heappop(free) + w
        heapq.heappush(free, t)
        end = max(end, t)
    return end


def _backward_plan(B, H, n, T, d, sms):
    """The backward's CTA-order rule, restated: a key tile's length is the
    query tiles that see it (+3); head groups hold at least twice the longest
    tile's steps on every SM and at most 48 MB of Q, dO and fp32 dQ; they win
    over head by head when the modelled launch ends >= 1% earlier."""
    BH, N = B * H, n * T
    N_pad = -(-N // 128) * 128
    if d > 80 and d != 64:
        return BH
    D = 64 if d == 64 else 128
    kt_len = [N_pad // 128 - (kt * 128 // T * T) // 128 + 3 for kt in range(N_pad // 128)]
    cap = (48 << 20) // (N_pad * (4 * d + 4 * D + 32))
    per_group = max(1, min(BH, cap, -(-2 * max(kt_len) * sms // sum(kt_len))))
    cand = -(-BH // per_group)

    def order(groups):
        base, rem = divmod(BH, groups)
        return [w for g in range(groups) for w in kt_len for _ in range(base + (g < rem))]

    if cand < BH and BH * len(kt_len) <= 1 << 18 and \
            100 * _makespan(order(cand), sms) <= 99 * _makespan(order(BH), sms):
        return cand
    return BH


@pytest.mark.parametrize("B,H,n,T,d,expect", [
    (2, 12, 16, 880, 64, 4),     # the d=64 training workload: 4 groups of 6 heads
    (1, 16, 16, 880, 72, 4),     # 80-wide MMAs, 16 heads: 4 groups of 4
    (1, 11, 8, 2048, 64, 3),     # 4 + 4 + 3 heads
    (1, 16, 21, 880, 128, 16),   # head dims over 80: head by head
    (1, 12, 32, 600, 96, 12),
    (1, 1, 4, 64, 64, 1),
    (8, 16, 2, 256, 64, None),   # short sequences, many heads: whatever the model says
    (64, 32, 16, 880, 64, 2048),  # 2^19 CTAs: past the model's limit, head by head
])
def test_backward_head_groups_follow_the_list_scheduling_rule(mw, B, H, n, T, d, expect):
    got = mw.mw_bca_bwd_head_groups(B, H, n, T, d, sm_count=152)
    assert got == _backward_plan(B, H, n, T, d, 152)
    if expect is not None:
        assert got == expect
    # the modelled grouped launch never ends later than head by head
    assert 1 <= got <= B * H


def test_backward_head_groups_override_and_errors(mw):
    lib = mw.library()
    try:
        assert lib.mw_set_option(b"bwd_group_heads", 5) == OK
        assert mw.mw_bca_bwd_head_groups(2, 12, 16, 880, 64, sm_count=152) == 5   # ceil(24 / 5)
        assert mw.mw_bca_bwd_head_groups(1, 16, 21, 880, 128, sm_count=152) == 16  # d > 80: head by head
    finally:
        lib.mw_set_option(b"bwd_group_heads", 0)
    assert lib.mw_bca_bwd_head_groups(0, 1, 1, 1, 64, 152) == -1
    assert lib.mw_bca_bwd_head_groups(1, 1, 0, 1, 64, 152) == -1
    assert lib.mw_bca_bwd_head_groups(1, 1, 1, 1, 65, 152) == -1


def test_python_binding_has_no_cpu_path(mw):
    q = torch.zeros(1, 1, 64, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        mw.mw_bca_fwd(q, q, q, 64)


def _bf(*shape):
    return torch.zeros(*shape, dtype=torch.bfloat16)


def test_python_binding_checks_every_buffer_before_the_device(mw):
    """The library cannot see buffer sizes, so the binding checks the shape,
    dtype and layout of every argument, caller-supplied outputs included, and
    the chunking, before anything is launched.  The device comes last: CPU
    tensors that pass every other check still get no CPU path."""
    q = _bf(1, 2, 128, 64)
    lse = torch.zeros(1, 2, 128)
    ring = _bf(1, 2, 512, 64)
    qkv = _bf(1, 128, 3, 2, 64)
    strided = _bf(1, 2, 64, 128).transpose(2, 3)   # [1, 2, 128, 64], not contiguous
    cases = [
        (lambda: mw.mw_bca_fwd(q, q, q, 0), "T_chunk must be >= 1"),
        (lambda: mw.mw_bca_fwd(q, q, q, 48), "not a multiple of T_chunk"),
        (lambda: mw.mw_bca_fwd(q, q, q, 64, out=(_bf(1, 2, 64, 64), None)), "o must be"),
        (lambda: mw.mw_bca_fwd(q, q, q, 64, out=(strided, None)), "o must be"),
        (lambda: mw.mw_bca_fwd(q, q, q, 64, out=(_bf(1, 2, 128, 64), lse.double())),
         "lse must be"),
        (lambda: mw.mw_bca_fwd(q, q, q, 64, out=(_bf(1, 2, 128, 64), lse[:, :, :64])),
         "lse must be"),
        (lambda: mw.mw_bca_bwd(q, q, q, q, lse.double(), q, 64), "lse must be"),
        (lambda: mw.mw_bca_bwd(q, q, q, q, lse, q, -64), "T_chunk must be >= 1"),
        (lambda: mw.mw_bca_bwd(q, q, q, q, lse, q, 64,
                               out=(_bf(1, 2, 128, 64), _bf(1, 2, 128, 64), _bf(1, 2, 128, 32))),
         "dv must be"),
        (lambda: mw.mw_bca_bwd(q, q, q, q, lse, q, 64,
                               out=(strided, _bf(1, 2, 128, 64), _bf(1, 2, 128, 64))),
         "dq must be"),
        (lambda: mw.mw_bca_cache_fwd(q, q, q, ring, ring, 0, 256, 64, out=_bf(1, 2, 64, 64)),
         "out must be"),
        (lambda: mw.mw_bca_cache_fwd(q, q, q, ring, ring, 0, 256, 0), "T_chunk must be >= 1"),
        (lambda: mw.mw_bca_cache_step(q, q, q, ring, ring, 0, 256, 256, 64, 64,
                                      out=torch.zeros(1, 2, 128, 64)), "out must be"),
        (lambda: mw.mw_bca_cache_commit(ring, _bf(1, 2, 256, 64), 0, q, q), "same shape"),
        (lambda: mw.mw_qkv_rope_split(qkv, out=(q, q)), "out must be"),
        (lambda: mw.mw_qkv_rope_split(qkv, out=(q, q, _bf(2, 2, 128, 64))), "v must be"),
        # everything right but the device
        (lambda: mw.mw_bca_fwd(q, q, q, 64), "CUDA tensors"),
        (lambda: mw.mw_bca_bwd(q, q, q, q, lse, q, 64), "CUDA tensors"),
        (lambda: mw.mw_bca_cache_fwd(q, q, q, ring, ring, 0, 256, 64), "CUDA tensors"),
        (lambda: mw.mw_bca_cache_commit(ring, ring, 0, q, q), "CUDA tensors"),
        (lambda: mw.mw_qkv_rope_split(qkv), "CUDA tensors"),
    ]
    for fn, msg in cases:
        with pytest.raises(ValueError, match=msg):
            fn()
    with pytest.raises(TypeError):
        mw.mw_bca_fwd(q, q.float(), q, 64)
    with pytest.raises(TypeError):
        mw.mw_bca_cache_fwd_sink(q, q, q, _bf(1, 2, 64, 64), None, ring, ring, 0, 256, 64)


def test_alias_check(mw):
    """Outputs may share no byte with an input or with another output."""
    from paper_2608_01127_gb300 import _no_alias
    buf = torch.zeros(4, 100, dtype=torch.bfloat16)
    a, b, c = buf[0], buf[1], buf[2]
    _no_alias((("o", a), ("lse", b)), (("q", c), ("k", c), ("none", None)))  # inputs may share
    with pytest.raises(ValueError, match="output o overlaps input q"):
        _no_alias((("o", a),), (("q", buf[0, 50:]),))
    with pytest.raises(ValueError, match="output dq overlaps output dk"):
        _no_alias((("dq", buf[1:3].reshape(-1)), ("dk", buf[2])), (("q", a),))
    # adjacent but disjoint byte ranges are fine
    _no_alias((("o", buf[0, :50]),), (("q", buf[0, 50:]),))
    _no_alias((("o", buf[0, :0]),), (("q", buf[0]),))                      # empty output


def test_workspace_is_counted_in_bytes(mw):
    from paper_2608_01127_gb300 import _workspace
    cpu = torch.device("cpu")
    assert _workspace(torch.zeros(4), 0, cpu) is None                      # none needed
    ws = torch.zeros(4, dtype=torch.float32)                               # 16 bytes
    assert _workspace(ws, 16, cpu) is ws
    grown = _workspace(ws, 17, cpu)
    assert grown is not ws and grown.dtype == torch.uint8 and grown.numel() == 17
    assert _workspace(None, 8, cpu).numel() == 8
    with pytest.raises(ValueError, match="contiguous"):
        _workspace(torch.zeros(8, 2)[:, 0], 4, cpu)
