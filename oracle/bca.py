"""fp64 CPU oracle for block-causal attention (test infrastructure only).

This module is the checker, not the product: only ``tests/``, the package's
``smoke()`` and the benchmark's CPU-baseline / reference arm may import it.
It shares no code with the CUDA path.

What it computes (Sec. 3.2, block-causal self-attention): the token sequence
is cut into temporally ordered chunks of ``T`` tokens; a query attends to every
key of its own chunk (bidirectionally) and of all earlier chunks (strictly
causal across chunks).  With chunk(i) = floor(i / T):

    visible(i, j)  <=>  chunk(j) <= chunk(i)
    s_ij   = scale * <q_i, k_j>                       (visible pairs only)
    LSE_i  = ln sum_{j visible} exp(s_ij)
    P_ij   = exp(s_ij - LSE_i)   (0 where not visible)
    O_i    = sum_j P_ij v_j

The paper does not write the attention formula itself; the above is standard
scaled dot-product attention restricted by the chunk mask.  The backward
(training is bf16 mixed precision, Sec. 4.1) is the analytic gradient:

    dV_j  = sum_i P_ij dO_i
    dP_ij = <dO_i, v_j>
    D_i   = <dO_i, O_i>
    dS_ij = P_ij (dP_ij - D_i)
    dQ_i  = scale * sum_j dS_ij k_j
    dK_j  = scale * sum_i dS_ij q_i

Streaming (Sec. 3.5): in-flight chunks attend to the committed history (the
rolling KV cache, a FIFO of finished chunks) and to preceding in-flight chunks
under the same chunk-causal rule.  Committed K/V are written once and never
change.

All arithmetic is fp64 (inputs are the bf16 tensors the GPU sees, widened).
Three forms of the forward are kept and cross-checked: scalar loops (tiny
shapes), a dense N x N masked matrix, and a row-block form that builds, per
query chunk c, the [T, (c+1)T] block of visible scores (which is the mask).
"""
from __future__ import annotations

import math
from typing import List, Sequence, Tuple

import torch

F64 = torch.float64


def chunk_of(i: int, T: int) -> int:
    """Chunk index of token i for chunks of T tokens."""
    return i // T


def block_causal_mask(N: int, T: int) -> torch.Tensor:
    """Boolean [N, N]: True where query i may attend key j (Sec. 3.2)."""
    idx = torch.arange(N)
    return (idx.view(1, N) // T) <= (idx.view(N, 1) // T)


# --------------------------------------------------------------------------
# form (i): scalar loops, one head, python floats; tiny shapes only
# --------------------------------------------------------------------------

def fwd_loops(q: Sequence[Sequence[float]], k: Sequence[Sequence[float]],
              v: Sequence[Sequence[float]], T: int, scale: float
              ) -> Tuple[List[List[float]], List[float]]:
    """Forward of one head by explicit loops over i, j and the feature index."""
    N = len(q)
    d = len(q[0])
    dv = len(v[0])
    out, lse = [], []
    for i in range(N):
        scores = []
        for j in range(N):
            if chunk_of(j, T) <= chunk_of(i, T):
                dot = 0.0
                for x in range(d):
                    dot += q[i][x] * k[j][x]
                scores.append((j, scale * dot))
        assert scores, "a query always sees its own chunk"
        top = max(s for _, s in scores)
        total = 0.0
        for _, s in scores:
            total += math.exp(s - top)
        l_i = top + math.log(total)
        row = [0.0] * dv
        for j, s in scores:
            p = math.exp(s - l_i)
            for x in range(dv):
                row[x] += p * v[j][x]
        out.append(row)
        lse.append(l_i)
    return out, lse


# --------------------------------------------------------------------------
# form (ii): dense masked matrices, [..., N, d]
# --------------------------------------------------------------------------

def probs_dense(q: torch.Tensor, k: torch.Tensor, T: int, scale: float) -> torch.Tensor:
    """P [..., N, N] with zeros at masked positions (small N only)."""
    q = q.to(F64)
    k = k.to(F64)
    N = q.shape[-2]
    s = scale * torch.matmul(q, k.transpose(-1, -2))
    s = s.masked_fill(~block_causal_mask(N, T), float("-inf"))
    lse = _row_lse(s)
    return torch.exp(s - lse.unsqueeze(-1))


def fwd_dense(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, T: int,
              scale: float) -> Tuple[torch.Tensor, torch.Tensor]:
    """(O, LSE) through the explicit N x N mask."""
    q, k, v = q.to(F64), k.to(F64), v.to(F64)
    N = q.shape[-2]
    s = scale * torch.matmul(q, k.transpose(-1, -2))
    s = s.masked_fill(~block_causal_mask(N, T), float("-inf"))
    lse = _row_lse(s)
    p = torch.exp(s - lse.unsqueeze(-1))
    return torch.matmul(p, v), lse


def bwd_dense(q, k, v, do, T: int, scale: float):
    """(dQ, dK, dV) through the explicit N x N mask."""
    q, k, v, do = (t.to(F64) for t in (q, k, v, do))
    p = probs_dense(q, k, T, scale)
    o = torch.matmul(p, v)
    dv = torch.matmul(p.transpose(-1, -2), do)
    dp = torch.matmul(do, v.transpose(-1, -2))
    D = (do * o).sum(-1, keepdim=True)
    ds = p * (dp - D)
    dq = scale * torch.matmul(ds, k)
    dk = scale * torch.matmul(ds.transpose(-1, -2), q)
    return dq, dk, dv


def _row_lse(s: torch.Tensor) -> torch.Tensor:
    """ln sum_j exp(s_j) over the last axis; the row maximum is factored out
    (ln sum exp(s) = m + ln sum exp(s - m)) so that exp never overflows."""
    m = s.max(dim=-1, keepdim=True).values
    return (m + torch.log(torch.exp(s - m).sum(dim=-1, keepdim=True))).squeeze(-1)


# --------------------------------------------------------------------------
# form (iii): row blocks per query chunk, [B, H, N, d]
# --------------------------------------------------------------------------

def fwd(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, T: int,
        scale: float) -> Tuple[torch.Tensor, torch.Tensor]:
    """(O [B,H,N,dv], LSE [B,H,N]) for Q, K, V [B,H,N,d]; N a multiple of T.

    Query chunk c sees keys [0, (c+1) T): its score block is that slice, so the
    mask is the slicing itself.
    """
    q, k, v = q.to(F64), k.to(F64), v.to(F64)
    B, H, N, _ = q.shape
    assert N % T == 0, "sequence length must be a whole number of chunks"
    n = N // T
    o = torch.empty(B, H, N, v.shape[-1], dtype=F64)
    lse = torch.empty(B, H, N, dtype=F64)
    for b in range(B):
        for h in range(H):
            for c in range(n):
                rows = slice(c * T, (c + 1) * T)
                keys = slice(0, (c + 1) * T)
                s = scale * (q[b, h, rows] @ k[b, h, keys].T)
                l_c = _row_lse(s)
                p = torch.exp(s - l_c.unsqueeze(-1))
                o[b, h, rows] = p @ v[b, h, keys]
                lse[b, h, rows] = l_c
    return o, lse


def bwd(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, do: torch.Tensor,
        T: int, scale: float) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """(dQ, dK, dV) of sum(O * dO) for Q, K, V, dO [B,H,N,d]; P is recomputed."""
    q, k, v, do = (t.to(F64) for t in (q, k, v, do))
    B, H, N, _ = q.shape
    assert N % T == 0
    n = N // T
    dq = torch.zeros_like(q)
    dk = torch.zeros_like(k)
    dv = torch.zeros_like(v)
    for b in range(B):
        for h in range(H):
            for c in range(n):
                rows = slice(c * T, (c + 1) * T)
                keys = slice(0, (c + 1) * T)
                qc, kc, vc, doc = q[b, h, rows], k[b, h, keys], v[b, h, keys], do[b, h, rows]
                s = scale * (qc @ kc.T)
                p = torch.exp(s - _row_lse(s).unsqueeze(-1))
                oc = p @ vc
                dv[b, h, keys] += p.T @ doc
                dp = doc @ vc.T
                D = (doc * oc).sum(-1, keepdim=True)
                ds = p * (dp - D)
                dq[b, h, rows] = scale * (ds @ kc)
                dk[b, h, keys] += scale * (ds.T @ qc)
    return dq, dk, dv


def fwd_rows(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, T: int,
             scale: float, rows: Sequence[int]) -> Tuple[torch.Tensor, torch.Tensor]:
    """(O, LSE) of selected query rows of one head (Q,K,V [N,d]), row by row."""
    q, k, v = q.to(F64), k.to(F64), v.to(F64)
    outs, lses = [], []
    for i in rows:
        end = (chunk_of(i, T) + 1) * T
        s = scale * (k[:end] @ q[i])
        l_i = _row_lse(s.unsqueeze(0))[0]
        outs.append(torch.exp(s - l_i) @ v[:end])
        lses.append(l_i)
    return torch.stack(outs), torch.stack(lses)


def dq_rows(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, do: torch.Tensor, T: int,
            scale: float, rows: Sequence[int]) -> torch.Tensor:
    """dQ of selected query rows of one head (Q,K,V,dO [N,d]), row by row.

    Row i needs only its own visible scores: P_i = exp(s_i - LSE_i),
    O_i = P_i V, D_i = <dO_i, O_i>, dS_ij = P_ij (<dO_i, v_j> - D_i),
    dQ_i = scale * sum_j dS_ij k_j.
    """
    q, k, v, do = q.to(F64), k.to(F64), v.to(F64), do.to(F64)
    out = []
    for i in rows:
        end = (chunk_of(i, T) + 1) * T
        s = scale * (k[:end] @ q[i])
        p = torch.exp(s - _row_lse(s.unsqueeze(0))[0])
        o_i = p @ v[:end]
        ds = p * (v[:end] @ do[i] - do[i] @ o_i)
        out.append(scale * (ds @ k[:end]))
    return torch.stack(out)


def dkv_rows(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, do: torch.Tensor, T: int,
             scale: float, rows: Sequence[int], block: int = 256
             ) -> Tuple[torch.Tensor, torch.Tensor]:
    """(dK, dV) of selected key rows of one head (Q,K,V,dO [N,d]).

    Key j is seen by the queries i with chunk(i) >= chunk(j).  Each such
    query needs its own LSE_i and D_i = <dO_i, O_i> over its visible keys
    [0, (chunk(i)+1) T); then P_ij = exp(s_ij - LSE_i),
    dS_ij = P_ij (<dO_i, v_j> - D_i), dV_j = sum_i P_ij dO_i and
    dK_j = scale * sum_i dS_ij q_i.  The queries are taken ``block`` rows at a
    time (rows of one block share no state), starting at the first query that
    sees the earliest selected key, so sampling late keys stays cheap.
    """
    q, k, v, do = q.to(F64), k.to(F64), v.to(F64), do.to(F64)
    N = q.shape[0]
    rows = list(rows)
    sel = torch.tensor(rows, dtype=torch.long)
    sel_chunk = sel // T
    dk = torch.zeros(len(rows), k.shape[1], dtype=F64)
    dv = torch.zeros(len(rows), v.shape[1], dtype=F64)
    i0 = int(sel_chunk.min()) * T
    for c in range(i0 // T, N // T):
        end = (c + 1) * T                      # keys visible to chunk c
        for b0 in range(c * T, end, block):
            qi, doi = q[b0:min(end, b0 + block)], do[b0:min(end, b0 + block)]
            s = scale * (qi @ k[:end].T)
            lse = _row_lse(s)
            p = torch.exp(s - lse.unsqueeze(-1))
            D = (doi * (p @ v[:end])).sum(-1)
            seen = sel_chunk <= c              # selected keys this chunk sees
            if not bool(seen.any()):
                continue
            idx = sel[seen]
            ps = p[:, idx]
            ds = ps * (doi @ v[idx].T - D.unsqueeze(-1))
            dv[seen] += ps.T @ doi
            dk[seen] += scale * (ds.T @ qi)
    return dk, dv


# --------------------------------------------------------------------------
# rolling KV cache (Sec. 3.5): ring of committed chunks + in-flight chunks
# --------------------------------------------------------------------------

def ring_logical(ring: torch.Tensor, cap: int, head: int, length: int) -> torch.Tensor:
    """Cached rows in logical (oldest first) order: logical t -> physical (head+t) mod cap.

    ``ring`` is [B, H, cap, d]; the result is [B, H, length, d].
    """
    assert ring.shape[-2] == cap and 0 <= head < cap and 0 <= length <= cap
    idx = torch.tensor([(head + t) % cap for t in range(length)], dtype=torch.long)
    return ring.index_select(-2, idx)


def rope_rotate(x: torch.Tensor, frames: torch.Tensor, rope_dims: int,
                base: float) -> torch.Tensor:
    """Temporal rotary embedding of the rows of ``x`` [..., N, d] (fp64 copy).

    Row n sits at temporal position ``frames[n]``; channel pair (2i, 2i+1)
    for i < rope_dims / 2 turns by the angle frames[n] * base^(-2i/rope_dims);
    the other channels are unchanged.  (The paper implies RoPE on the latent
    tokens and re-shifts the temporal positions of cached keys, Sec. 3.5, but
    states neither the channel layout nor the frequencies: both are inputs.)
    """
    x = x.to(F64).clone()
    for i in range(rope_dims // 2):
        theta = frames.to(F64) * (float(base) ** (-2.0 * i / rope_dims))
        c, s = torch.cos(theta), torch.sin(theta)
        a, b = x[..., 2 * i].clone(), x[..., 2 * i + 1].clone()
        x[..., 2 * i] = a * c - b * s
        x[..., 2 * i + 1] = a * s + b * c
    return x


def qkv_split_rope(qkv: torch.Tensor, rope_dims: int = 0, base: float = 10000.0,
                   tokens_per_frame: int = 1, first_frame: int = 0
                   ) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Head-major Q, K, V [B, H, N, d] (fp64) from a fused QKV projection
    ``qkv`` [B, N, 3, H, d] (index 0 = Q, 1 = K, 2 = V along dim 2).

    Token t sits at frame first_frame + t // tokens_per_frame; Q and K are
    turned by ``rope_rotate`` at those frames (the temporal positions of
    Sec. 3.5), V is moved unchanged.
    """
    x = qkv.to(F64).permute(2, 0, 3, 1, 4)  # [3, B, H, N, d]
    N = qkv.shape[1]
    frames = first_frame + torch.arange(N) // tokens_per_frame
    q = rope_rotate(x[0], frames, rope_dims, base)
    k = rope_rotate(x[1], frames, rope_dims, base)
    return q, k, x[2].clone()


def cache_fwd(q: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor,
              k_ring: torch.Tensor, v_ring: torch.Tensor, cap: int, head: int,
              length: int, T: int, scale: float, k_sink: torch.Tensor = None,
              v_sink: torch.Tensor = None, rope=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """(O, LSE) of W in-flight chunks (Q, K_new, V_new [B,H,W*T,d]).

    In-flight chunk j sees every cached token (the committed history, in
    logical order) and in-flight chunks 0..j (Sec. 3.5: a future chunk attends
    only to the committed history and to preceding chunks of the active window,
    itself included as in Sec. 3.2).  The committed history is the sink
    anchor (``k_sink``/``v_sink`` [B,H,S,d], the initial context that is never
    evicted and always comes first, Sec. 3.5 "Structured Rolling KV Cache"),
    if given, followed by the ring's ``length`` tokens.

    RoPE re-shifting (Sec. 3.5: after evictions the retained keys are
    re-indexed from the start of the window; the sink keeps the first
    position and is not re-shifted): with ``rope = (rope_dims, base,
    tokens_per_frame, first_frame)`` the ring holds keys without their
    temporal rotation, and ring token t (logical order) is rotated to frame
    first_frame + t // tokens_per_frame before it is used.  Sink and
    in-flight keys are used as given.
    """
    q, k_new, v_new = q.to(F64), k_new.to(F64), v_new.to(F64)
    kc = ring_logical(k_ring.to(F64), cap, head, length)
    vc = ring_logical(v_ring.to(F64), cap, head, length)
    if rope is not None and rope[0] > 0:
        rope_dims, base, per_frame, first_frame = rope
        frames = first_frame + torch.arange(length) // per_frame
        kc = rope_rotate(kc, frames, rope_dims, base)
    if k_sink is not None:
        kc = torch.cat([k_sink.to(F64), kc], dim=-2)
        vc = torch.cat([v_sink.to(F64), vc], dim=-2)
        length = length + k_sink.shape[-2]
    keys = torch.cat([kc, k_new], dim=-2)
    vals = torch.cat([vc, v_new], dim=-2)
    B, H, M, _ = q.shape
    assert M % T == 0
    W = M // T
    o = torch.empty(B, H, M, v_new.shape[-1], dtype=F64)
    lse = torch.empty(B, H, M, dtype=F64)
    for b in range(B):
        for h in range(H):
            for j in range(W):
                rows = slice(j * T, (j + 1) * T)
                visible = slice(0, length + (j + 1) * T)
                s = scale * (q[b, h, rows] @ keys[b, h, visible].T)
                l_j = _row_lse(s)
                o[b, h, rows] = torch.exp(s - l_j.unsqueeze(-1)) @ vals[b, h, visible]
                lse[b, h, rows] = l_j
    return o, lse


def cache_fwd_reshift(q: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor,
                      k_ring: torch.Tensor, v_ring: torch.Tensor, cap: int, head: int,
                      length: int, T: int, scale: float, k_sink: torch.Tensor,
                      v_sink: torch.Tensor, rope_dims: int, base: float,
                      shift: int) -> Tuple[torch.Tensor, torch.Tensor]:
    """(O, LSE) of the streaming forward with RoPE re-shifting (Sec. 3.5).

    The inputs carry their temporal RoPE: queries, in-flight keys and ring
    keys at their stream positions (frames counted from the start of the
    stream), the sink anchor at its own first position(s).  ``shift`` frames
    have been evicted from the FIFO.  Re-shifting subtracts that offset from
    the positions of the retained keys, and the active window (queries and
    in-flight keys) is re-indexed with them, so that every position stays in
    the trained range; the sink keeps its position.  Here that is done
    literally: the non-sink rows are turned back by ``shift`` frames, then the
    sink-anchored cache forward runs on the re-indexed tensors.
    """
    back = torch.full((1,), -int(shift))
    qs = rope_rotate(q, back, rope_dims, base)
    kns = rope_rotate(k_new, back, rope_dims, base)
    krs = rope_rotate(k_ring, back, rope_dims, base)
    return cache_fwd(qs, kns, v_new, krs, v_ring, cap, head, length, T, scale, k_sink, v_sink)


def cache_commit(k_ring: torch.Tensor, v_ring: torch.Tensor, cap: int, slot: int,
                 k_src: torch.Tensor, v_src: torch.Tensor) -> Tuple[torch.Tensor, torch.Tensor]:
    """New ring contents after writing ``rows`` tokens at physical rows (slot+r) mod cap.

    Returns copies; the inputs are not modified.
    """
    rows = k_src.shape[-2]
    assert 0 <= slot < cap and rows <= cap
    k_out, v_out = k_ring.clone(), v_ring.clone()
    for r in range(rows):
        p = (slot + r) % cap
        k_out[..., p, :] = k_src[..., r, :]
        v_out[..., p, :] = v_src[..., r, :]
    return k_out, v_out


def ring_advance(cap: int, head: int, length: int, rows: int) -> Tuple[int, int, int]:
    """FIFO bookkeeping for committing ``rows`` tokens (Sec. 3.5).

    Returns (slot, new_head, new_length): the new rows go after the newest
    cached token, at physical (head + length) mod cap; when the ring would
    overflow, the oldest rows are evicted by moving ``head`` forward.
    """
    slot = (head + length) % cap
    total = length + rows
    if total <= cap:
        return slot, head, total
    evicted = total - cap
    return slot, (head + evicted) % cap, cap
