"""GB300 (sm_103a) block-causal attention for streaming video world models.

Python binding of the C ABI in ``include/mw_bca.h`` (argument marshalling
only; every step of the computation runs in the library's CUDA kernels).
PyTorch provides device memory and the current stream.  There is no CPU
path: without the built library every call raises.

Entry points (same names as the C ABI, taking torch tensors):
  mw_bca_fwd(q, k, v, T_chunk, scale=None, need_lse=True) -> (o, lse)
  mw_bca_bwd(q, k, v, o, lse, dout, T_chunk, scale=None) -> (dq, dk, dv)
  mw_bca_cache_fwd(q, k_new, v_new, k_cache, v_cache, cache_head, cache_len,
                   T_chunk, scale=None, need_lse=True) -> (o, lse)
  mw_bca_cache_fwd_sink(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache,
                        cache_head, cache_len, T_chunk, ...) -> (o, lse)
  mw_bca_cache_fwd_rope(..., rope_dims, rope_base, shift_frames)
  mw_bca_cache_commit(k_cache, v_cache, slot_start, k_src, v_src)
  mw_device_status(clear=True), mw_set_option(name, value)
Tensors are contiguous bf16 [B, H, rows, d] on the current CUDA device.
"""
from __future__ import annotations

import ctypes
import math
import os
from typing import Optional, Tuple

import torch

__all__ = [
    "MWError", "library", "lib_path", "mw_bca_fwd", "mw_bca_bwd", "mw_bca_cache_fwd",
    "mw_bca_cache_fwd_sink", "mw_bca_cache_fwd_rope", "mw_bca_cache_step",
    "mw_bca_cache_commit", "mw_bca_bwd_workspace_size", "mw_bca_bwd_head_groups",
    "mw_bca_cache_workspace_size",
    "mw_device_status", "mw_set_option", "mw_qkv_rope_split", "BlockCausalAttention",
    "EXPORTED_SYMBOLS",
    "RingState",
]

_PKG = os.path.dirname(os.path.abspath(__file__))
lib_path = os.path.join(_PKG, "_lib", "libmw_bca.so")

EXPORTED_SYMBOLS = (
    "mw_bca_fwd", "mw_bca_bwd_workspace_size", "mw_bca_bwd", "mw_bca_bwd_stage",
    "mw_bca_cache_workspace_size",
    "mw_bca_cache_fwd", "mw_bca_cache_commit", "mw_status_string", "mw_last_error",
    "mw_device_status", "mw_set_option", "mw_bca_cache_fwd_noalloc", "mw_bca_cache_fwd_sink",
    "mw_bca_cache_fwd_rope", "mw_qkv_rope_split", "mw_bca_cache_step", "mw_bca_bwd_head_groups",
)

STATUS = {0: "MW_OK", 1: "MW_ERR_INVALID_ARG", 2: "MW_ERR_UNSUPPORTED", 3: "MW_ERR_CUDA",
          4: "MW_ERR_TIMEOUT", 5: "MW_ERR_WORKSPACE"}


class MWError(RuntimeError):
    """A non-zero mw_status from the library, with mw_last_error()'s text."""

    def __init__(self, code: int, message: str):
        super().__init__(f"{STATUS.get(code, code)}: {message}")
        self.code = code


_lib: Optional[ctypes.CDLL] = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_Z = ctypes.c_size_t


def library() -> ctypes.CDLL:
    """The loaded C library (raises when it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(lib_path):
        raise RuntimeError(
            f"{lib_path} is missing: build it with `python -c 'import __graft_entry__ as g; "
            "g.build()'` (there is no CPU fallback)")
    lib = ctypes.CDLL(lib_path)
    sig = {
        "mw_bca_fwd": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_bwd_workspace_size": (_Z, [_I, _I, _I, _I, _I]),
        "mw_bca_bwd_head_groups": (_I, [_I, _I, _I, _I, _I, _I]),
        "mw_bca_bwd": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _Z,
                            _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_bwd_stage": (_I, [_I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _Z,
                                  _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_cache_workspace_size": (_Z, [_I, _I, _I, _I, _I, _I]),
        "mw_bca_cache_fwd": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _Z,
                                  _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_cache_fwd_sink": (_I, [_P, _P, _P, _P, _P, _I, _P, _P, _I, _I, _I, _P, _P, _P,
                                       _Z, _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_cache_fwd_rope": (_I, [_P, _P, _P, _P, _P, _I, _P, _P, _I, _I, _I, _I, _F, _I,
                                       _P, _P, _P, _Z, _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_cache_commit": (_I, [_P, _P, _I, _I, _P, _P, _I, _I, _I, _I, _P]),
        "mw_qkv_rope_split": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _F, _I, _I, _P]),
        "mw_bca_cache_step": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _Z,
                                   _I, _I, _I, _I, _I, _F, _P]),
        "mw_bca_cache_fwd_noalloc": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _P, _P,
                                          _I, _I, _I, _I, _I, _F, _P]),
        "mw_status_string": (ctypes.c_char_p, [_I]),
        "mw_last_error": (ctypes.c_char_p, []),
        "mw_device_status": (_I, [_P, _I]),
        "mw_set_option": (_I, [ctypes.c_char_p, ctypes.c_longlong]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(code: int) -> None:
    if code != 0:
        msg = library().mw_last_error().decode(errors="replace")
        raise MWError(code, msg)


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _bhnd(t: torch.Tensor, name: str) -> Tuple[int, int, int, int]:
    """Shape of a contiguous bf16 [B, H, rows, d] tensor (its device is
    checked by _on_device, once every shape is known to be right)."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor, got {type(t).__name__}")
    if t.dtype != torch.bfloat16:
        raise TypeError(f"{name} must be bfloat16, got {t.dtype}")
    if t.dim() != 4 or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous [B, H, rows, d] tensor")
    return tuple(t.shape)  # type: ignore[return-value]


def _expect(t, name: str, shape, dtype=torch.bfloat16) -> None:
    """A caller-supplied output buffer: exactly this shape and dtype,
    contiguous.  The library cannot see buffer sizes, so a short buffer
    would be written past its end."""
    if not isinstance(t, torch.Tensor) or t.dtype != dtype or not t.is_contiguous() \
            or tuple(t.shape) != tuple(shape):
        got = (f"{t.dtype} {tuple(t.shape)}" + ("" if t.is_contiguous() else " non-contiguous")
               if isinstance(t, torch.Tensor) else type(t).__name__)
        raise ValueError(f"{name} must be a contiguous {dtype} tensor of shape {tuple(shape)}, "
                         f"got {got}")


def _chunks(rows: int, T_chunk: int, what: str) -> int:
    if int(T_chunk) < 1:
        raise ValueError(f"T_chunk must be >= 1, got {T_chunk}")
    if rows % T_chunk != 0:
        raise ValueError(f"{what} {rows} is not a multiple of T_chunk={T_chunk}")
    return rows // T_chunk


def _on_device(ref: torch.Tensor, named) -> None:
    """Every tensor on ref's CUDA device, and that device current (the
    library launches on the current device and stream)."""
    if not ref.is_cuda:
        raise ValueError("the tensors must be CUDA tensors (there is no CPU path)")
    for name, t in named:
        if t is not None and t.device != ref.device:
            raise ValueError(f"{name} is on {t.device}, the other tensors on {ref.device}")
    if ref.device.index != torch.cuda.current_device():
        raise ValueError(f"the tensors are on {ref.device} but the current device is "
                         f"cuda:{torch.cuda.current_device()}: call under torch.cuda.device")


def _no_alias(outputs, inputs) -> None:
    """No output buffer shares bytes with an input or with another output
    (the kernels read inputs while they write outputs)."""
    spans = []
    for kind, group in (("output", outputs), ("input", inputs)):
        for name, t in group:
            if t is not None and t.numel() > 0:
                p = t.data_ptr()
                spans.append((f"{kind} {name}", p, p + t.numel() * t.element_size()))
    n_out = sum(1 for _, t in outputs if t is not None and t.numel() > 0)
    for a in range(n_out):
        for b in range(a + 1, len(spans)):
            if spans[a][1] < spans[b][2] and spans[b][1] < spans[a][2]:
                raise ValueError(f"{spans[a][0]} overlaps {spans[b][0]}")


def _workspace(ws: Optional[torch.Tensor], nbytes: int,
               device: torch.device) -> Optional[torch.Tensor]:
    """At least nbytes of device scratch (None when none is needed): the
    caller's buffer when it is large enough, else a new one."""
    if nbytes == 0:
        return None
    if ws is not None:
        if not ws.is_contiguous():
            raise ValueError("workspace must be contiguous")
        if ws.numel() * ws.element_size() >= nbytes:
            return ws
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def _scale(scale: Optional[float], d: int) -> float:
    return 1.0 / math.sqrt(d) if scale is None else float(scale)


def mw_bca_fwd(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, T_chunk: int,
               scale: Optional[float] = None, need_lse: bool = True,
               out: Optional[Tuple[torch.Tensor, Optional[torch.Tensor]]] = None
               ) -> Tuple[torch.Tensor, Optional[torch.Tensor]]:
    """Block-causal attention forward (Sec. 3.2); returns (O, LSE or None).

    ``out`` = (o, lse) reuses caller buffers (lse may be None)."""
    B, H, N, d = _bhnd(q, "q")
    for t, n in ((k, "k"), (v, "v")):
        if _bhnd(t, n) != (B, H, N, d):
            raise ValueError(f"{n} shape {tuple(t.shape)} != q shape {(B, H, N, d)}")
    n_chunks = _chunks(N, T_chunk, "sequence length")
    o, lse = out if out is not None else (None, None)
    if out is not None:
        _expect(o, "o", (B, H, N, d))
        if lse is not None:
            _expect(lse, "lse", (B, H, N), torch.float32)
    _on_device(q, (("k", k), ("v", v), ("o", o), ("lse", lse)))
    if out is None:
        o = torch.empty_like(q)
        lse = torch.empty((B, H, N), dtype=torch.float32, device=q.device) if need_lse else None
    else:
        _no_alias((("o", o), ("lse", lse)), (("q", q), ("k", k), ("v", v)))
    _check(library().mw_bca_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), B, H,
                                n_chunks, T_chunk, d, _scale(scale, d), _stream()))
    return o, lse


def mw_bca_bwd_workspace_size(B: int, H: int, n_chunks: int, T_chunk: int, d: int) -> int:
    return int(library().mw_bca_bwd_workspace_size(B, H, n_chunks, T_chunk, d))


def mw_bca_bwd_head_groups(B: int, H: int, n_chunks: int, T_chunk: int, d: int,
                           sm_count: int = 0) -> int:
    """Head groups of the backward's CTA order for these sizes (B*H = head by
    head); host-side planning only."""
    g = int(library().mw_bca_bwd_head_groups(B, H, n_chunks, T_chunk, d, sm_count))
    if g < 0:
        raise MWError(1, library().mw_last_error().decode(errors="replace"))
    return g


def mw_bca_bwd(q, k, v, o, lse, dout, T_chunk: int, scale: Optional[float] = None,
               workspace: Optional[torch.Tensor] = None, stage: int = 0, out=None):
    """Gradients (dQ, dK, dV) of sum(O * dout) through mw_bca_fwd.

    ``stage`` 1/2/3 runs one stage of the backward (see mw_bca_bwd_stage);
    ``out`` = (dq, dk, dv) preallocated outputs."""
    B, H, N, d = _bhnd(q, "q")
    for t, n in ((k, "k"), (v, "v"), (o, "o"), (dout, "dout")):
        if _bhnd(t, n) != (B, H, N, d):
            raise ValueError(f"{n} shape {tuple(t.shape)} != q shape {(B, H, N, d)}")
    _expect(lse, "lse", (B, H, N), torch.float32)
    n = _chunks(N, T_chunk, "sequence length")
    dq, dk, dv = out if out is not None else (None, None, None)
    if out is not None:
        for t, name in ((dq, "dq"), (dk, "dk"), (dv, "dv")):
            _expect(t, name, (B, H, N, d))
    _on_device(q, (("k", k), ("v", v), ("o", o), ("lse", lse), ("dout", dout), ("dq", dq),
                   ("dk", dk), ("dv", dv), ("workspace", workspace)))
    ws_bytes = mw_bca_bwd_workspace_size(B, H, n, T_chunk, d)
    workspace = _workspace(workspace, ws_bytes, q.device)
    if out is None:
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    _no_alias((("dq", dq), ("dk", dk), ("dv", dv), ("workspace", workspace)),
              (("q", q), ("k", k), ("v", v), ("o", o), ("lse", lse), ("dout", dout)))
    _check(library().mw_bca_bwd_stage(stage, _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse),
                                      _ptr(dout), _ptr(dq), _ptr(dk), _ptr(dv), _ptr(workspace),
                                      ws_bytes, B, H, n, T_chunk, d, _scale(scale, d), _stream()))
    return dq, dk, dv


def mw_bca_cache_workspace_size(B: int, H: int, n_q_chunks: int, T_chunk: int, d: int,
                                cache_len: int) -> int:
    return int(library().mw_bca_cache_workspace_size(B, H, n_q_chunks, T_chunk, d, cache_len))


def mw_bca_cache_fwd(q, k_new, v_new, k_cache, v_cache, cache_head: int, cache_len: int,
                     T_chunk: int, scale: Optional[float] = None, need_lse: bool = True,
                     workspace: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None):
    """In-flight chunks against the rolling KV cache (Sec. 3.5); returns (O, LSE or None)."""
    return _cache_fwd(q, k_new, v_new, None, None, k_cache, v_cache, cache_head, cache_len,
                      T_chunk, scale, need_lse, workspace, out)


def mw_bca_cache_fwd_sink(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache, cache_head: int,
                          cache_len: int, T_chunk: int, scale: Optional[float] = None,
                          need_lse: bool = True, workspace: Optional[torch.Tensor] = None,
                          out: Optional[torch.Tensor] = None):
    """As mw_bca_cache_fwd with a sink anchor k_sink / v_sink [B, H, S, d] that
    every in-flight chunk sees ahead of the ring (Sec. 3.5); returns (O, LSE or None)."""
    return _cache_fwd(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache, cache_head, cache_len,
                      T_chunk, scale, need_lse, workspace, out)


def mw_bca_cache_fwd_rope(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache, cache_head: int,
                          cache_len: int, T_chunk: int, rope_dims: int, rope_base: float,
                          shift_frames: int, scale: Optional[float] = None,
                          need_lse: bool = True, workspace: Optional[torch.Tensor] = None,
                          out: Optional[torch.Tensor] = None):
    """As mw_bca_cache_fwd_sink (k_sink may be None) with RoPE re-shifting
    (Sec. 3.5): queries, in-flight and ring keys rotated at their stream
    positions, the sink at its own, ``shift_frames`` frames evicted; the
    sink's keys turn forward by the shift as they are read.  Returns
    (O, LSE or None)."""
    return _cache_fwd(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache, cache_head, cache_len,
                      T_chunk, scale, need_lse, workspace, out,
                      rope=(rope_dims, rope_base, shift_frames))


def _cache_fwd(q, k_new, v_new, k_sink, v_sink, k_cache, v_cache, cache_head, cache_len,
               T_chunk, scale, need_lse, workspace, out, rope=None, commit=None):
    B, H, M, d = _bhnd(q, "q")
    for t, n in ((k_new, "k_new"), (v_new, "v_new")):
        if _bhnd(t, n) != (B, H, M, d):
            raise ValueError(f"{n} shape {tuple(t.shape)} != q shape {(B, H, M, d)}")
    Bc, Hc, cap, dc = _bhnd(k_cache, "k_cache")
    if (Bc, Hc, dc) != (B, H, d) or tuple(v_cache.shape) != tuple(k_cache.shape):
        raise ValueError("k_cache / v_cache must be [B, H, cap, d] matching q")
    _bhnd(v_cache, "v_cache")
    W = _chunks(M, T_chunk, "query rows")
    sink_len = 0
    if k_sink is not None:
        Bs, Hs, sink_len, ds = _bhnd(k_sink, "k_sink")
        _bhnd(v_sink, "v_sink")
        if (Bs, Hs, ds) != (B, H, d) or tuple(v_sink.shape) != tuple(k_sink.shape):
            raise ValueError("k_sink / v_sink must be [B, H, S, d] matching q")
    if out is not None:
        _expect(out, "out", (B, H, M, d))
    _on_device(q, (("k_new", k_new), ("v_new", v_new), ("k_cache", k_cache),
                   ("v_cache", v_cache), ("k_sink", k_sink), ("v_sink", v_sink), ("out", out),
                   ("workspace", workspace)))
    ws_bytes = mw_bca_cache_workspace_size(B, H, W, T_chunk, d, sink_len + cache_len)
    workspace = _workspace(workspace, ws_bytes, q.device)
    o = torch.empty_like(q) if out is None else out
    lse = torch.empty((B, H, M), dtype=torch.float32, device=q.device) if need_lse else None
    # the streaming step also writes the ring (its commit)
    ring = (("k_cache", k_cache), ("v_cache", v_cache))
    _no_alias((("out", o), ("lse", lse), ("workspace", workspace))
              + (ring if commit is not None else ()),
              (("q", q), ("k_new", k_new), ("v_new", v_new), ("k_sink", k_sink),
               ("v_sink", v_sink)) + (ring if commit is None else ()))
    if commit is not None:
        _check(library().mw_bca_cache_step(
            _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), cap, cache_head,
            cache_len, int(commit[0]), int(commit[1]), _ptr(o), _ptr(lse),
            _ptr(workspace), ws_bytes, B, H, W, T_chunk, d,
            _scale(scale, d), _stream()))
    elif rope is not None:
        _check(library().mw_bca_cache_fwd_rope(
            _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_sink), _ptr(v_sink), sink_len,
            _ptr(k_cache), _ptr(v_cache), cap, cache_head, cache_len, int(rope[0]),
            float(rope[1]), int(rope[2]), _ptr(o), _ptr(lse),
            _ptr(workspace), ws_bytes, B, H, W, T_chunk, d,
            _scale(scale, d), _stream()))
    elif k_sink is None:
        _check(library().mw_bca_cache_fwd(
            _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), cap, cache_head,
            cache_len, _ptr(o), _ptr(lse), _ptr(workspace), ws_bytes,
            B, H, W, T_chunk, d, _scale(scale, d), _stream()))
    else:
        _check(library().mw_bca_cache_fwd_sink(
            _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_sink), _ptr(v_sink), sink_len,
            _ptr(k_cache), _ptr(v_cache), cap, cache_head, cache_len, _ptr(o), _ptr(lse),
            _ptr(workspace), ws_bytes, B, H, W, T_chunk, d,
            _scale(scale, d), _stream()))
    return o, lse


def mw_bca_cache_step(q, k_new, v_new, k_cache, v_cache, cache_head: int, cache_len: int,
                      commit_slot: int, commit_rows: int, T_chunk: int,
                      scale: Optional[float] = None, need_lse: bool = True,
                      workspace: Optional[torch.Tensor] = None, out: Optional[torch.Tensor] = None):
    """One streaming step (Sec. 3.5): mw_bca_cache_fwd, then the first
    ``commit_rows`` rows of k_new / v_new go to ring rows (commit_slot + r) mod
    cap (FIFO eviction); returns (O, LSE or None)."""
    return _cache_fwd(q, k_new, v_new, None, None, k_cache, v_cache, cache_head, cache_len,
                      T_chunk, scale, need_lse, workspace, out,
                      commit=(commit_slot, commit_rows))


def mw_bca_cache_commit(k_cache, v_cache, slot_start: int, k_src, v_src) -> None:
    """Write k_src / v_src rows at ring rows (slot_start + r) mod cap (Sec. 3.5)."""
    B, H, cap, d = _bhnd(k_cache, "k_cache")
    _bhnd(v_cache, "v_cache")
    Bs, Hs, rows, ds = _bhnd(k_src, "k_src")
    _bhnd(v_src, "v_src")
    if (Bs, Hs, ds) != (B, H, d) or tuple(v_src.shape) != tuple(k_src.shape):
        raise ValueError("k_src / v_src must be [B, H, rows, d] matching the cache")
    if tuple(v_cache.shape) != (B, H, cap, d):
        raise ValueError("k_cache / v_cache must have the same shape")
    _on_device(k_cache, (("v_cache", v_cache), ("k_src", k_src), ("v_src", v_src)))
    _no_alias((("k_cache", k_cache), ("v_cache", v_cache)), (("k_src", k_src), ("v_src", v_src)))
    _check(library().mw_bca_cache_commit(_ptr(k_cache), _ptr(v_cache), cap, slot_start,
                                         _ptr(k_src), _ptr(v_src), rows, B, H, d, _stream()))


def mw_qkv_rope_split(qkv: torch.Tensor, rope_dims: int = 0, rope_base: float = 10000.0,
                      tokens_per_frame: int = 1, first_frame: int = 0,
                      out: Optional[Tuple[torch.Tensor, torch.Tensor, torch.Tensor]] = None
                      ) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Split a fused QKV projection [B, N, 3, H, d] into head-major Q, K, V
    [B, H, N, d], turning the first ``rope_dims`` channels of Q and K by their
    frame's temporal rotary angle (token t at frame first_frame + t //
    tokens_per_frame; Sec. 3.2 inputs, Sec. 3.5 positions)."""
    if not isinstance(qkv, torch.Tensor) or qkv.dtype != torch.bfloat16:
        raise TypeError("qkv must be a bfloat16 tensor")
    if qkv.dim() != 5 or qkv.shape[2] != 3 or not qkv.is_contiguous():
        raise ValueError("qkv must be a contiguous [B, N, 3, H, d] tensor")
    B, N, _, H, d = qkv.shape
    if out is not None:
        if len(out) != 3:
            raise ValueError("out must be (q, k, v)")
        for t, name in zip(out, ("q", "k", "v")):
            _expect(t, name, (B, H, N, d))
    _on_device(qkv, tuple(zip(("q", "k", "v"), out)) if out is not None else ())
    if out is None:
        out = tuple(torch.empty(B, H, N, d, dtype=torch.bfloat16, device=qkv.device)
                    for _ in range(3))
    q, k, v = out
    _no_alias((("q", q), ("k", k), ("v", v)), (("qkv", qkv),))
    _check(library().mw_qkv_rope_split(_ptr(qkv), _ptr(q), _ptr(k), _ptr(v), B, N, H, d,
                                       int(rope_dims), float(rope_base), int(tokens_per_frame),
                                       int(first_frame), _stream()))
    return q, k, v


def mw_device_status(clear: bool = True) -> int:
    """Synchronises the current stream and returns the device status code."""
    return int(library().mw_device_status(_stream(), 1 if clear else 0))


def mw_set_option(name: str, value: int) -> None:
    _check(library().mw_set_option(name.encode(), int(value)))


class RingState:
    """Host-side FIFO bookkeeping of a rolling KV cache (Sec. 3.5).

    ``head`` is the physical row of the logically oldest cached token and
    ``length`` the number of cached tokens.  ``commit(rows)`` returns the
    physical slot where the next ``rows`` tokens are written -- right after
    the newest token -- and evicts the oldest tokens when the ring overflows.
    """

    def __init__(self, cap: int, head: int = 0, length: int = 0):
        if not (cap >= 1 and 0 <= head < cap and 0 <= length <= cap):
            raise ValueError(f"bad ring state cap={cap} head={head} length={length}")
        self.cap, self.head, self.length = cap, head, length

    def commit(self, rows: int) -> int:
        if not 1 <= rows <= self.cap:
            raise ValueError(f"rows={rows} not in [1, {self.cap}]")
        slot = (self.head + self.length) % self.cap
        overflow = max(0, self.length + rows - self.cap)
        self.head = (self.head + overflow) % self.cap
        self.length = min(self.cap, self.length + rows)
        return slot


class BlockCausalAttention(torch.autograd.Function):
    """Autograd wrapper: O = block-causal attention(q, k, v) with chunks of T_chunk."""

    @staticmethod
    def forward(ctx, q, k, v, T_chunk: int, scale: Optional[float] = None):
        o, lse = mw_bca_fwd(q, k, v, T_chunk, scale, need_lse=True)
        ctx.save_for_backward(q, k, v, o, lse)
        ctx.T_chunk, ctx.scale = T_chunk, scale
        return o

    @staticmethod
    def backward(ctx, do):
        q, k, v, o, lse = ctx.saved_tensors
        dq, dk, dv = mw_bca_bwd(q, k, v, o, lse, do.contiguous(), ctx.T_chunk, ctx.scale)
        return dq, dk, dv, None, None
