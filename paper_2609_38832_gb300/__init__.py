"""NAMOH routed attention on GB300 (sm_103a): Python binding of the C ABI.

The three calls keep the C names (``namoh_route``, ``namoh_prefill``,
``namoh_decode``).  They only marshal torch tensors into device pointers and the
current CUDA stream; every step of the path runs in the CUDA kernels of
``libnamoh.so``.  PyTorch supplies device memory and streams.  There is no CPU
or PyTorch fallback: a missing library or a non-CUDA tensor is an error.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch

from . import _abi
from ._abi import (NAMOH_DEV_BAD_SEQLENS, NAMOH_DEV_CAPACITY, NAMOH_DEV_NONFINITE_SCORE, NAMOH_DEV_TIMEOUT,
                   NAMOH_ROPE_GLOBAL, NAMOH_ROPE_INTERLEAVED, NamohError)

__all__ = ["namoh_route", "namoh_route_varlen", "namoh_prefill", "namoh_prefill_varlen", "namoh_decode",
           "namoh_proj_qkv", "namoh_proj_out", "namoh_shared_prefill", "namoh_shared_decode", "namoh_sa_prefill",
           "namoh_rope_pack", "namoh_attention_plan", "namoh_attention", "RouteOutputs", "Workspace", "NamohError",
           "NAMOH_DEV_BAD_SEQLENS", "NAMOH_DEV_CAPACITY", "NAMOH_DEV_NONFINITE_SCORE", "NAMOH_DEV_TIMEOUT",
           "NAMOH_ROPE_GLOBAL", "NAMOH_ROPE_INTERLEAVED", "library_path"]


def library_path() -> str:
    return _abi.LIB_PATH


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("namoh: every tensor argument must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("namoh: tensor arguments must be contiguous")
    return t.data_ptr()


def _stream(stream: Optional[torch.cuda.Stream]):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


class Workspace:
    """A reusable device scratch buffer (grown on demand, 256-byte aligned by the allocator)."""

    def __init__(self, device=None):
        self.device = device
        self.buf: Optional[torch.Tensor] = None

    def get(self, nbytes: int, device) -> torch.Tensor:
        nbytes = max(int(nbytes), 256)
        if self.buf is None or self.buf.numel() < nbytes or self.buf.device != torch.device(device):
            self.buf = torch.empty(nbytes, dtype=torch.uint8, device=device)
        return self.buf


def _ws(ws: Optional[Workspace], nbytes: int, device) -> torch.Tensor:
    return (ws or Workspace()).get(nbytes, device)


def _status(status: Optional[torch.Tensor], device) -> torch.Tensor:
    if status is None:
        status = torch.zeros(1, dtype=torch.int32, device=device)
    return status


@dataclasses.dataclass
class RouteOutputs:
    topk_head: torch.Tensor
    gate: torch.Tensor
    rank: Optional[torch.Tensor]
    row: Optional[torch.Tensor]
    seg_offsets: Optional[torch.Tensor]
    row_src: Optional[torch.Tensor]
    status: torch.Tensor


def namoh_route(scores: torch.Tensor, K: int, compact: bool = True, workspace: Optional[Workspace] = None,
                status: Optional[torch.Tensor] = None, out: Optional[RouteOutputs] = None,
                stream=None, bias: Optional[torch.Tensor] = None) -> RouteOutputs:
    """Routing and dispatch of scores [B, T, H] fp32 (see namoh_route in include/namoh.h).

    With ``bias`` ([H] fp32 on the device) the selection is TopK(a + b) on the softmax
    affinities while the gates stay a (namoh_route_biased)."""
    lib = _abi.load()
    if scores.dtype != torch.float32 or scores.dim() != 3:
        raise ValueError("scores must be a [B, T, H] float32 tensor")
    B, T, H = scores.shape
    dev = scores.device
    if bias is not None and (bias.dtype != torch.float32 or bias.shape != (H,) or bias.device != dev
                             or not bias.is_contiguous()):
        raise ValueError("bias must be a contiguous [H] float32 tensor on the scores' device")
    if out is None:
        i32 = dict(dtype=torch.int32, device=dev)
        out = RouteOutputs(
            topk_head=torch.empty((B, T, K), **i32), gate=torch.empty((B, T, K), dtype=torch.float32, device=dev),
            rank=torch.empty((B, T, K), **i32) if compact else None,
            row=torch.empty((B, T, K), **i32) if compact else None,
            seg_offsets=torch.empty(B * H + 1, **i32) if compact else None,
            row_src=torch.empty(B * T * K, **i32) if compact else None,
            status=_status(status, dev))
    nbytes = lib.namoh_route_workspace_size(B, T, H, K)
    ws = _ws(workspace, nbytes, dev)
    outs = (_ptr(out.topk_head), _ptr(out.gate), _ptr(out.rank), _ptr(out.row), _ptr(out.seg_offsets),
            _ptr(out.row_src), _ptr(ws), ws.numel(), _ptr(out.status), _stream(stream))
    if bias is None:
        _abi.check("namoh_route", lib.namoh_route(_ptr(scores), B, T, H, K, *outs))
    else:
        _abi.check("namoh_route_biased", lib.namoh_route_biased(_ptr(scores), _ptr(bias), B, T, H, K, *outs))
    return out


def namoh_route_varlen(scores: torch.Tensor, cu_seqlens: torch.Tensor, max_seqlen: int, K: int,
                       compact: bool = True, workspace: Optional[Workspace] = None,
                       status: Optional[torch.Tensor] = None, out: Optional[RouteOutputs] = None, stream=None,
                       bias: Optional[torch.Tensor] = None) -> RouteOutputs:
    """Routing of a ragged batch (see namoh_route_varlen in include/namoh.h): scores [N, H] fp32
    over the flat token axis, cu_seqlens [B + 1] int32 on the device, max_seqlen the longest
    sequence.  Per-token outputs are [N, K]; row_src[row] = tok*K + slot."""
    lib = _abi.load()
    if scores.dtype != torch.float32 or scores.dim() != 2:
        raise ValueError("scores must be a [N, H] float32 tensor")
    if cu_seqlens.dtype != torch.int32 or cu_seqlens.dim() != 1 or cu_seqlens.device != scores.device:
        raise ValueError("cu_seqlens must be a 1-D int32 tensor on the scores' device")
    N, H = scores.shape
    B = cu_seqlens.numel() - 1
    dev = scores.device
    if bias is not None and (bias.dtype != torch.float32 or bias.shape != (H,) or bias.device != dev
                             or not bias.is_contiguous()):
        raise ValueError("bias must be a contiguous [H] float32 tensor on the scores' device")
    if out is None:
        i32 = dict(dtype=torch.int32, device=dev)
        out = RouteOutputs(
            topk_head=torch.empty((N, K), **i32), gate=torch.empty((N, K), dtype=torch.float32, device=dev),
            rank=torch.empty((N, K), **i32) if compact else None,
            row=torch.empty((N, K), **i32) if compact else None,
            seg_offsets=torch.empty(B * H + 1, **i32) if compact else None,
            row_src=torch.empty(N * K, **i32) if compact else None,
            status=_status(status, dev))
    nbytes = lib.namoh_route_workspace_size(B, max_seqlen, H, K)
    ws = _ws(workspace, nbytes, dev)
    rc = lib.namoh_route_varlen(_ptr(scores), _ptr(bias), _ptr(cu_seqlens), B, N, int(max_seqlen), H, K,
                                _ptr(out.topk_head), _ptr(out.gate), _ptr(out.rank), _ptr(out.row),
                                _ptr(out.seg_offsets), _ptr(out.row_src), _ptr(ws), ws.numel(), _ptr(out.status),
                                _stream(stream))
    _abi.check("namoh_route_varlen", rc)
    return out


def _rope_flags(interleaved: bool, global_positions: bool) -> int:
    return (_abi.NAMOH_ROPE_INTERLEAVED if interleaved else 0) | (_abi.NAMOH_ROPE_GLOBAL if global_positions else 0)


def namoh_prefill(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, seg_offsets: torch.Tensor,
                  row_src: torch.Tensor, gate: torch.Tensor, *, B: int, T: int, H: int, K: int, group: int = 1,
                  rope_base: float = 10000.0, interleaved: bool = False, global_positions: bool = False,
                  y: Optional[torch.Tensor] = None,
                  k_cache: Optional[torch.Tensor] = None, v_cache: Optional[torch.Tensor] = None,
                  seg_base: Optional[torch.Tensor] = None, seg_cap: Optional[torch.Tensor] = None,
                  seg_len: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
                  status: Optional[torch.Tensor] = None, stream=None):
    """Prefill over packed rows (see namoh_prefill in include/namoh.h).

    q [R*g, d], k / v [R, d] bf16; returns (y [B, T, K, d], k_cache, v_cache).
    With v_cache omitted and no seg_base, v itself serves as the value cache.
    interleaved / global_positions select the RoPE variants (NAMOH_ROPE_* in the header).
    """
    lib = _abi.load()
    d = q.shape[-1]
    dev = q.device
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16:
            raise ValueError(f"{name} must be bfloat16")
    if y is None:
        y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    if k_cache is None:
        k_cache = torch.empty_like(k)
    if v_cache is None:
        v_cache = v if seg_base is None else torch.empty_like(v)
    cache_rows = k_cache.shape[0]
    nbytes = lib.namoh_prefill_workspace_size(B, T, H, K, d, group)
    if nbytes == 0:
        raise NamohError("namoh_prefill_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    rc = lib.namoh_prefill_ex(_ptr(q), _ptr(k), _ptr(v), B, T, H, K, d, group, float(rope_base),
                              _rope_flags(interleaved, global_positions), _ptr(seg_offsets), _ptr(row_src),
                              _ptr(gate), _ptr(y), _ptr(k_cache), _ptr(v_cache), _ptr(seg_base), _ptr(seg_cap),
                              cache_rows, _ptr(seg_len), _ptr(ws), ws.numel(), _ptr(st), _stream(stream))
    _abi.check("namoh_prefill_ex", rc)
    return y, k_cache, v_cache


def namoh_sa_prefill(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, seg_offsets: torch.Tensor,
                     row_src: torch.Tensor, gate: torch.Tensor, *, B: int, T: int, H: int, K: int, block: int = 32,
                     alpha_num: int = 1, alpha_den: int = 5, group: int = 1, rope_base: float = 10000.0,
                     interleaved: bool = False, global_positions: bool = False, y: Optional[torch.Tensor] = None,
                     sa_mask: Optional[torch.Tensor] = None, k_cache: Optional[torch.Tensor] = None,
                     v_cache: Optional[torch.Tensor] = None, seg_base: Optional[torch.Tensor] = None,
                     seg_cap: Optional[torch.Tensor] = None, seg_len: Optional[torch.Tensor] = None,
                     workspace: Optional[Workspace] = None, status: Optional[torch.Tensor] = None, stream=None):
    """SA + NAMOH prefill (see namoh_sa_prefill in include/namoh.h): block selection inside each routed
    history (blocks of `block` keys, retained fraction alpha_num / alpha_den), then the routed attention
    over the kept blocks.  Arguments as namoh_prefill; returns (y [B, T, K, d], sa_mask [R*g, W] int32
    bit patterns of the kept earlier blocks, k_cache, v_cache)."""
    lib = _abi.load()
    d = q.shape[-1]
    dev = q.device
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16:
            raise ValueError(f"{name} must be bfloat16")
    words = lib.namoh_sa_mask_words(T, block)
    if words == 0:
        raise NamohError("namoh_sa_mask_words", _abi.NAMOH_ERR_INVALID_ARG)
    if y is None:
        y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    if sa_mask is None:
        sa_mask = torch.empty((k.shape[0] * group, words), dtype=torch.int32, device=dev)
    if k_cache is None:
        k_cache = torch.empty_like(k)
    if v_cache is None:
        v_cache = v if seg_base is None else torch.empty_like(v)
    nbytes = lib.namoh_sa_prefill_workspace_size(B, T, H, K, d, group, block)
    if nbytes == 0:
        raise NamohError("namoh_sa_prefill_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    rc = lib.namoh_sa_prefill(_ptr(q), _ptr(k), _ptr(v), B, T, H, K, d, group, float(rope_base),
                              _rope_flags(interleaved, global_positions), _ptr(seg_offsets), _ptr(row_src),
                              _ptr(gate), int(block), int(alpha_num), int(alpha_den), _ptr(sa_mask), _ptr(y),
                              _ptr(k_cache), _ptr(v_cache), _ptr(seg_base), _ptr(seg_cap), k_cache.shape[0],
                              _ptr(seg_len), _ptr(ws), ws.numel(), _ptr(st), _stream(stream))
    _abi.check("namoh_sa_prefill", rc)
    return y, sa_mask, k_cache, v_cache


def namoh_prefill_varlen(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, cu_seqlens: torch.Tensor,
                         max_seqlen: int, seg_offsets: torch.Tensor, row_src: torch.Tensor, gate: torch.Tensor, *,
                         H: int, K: int, group: int = 1, rope_base: float = 10000.0, interleaved: bool = False,
                         global_positions: bool = False, y: Optional[torch.Tensor] = None,
                         k_cache: Optional[torch.Tensor] = None, v_cache: Optional[torch.Tensor] = None,
                         seg_base: Optional[torch.Tensor] = None, seg_cap: Optional[torch.Tensor] = None,
                         seg_len: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
                         status: Optional[torch.Tensor] = None, stream=None):
    """Prefill over a ragged batch routed by namoh_route_varlen (see namoh_prefill_varlen in
    include/namoh.h).  q [N*Kr*g, d], k / v [N*Kr, d] bf16 packed rows; returns
    (y [N, K, d], k_cache, v_cache) with N = gate.shape[0] tokens."""
    lib = _abi.load()
    d = q.shape[-1]
    dev = q.device
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16:
            raise ValueError(f"{name} must be bfloat16")
    B = cu_seqlens.numel() - 1
    N = gate.shape[0]
    if y is None:
        y = torch.empty((N, K, d), dtype=torch.bfloat16, device=dev)
    if k_cache is None:
        k_cache = torch.empty_like(k)
    if v_cache is None:
        v_cache = v if seg_base is None else torch.empty_like(v)
    nbytes = lib.namoh_prefill_varlen_workspace_size(B, N, int(max_seqlen), H, K, d, group)
    if nbytes == 0:
        raise NamohError("namoh_prefill_varlen_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    rc = lib.namoh_prefill_varlen(_ptr(q), _ptr(k), _ptr(v), _ptr(cu_seqlens), B, N, int(max_seqlen), H, K, d, group,
                                  float(rope_base), _rope_flags(interleaved, global_positions), _ptr(seg_offsets),
                                  _ptr(row_src), _ptr(gate), _ptr(y), _ptr(k_cache), _ptr(v_cache), _ptr(seg_base),
                                  _ptr(seg_cap), k_cache.shape[0], _ptr(seg_len), _ptr(ws), ws.numel(), _ptr(st),
                                  _stream(stream))
    _abi.check("namoh_prefill_varlen", rc)
    return y, k_cache, v_cache


def namoh_rope_pack(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, seg_offsets: torch.Tensor, *, B: int, T: int,
                    H: int, K: int, group: int = 1, rope_base: float = 10000.0, interleaved: bool = False,
                    row_src: Optional[torch.Tensor] = None, q_rot: Optional[torch.Tensor] = None,
                    k_cache: Optional[torch.Tensor] = None, v_cache: Optional[torch.Tensor] = None,
                    seg_base: Optional[torch.Tensor] = None, seg_cap: Optional[torch.Tensor] = None,
                    status: Optional[torch.Tensor] = None, plan: Optional[torch.Tensor] = None, stream=None):
    """Prefill stage 1: RoPE at rank and cache pack.  Returns (q_rot, k_cache, v_cache).

    With ``plan`` (a buffer from namoh_attention_plan) the same launch also rebuilds the
    attention plan for these seg_offsets.  Passing ``row_src`` selects global positions
    (NAMOH_ROPE_GLOBAL); ``interleaved`` the (2j, 2j+1) pairing."""
    lib = _abi.load()
    d = q.shape[-1]
    dev = q.device
    q_rot = torch.empty_like(q) if q_rot is None else q_rot
    k_cache = torch.empty_like(k) if k_cache is None else k_cache
    if v_cache is None:
        v_cache = v if seg_base is None else torch.empty_like(v)
    st = _status(status, dev)
    rc = lib.namoh_rope_pack_ex(_ptr(q), _ptr(k), _ptr(v), B, T, H, K, d, group, float(rope_base),
                                _rope_flags(interleaved, row_src is not None), _ptr(seg_offsets), _ptr(row_src),
                                _ptr(q_rot), _ptr(k_cache), _ptr(v_cache), _ptr(seg_base), _ptr(seg_cap),
                                k_cache.shape[0], _ptr(st), _ptr(plan), 0 if plan is None else plan.numel(),
                                _stream(stream))
    _abi.check("namoh_rope_pack_ex", rc)
    return q_rot, k_cache, v_cache


def namoh_attention_plan(seg_offsets: torch.Tensor, *, B: int, T: int, H: int, K: int, group: int = 1,
                         seg_cap: Optional[torch.Tensor] = None, plan: Optional[torch.Tensor] = None,
                         stream=None) -> torch.Tensor:
    """Prefill stage 2: the longest-first tile list.  Returns the plan buffer (uint8 tensor)."""
    lib = _abi.load()
    nbytes = lib.namoh_attention_plan_size(B, T, H, K, group)
    if nbytes == 0:
        raise NamohError("namoh_attention_plan_size", _abi.NAMOH_ERR_INVALID_ARG)
    if plan is None or plan.numel() < nbytes:
        plan = torch.empty(nbytes, dtype=torch.uint8, device=seg_offsets.device)
    rc = lib.namoh_attention_plan(_ptr(seg_offsets), B, T, H, K, group, _ptr(seg_cap), _ptr(plan), plan.numel(),
                                  _stream(stream))
    _abi.check("namoh_attention_plan", rc)
    return plan


def namoh_attention(q_rot: torch.Tensor, k_cache: torch.Tensor, v_cache: torch.Tensor, seg_offsets: torch.Tensor,
                    row_src: torch.Tensor, gate: torch.Tensor, plan: torch.Tensor, *, B: int, T: int, H: int, K: int,
                    group: int = 1, seg_base: Optional[torch.Tensor] = None, y: Optional[torch.Tensor] = None,
                    status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Prefill stage 3: routed causal attention + gate-weighted combine.  Returns y [B, T, K, d]."""
    lib = _abi.load()
    d = q_rot.shape[-1]
    dev = q_rot.device
    if y is None:
        y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    st = _status(status, dev)
    rc = lib.namoh_attention(_ptr(q_rot), _ptr(k_cache), _ptr(v_cache), B, T, H, K, d, group, _ptr(seg_offsets),
                             _ptr(row_src), _ptr(gate), _ptr(seg_base), k_cache.shape[0], _ptr(plan), plan.numel(),
                             _ptr(y), _ptr(st), _stream(stream))
    _abi.check("namoh_attention", rc)
    return y


def namoh_attention_timeout_probe(q_rot: torch.Tensor, k_cache: torch.Tensor, v_cache: torch.Tensor,
                                  seg_offsets: torch.Tensor, row_src: torch.Tensor, gate: torch.Tensor,
                                  plan: torch.Tensor, *, B: int, T: int, H: int, K: int, group: int = 1,
                                  wait_limit_ns: int = 1_000_000, y: Optional[torch.Tensor] = None,
                                  status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Check of the bounded waits (see namoh_attention_timeout_probe in include/namoh.h): namoh_attention
    with every CTA's first query tile withheld, so that the MMA issuer's wait runs out after wait_limit_ns
    and NAMOH_DEV_TIMEOUT is reported.  Returns the status tensor."""
    lib = _abi.load()
    d = q_rot.shape[-1]
    dev = q_rot.device
    if y is None:
        y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    st = _status(status, dev)
    rc = lib.namoh_attention_timeout_probe(_ptr(q_rot), _ptr(k_cache), _ptr(v_cache), B, T, H, K, d, group,
                                           _ptr(seg_offsets), _ptr(row_src), _ptr(gate), _ptr(plan), plan.numel(),
                                           _ptr(y), int(wait_limit_ns), _ptr(st), _stream(stream))
    _abi.check("namoh_attention_timeout_probe", rc)
    return st


def namoh_shared_prefill(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, *, window: int = 0,
                         rope_base: float = 10000.0, interleaved: bool = False, y: Optional[torch.Tensor] = None,
                         k_cache: Optional[torch.Tensor] = None, v_cache: Optional[torch.Tensor] = None,
                         seg_base: Optional[torch.Tensor] = None, seg_cap: Optional[torch.Tensor] = None,
                         seg_len: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
                         status: Optional[torch.Tensor] = None, stream=None):
    """Shared heads (see namoh_shared_prefill in include/namoh.h): q, k, v [B, Hs, T, d] bf16;
    window 0 = full causal prefix.  Returns (y [B, T, Hs, d], k_cache, v_cache)."""
    lib = _abi.load()
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16 or t.dim() != 4:
            raise ValueError(f"{name} must be a [B, Hs, T, d] bfloat16 tensor")
    B, Hs, T, d = q.shape
    dev = q.device
    if y is None:
        y = torch.empty((B, T, Hs, d), dtype=torch.bfloat16, device=dev)
    if k_cache is None:
        k_cache = torch.empty((B * Hs * T, d), dtype=torch.bfloat16, device=dev)
    if v_cache is None:
        v_cache = v if seg_base is None else torch.empty_like(k_cache)
    nbytes = lib.namoh_shared_workspace_size(B, T, Hs, d)
    if nbytes == 0:
        raise NamohError("namoh_shared_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    cache_rows = k_cache.numel() // d
    rc = lib.namoh_shared_prefill(_ptr(q), _ptr(k), _ptr(v), B, T, Hs, d, int(window), float(rope_base),
                                  _rope_flags(interleaved, False), _ptr(y), _ptr(k_cache), _ptr(v_cache),
                                  _ptr(seg_base), _ptr(seg_cap), cache_rows, _ptr(seg_len), _ptr(ws), ws.numel(),
                                  _ptr(st), _stream(stream))
    _abi.check("namoh_shared_prefill", rc)
    return y, k_cache, v_cache


def namoh_shared_decode(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, *, k_cache: torch.Tensor,
                        v_cache: torch.Tensor, seg_base: torch.Tensor, seg_len: torch.Tensor, seg_cap: torch.Tensor,
                        window: int = 0, rope_base: float = 10000.0, interleaved: bool = False,
                        y: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
                        status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """One decode step of the shared heads: q, k, v [B, Hs, d] bf16.  Returns y [B, Hs, d]."""
    lib = _abi.load()
    B, Hs, d = q.shape
    dev = q.device
    if y is None:
        y = torch.empty((B, Hs, d), dtype=torch.bfloat16, device=dev)
    nbytes = lib.namoh_shared_decode_workspace_size(B, Hs, d)
    if nbytes == 0:
        raise NamohError("namoh_shared_decode_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    rc = lib.namoh_shared_decode(_ptr(q), _ptr(k), _ptr(v), B, Hs, d, int(window), float(rope_base),
                                 _rope_flags(interleaved, False), _ptr(k_cache), _ptr(v_cache), _ptr(seg_base),
                                 _ptr(seg_len), _ptr(seg_cap), k_cache.shape[0], _ptr(y), _ptr(ws), ws.numel(),
                                 _ptr(st), _stream(stream))
    _abi.check("namoh_shared_decode", rc)
    return y


def namoh_proj_qkv(x: torch.Tensor, w_qkv: torch.Tensor, seg_offsets: torch.Tensor, row_src: torch.Tensor, *,
                   B: int, H: int, K: int, group: int = 1, q: Optional[torch.Tensor] = None,
                   k: Optional[torch.Tensor] = None, v: Optional[torch.Tensor] = None,
                   workspace: Optional[Workspace] = None, status: Optional[torch.Tensor] = None, stream=None):
    """Eq. (namoh-qkv) for the active pairs only (see namoh_proj_qkv in include/namoh.h).

    x [N, d_model], w_qkv [Hr, (g+2) d, d_model] bf16; returns packed q [R*g, d], k [R, d],
    v [R, d] (R = N*K/g), ready for namoh_prefill."""
    lib = _abi.load()
    if x.dtype != torch.bfloat16 or w_qkv.dtype != torch.bfloat16 or w_qkv.dim() != 3:
        raise ValueError("x and w_qkv must be bfloat16; w_qkv [Hr, (g+2) d, d_model]")
    N, d_model = x.shape
    Hr, ncols, wd = w_qkv.shape
    d = ncols // (group + 2)
    if Hr != H // group or ncols != (group + 2) * d or wd != d_model:
        raise ValueError("w_qkv must be [H/g, (g+2) d_head, d_model]")
    R = N * (K // group)
    dev = x.device
    q = torch.empty((R * group, d), dtype=torch.bfloat16, device=dev) if q is None else q
    k = torch.empty((R, d), dtype=torch.bfloat16, device=dev) if k is None else k
    v = torch.empty((R, d), dtype=torch.bfloat16, device=dev) if v is None else v
    ws = _ws(workspace, lib.namoh_proj_workspace_size(B, N, d_model, H, K, group), dev)
    st = _status(status, dev)
    rc = lib.namoh_proj_qkv(_ptr(x), N, d_model, _ptr(w_qkv), B, H, K, d, group, _ptr(seg_offsets), _ptr(row_src),
                            _ptr(q), _ptr(k), _ptr(v), _ptr(ws), ws.numel(), _ptr(st), _stream(stream))
    _abi.check("namoh_proj_qkv", rc)
    return q, k, v


def namoh_proj_out(y: torch.Tensor, w_o: torch.Tensor, seg_offsets: torch.Tensor, row_src: torch.Tensor, *,
                   B: int, H: int, K: int, group: int = 1, o: Optional[torch.Tensor] = None,
                   accumulate: bool = False, workspace: Optional[Workspace] = None,
                   status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """o_t = sum over the token's slots of y W_O (see namoh_proj_out in include/namoh.h).

    y [N, K, d] bf16 (namoh_prefill's output), w_o [Hr, d_model, g d] bf16; returns o [N, d_model]
    fp32 (added onto ``o`` when accumulate)."""
    lib = _abi.load()
    if y.dtype != torch.bfloat16 or w_o.dtype != torch.bfloat16 or w_o.dim() != 3:
        raise ValueError("y and w_o must be bfloat16; w_o [Hr, d_model, g d]")
    d = y.shape[-1]
    N = y.numel() // (K * d)  # y is [N, K, d] or [B, T, K, d]
    Hr, d_model, gd = w_o.shape
    if Hr != H // group or gd != group * d:
        raise ValueError("w_o must be [H/g, d_model, g d_head]")
    dev = y.device
    if o is None:
        o = torch.empty((N, d_model), dtype=torch.float32, device=dev)
        accumulate = False
    ws = _ws(workspace, lib.namoh_proj_workspace_size(B, N, d_model, H, K, group), dev)
    st = _status(status, dev)
    rc = lib.namoh_proj_out(_ptr(y), N, d_model, _ptr(w_o), B, H, K, d, group, _ptr(seg_offsets), _ptr(row_src),
                            _ptr(o), 1 if accumulate else 0, _ptr(ws), ws.numel(), _ptr(st), _stream(stream))
    _abi.check("namoh_proj_out", rc)
    return o


def namoh_decode(topk_head: torch.Tensor, gate: torch.Tensor, q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, *,
                 H: int, K: int, group: int = 1, rope_base: float = 10000.0, interleaved: bool = False,
                 token_pos: Optional[torch.Tensor] = None, k_cache: torch.Tensor,
                 v_cache: torch.Tensor, seg_base: torch.Tensor, seg_len: torch.Tensor, seg_cap: torch.Tensor,
                 y: Optional[torch.Tensor] = None, workspace: Optional[Workspace] = None,
                 status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """One decode step (see namoh_decode in include/namoh.h).  Returns y [B, K, d] bf16.

    token_pos (int64 [B], the new tokens' indices) selects global positions (NAMOH_ROPE_GLOBAL);
    interleaved the (2j, 2j+1) pairing."""
    lib = _abi.load()
    B = topk_head.shape[0]
    d = q.shape[-1]
    dev = q.device
    if y is None:
        y = torch.empty((B, K, d), dtype=torch.bfloat16, device=dev)
    nbytes = lib.namoh_decode_workspace_size(B, H, K, d, group)
    if nbytes == 0:
        raise NamohError("namoh_decode_workspace_size", _abi.NAMOH_ERR_UNSUPPORTED)
    ws = _ws(workspace, nbytes, dev)
    st = _status(status, dev)
    if token_pos is not None and (token_pos.dtype != torch.int64 or token_pos.numel() != B):
        raise ValueError("token_pos must be int64 with one entry per sequence")
    rc = lib.namoh_decode_ex(_ptr(topk_head), _ptr(gate), _ptr(q), _ptr(k), _ptr(v), B, H, K, d, group,
                             float(rope_base), _rope_flags(interleaved, token_pos is not None), _ptr(token_pos),
                             _ptr(k_cache), _ptr(v_cache), _ptr(seg_base), _ptr(seg_len), _ptr(seg_cap),
                             k_cache.shape[0], _ptr(y), _ptr(ws), ws.numel(), _ptr(st), _stream(stream))
    _abi.check("namoh_decode_ex", rc)
    return y
