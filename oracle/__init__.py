"""fp64 CPU oracle for the NAMOH routed-attention path.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The CUDA library never
imports, links or executes anything here, and this package imports nothing from
the CUDA library: the two share only the seeded input generators in
``namoh_inputs``.

The arithmetic lives in ``namoh_oracle.c`` (plain C, fp64, built with gcc); this
module only marshals numpy arrays.  Each wrapper names the passage of the paper
it follows:

* ``route``        Sec. 3.1 Eq. (namoh-gates) and the ordered index sets I_i;
                   Sec. 3.2 Eq. (namoh-head-rope) for the rank rho.
* ``rope``         Sec. 3.2 Eq. (namoh-head-rope), half-split RoPE.
* ``prefill``      Sec. 3.1 Eq. (namoh-attention) over packed (batch, head)
                   subsequences (Sec. 3.2 "Efficient execution"); App. B.7
                   "Adopted KV-group routing" for g > 1.
* ``prefill_rows`` the same for a chosen subset of query rows.
* ``decode_step``  Sec. 3.1 (last paragraph): append to and attend within only
                   the selected heads' histories.
* ``sa_prefill``   App. B.8 "SA+NAMOH" with the block-selection model of App. B.3
                   (Eqs. app-block-budget, app-selected-entries): blocks of the routed
                   history in local order, the current block plus the highest-scoring
                   completed blocks against their mean-pooled keys.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "namoh_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK = 0
ERR_ARG = -1
ERR_NONFINITE = -2
ERR_NOMEM = -3
ERR_CAPACITY = -4


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc (fp64, no fast-math, no FMA contraction)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-D_POSIX_C_SOURCE=200809L", "-ffp-contract=off",
               "-fPIC", "-shared", "-pthread", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        P = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int, ctypes.c_long, ctypes.c_double
        lib.oracle_route_topk.argtypes = [P, i64, i32, i32, P, P]
        lib.oracle_route_biased.argtypes = [P, P, i64, i32, i32, P, P, P]
        lib.oracle_dispatch.argtypes = [P, i32, i32, i32, i32, P, P, P, P, P]
        lib.oracle_dispatch_varlen.argtypes = [P, P, i32, i32, i32, P, P, P, P, P]
        lib.oracle_rope.argtypes = [P, i64, i32, i64, P, f64, i32, P]
        lib.oracle_prefill.argtypes = [P, P, P, i32, i32, i32, f64, P, P, P, P, P, i32, i32, P]
        lib.oracle_prefill_rows.argtypes = [P, P, P, i32, i32, i32, f64, P, P, P, P, P, i64, P, i32, P]
        lib.oracle_decode_step.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, f64,
                                           P, P, P, P, P, P, i32, P, i32]
        lib.oracle_shared_prefill.argtypes = [P, P, P, i32, i32, i32, i32, i32, f64, i32, P, i32]
        lib.oracle_proj_qkv.argtypes = [P, i32, P, i32, i32, i32, i32, P, i32, P, P, P, P, i32]
        lib.oracle_proj_out.argtypes = [P, P, i64, i32, i32, i32, P, i32, i32, P, i32]
        lib.oracle_sa_prefill.argtypes = [P, P, P, i32, i32, i32, f64, P, P, P, i32, i64, i64, P, P, i32, P,
                                          i32, i32, P]
        lib.oracle_sa_scores_rows.argtypes = [P, P, i32, i32, i32, f64, P, i32, P, P, i64, i32, P, i32, P]
        lib.oracle_default_threads.argtypes = []
        for fn in ("oracle_route_topk", "oracle_route_biased", "oracle_dispatch", "oracle_dispatch_varlen",
                   "oracle_rope", "oracle_prefill",
                   "oracle_prefill_rows", "oracle_decode_step", "oracle_proj_qkv", "oracle_proj_out",
                   "oracle_shared_prefill",
                   "oracle_default_threads"):
            getattr(lib, fn).restype = ctypes.c_int
        _lib = lib
        return lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(rc: int, what: str):
    if rc != OK:
        raise OracleError(f"{what} failed with oracle status {rc}")


def default_threads() -> int:
    return int(_load().oracle_default_threads())


def route(scores: np.ndarray, K: int) -> dict:
    """Routing and dispatch for scores [B, T, H] (fp32 router logits).

    Returns topk_head [B,T,K] int32, gate [B,T,K] fp64, n [B,H], seg_offsets [B*H+1],
    rank [B,T,K], row [B,T,K] and row_src [B*T*K] (all int32).
    """
    lib = _load()
    scores = np.ascontiguousarray(scores, dtype=np.float32)
    B, T, H = scores.shape
    topk = np.empty((B, T, K), np.int32)
    gate = np.empty((B, T, K), np.float64)
    _check(lib.oracle_route_topk(_ptr(scores), B * T, H, K, _ptr(topk), _ptr(gate)), "route_topk")
    n = np.empty((B, H), np.int32)
    seg = np.empty(B * H + 1, np.int32)
    rank = np.empty((B, T, K), np.int32)
    row = np.empty((B, T, K), np.int32)
    row_src = np.empty(B * T * K, np.int32)
    _check(lib.oracle_dispatch(_ptr(topk), B, T, H, K, _ptr(n), _ptr(seg), _ptr(rank), _ptr(row),
                               _ptr(row_src)), "dispatch")
    return dict(topk_head=topk, gate=gate, n=n, seg_offsets=seg, rank=rank, row=row, row_src=row_src)


def dispatch(topk_head: np.ndarray, H: int) -> dict:
    """Dispatch (Sec. 3.1 index sets, Sec. 3.2 ranks and packing) of given picks topk_head [B, T, K]."""
    lib = _load()
    topk = np.ascontiguousarray(topk_head, dtype=np.int32)
    B, T, K = topk.shape
    n = np.empty((B, H), np.int32)
    seg = np.empty(B * H + 1, np.int32)
    rank = np.empty((B, T, K), np.int32)
    row = np.empty((B, T, K), np.int32)
    row_src = np.empty(B * T * K, np.int32)
    _check(lib.oracle_dispatch(_ptr(topk), B, T, H, K, _ptr(n), _ptr(seg), _ptr(rank), _ptr(row),
                               _ptr(row_src)), "dispatch")
    return dict(n=n, seg_offsets=seg, rank=rank, row=row, row_src=row_src)


def route_varlen(scores: np.ndarray, cu_seqlens: np.ndarray, K: int, bias: np.ndarray | None = None) -> dict:
    """Routing and dispatch of a ragged batch: scores [N, H] over the flat token axis, sequence
    b = tokens cu_seqlens[b] .. cu_seqlens[b+1]-1.  Biased selection when bias [H] is given.

    Returns topk_head [N,K], gate [N,K] fp64, n [B,H], seg_offsets [B*H+1], rank [N,K],
    row [N,K] and row_src [N*K] (row_src[row] = tok*K + slot).
    """
    lib = _load()
    scores = np.ascontiguousarray(scores, dtype=np.float32)
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    N, H = scores.shape
    B = len(cu) - 1
    if B < 0 or cu[0] != 0 or cu[-1] != N or np.any(np.diff(cu) < 0):
        raise OracleError("cu_seqlens must start at 0, not decrease and end at N")
    topk = np.empty((N, K), np.int32)
    gate = np.empty((N, K), np.float64)
    if bias is None:
        _check(lib.oracle_route_topk(_ptr(scores), N, H, K, _ptr(topk), _ptr(gate)), "route_topk")
    else:
        bias = np.ascontiguousarray(bias, dtype=np.float32)
        key = np.empty((N, H), np.float64)
        _check(lib.oracle_route_biased(_ptr(scores), _ptr(bias), N, H, K, _ptr(topk), _ptr(gate), _ptr(key)),
               "route_biased")
    n = np.empty((B, H), np.int32)
    seg = np.empty(B * H + 1, np.int32)
    rank = np.empty((N, K), np.int32)
    row = np.empty((N, K), np.int32)
    row_src = np.empty(N * K, np.int32)
    _check(lib.oracle_dispatch_varlen(_ptr(topk), _ptr(cu), B, H, K, _ptr(n), _ptr(seg), _ptr(rank), _ptr(row),
                                      _ptr(row_src)), "dispatch_varlen")
    return dict(topk_head=topk, gate=gate, n=n, seg_offsets=seg, rank=rank, row=row, row_src=row_src)


def route_biased(scores: np.ndarray, K: int, bias: np.ndarray) -> dict:
    """Biased routing (App. A, Eq. namoh-biased-routing) and dispatch for scores [B, T, H].

    As route(), plus key [B, T, H] = a + b in fp64, the quantity the selection ranks.
    """
    lib = _load()
    scores = np.ascontiguousarray(scores, dtype=np.float32)
    bias = np.ascontiguousarray(bias, dtype=np.float32)
    B, T, H = scores.shape
    if bias.shape != (H,):
        raise ValueError("bias must have shape [H]")
    topk = np.empty((B, T, K), np.int32)
    gate = np.empty((B, T, K), np.float64)
    key = np.empty((B, T, H), np.float64)
    _check(lib.oracle_route_biased(_ptr(scores), _ptr(bias), B * T, H, K, _ptr(topk), _ptr(gate), _ptr(key)),
           "route_biased")
    out = dispatch(topk, H)
    out.update(topk_head=topk, gate=gate, key=key)
    return out


def rope(x_bits: np.ndarray, pos: np.ndarray, base: float, interleaved: bool = False) -> np.ndarray:
    """Rotate bf16 rows x [rows, d] (raw uint16 bits) to positions pos [rows]; fp64 out.

    Pairs (j, j + d/2) by default, (2j, 2j+1) with interleaved."""
    lib = _load()
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    rows, d = x_bits.shape
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    out = np.empty((rows, d), np.float64)
    _check(lib.oracle_rope(_ptr(x_bits), rows, d, d, _ptr(pos), float(base), int(bool(interleaved)), _ptr(out)),
           "rope")
    return out


def global_positions(row_src: np.ndarray, T: int, K: int) -> np.ndarray:
    """Position of each packed row under global RoPE: the token's index t in its sequence
    (row_src[r] = (b*T + t)*K + slot)."""
    rs = np.asarray(row_src, dtype=np.int64)
    return np.ascontiguousarray((rs // K) % T, dtype=np.int64)


def dispatch_varlen(topk_head: np.ndarray, cu_seqlens: np.ndarray, H: int) -> dict:
    """Dispatch of given picks topk_head [N, K] over a ragged batch (oracle_dispatch_varlen)."""
    lib = _load()
    topk = np.ascontiguousarray(topk_head, dtype=np.int32)
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    N, K = topk.shape
    B = len(cu) - 1
    if cu[0] != 0 or cu[-1] != N or np.any(np.diff(cu) < 0):
        raise OracleError("cu_seqlens must start at 0, not decrease and end at N")
    n = np.empty((B, H), np.int32)
    seg = np.empty(B * H + 1, np.int32)
    rank = np.empty((N, K), np.int32)
    row = np.empty((N, K), np.int32)
    row_src = np.empty(N * K, np.int32)
    _check(lib.oracle_dispatch_varlen(_ptr(topk), _ptr(cu), B, H, K, _ptr(n), _ptr(seg), _ptr(rank), _ptr(row),
                                      _ptr(row_src)), "dispatch_varlen")
    return dict(n=n, seg_offsets=seg, rank=rank, row=row, row_src=row_src)


def global_positions_varlen(row_src: np.ndarray, cu_seqlens: np.ndarray, K: int) -> np.ndarray:
    """Global RoPE positions in a ragged batch: the token's index inside its own sequence."""
    tok = np.asarray(row_src, dtype=np.int64) // K
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    b = np.searchsorted(cu, tok, side="right") - 1
    return np.ascontiguousarray(tok - cu[b], dtype=np.int64)


def prefill(q: np.ndarray, k: np.ndarray, v: np.ndarray, seg_offsets: np.ndarray, row_src: np.ndarray,
            gate: np.ndarray, d: int, g: int, base: float, nthreads: int | None = None,
            return_krot: bool = False, interleaved: bool = False, pos: np.ndarray | None = None):
    """Prefill over packed rows.  q [R*g, d], k/v [R, d] as bf16 bits; gate indexed by row_src.

    Returns y [R*g, d] fp64 laid out by (row_src * g + j), i.e. [B, T, K, g, d] flattened.
    RoPE positions are the ranks, or pos [R] (e.g. global_positions) when given.
    """
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    seg = np.ascontiguousarray(seg_offsets, dtype=np.int32)
    rs = np.ascontiguousarray(row_src, dtype=np.int32)
    gt = np.ascontiguousarray(gate, dtype=np.float64).reshape(-1)
    R = int(seg[-1])
    y = np.zeros((R * g, d), np.float64)
    krot = np.empty((R, d), np.float64) if return_krot else None
    nthreads = default_threads() if nthreads is None else int(nthreads)
    pos = None if pos is None else np.ascontiguousarray(pos, dtype=np.int64)
    if pos is not None and pos.shape != (R,):
        raise OracleError("pos must hold one position per packed row")
    rc = lib.oracle_prefill(_ptr(q), _ptr(k), _ptr(v), len(seg) - 1, d, g, float(base), _ptr(seg), _ptr(rs),
                            _ptr(gt), _ptr(y), _ptr(krot) if krot is not None else None, nthreads,
                            int(bool(interleaved)), _ptr(pos) if pos is not None else None)
    _check(rc, "prefill")
    return (y, krot) if return_krot else y


def prefill_rows(q, k, v, seg_offsets, row_src, gate, d: int, g: int, base: float,
                 rows: np.ndarray, heads: np.ndarray, interleaved: bool = False,
                 pos: np.ndarray | None = None) -> np.ndarray:
    """Outputs g*h for the listed (packed row, group head) queries only: [len(rows), d] fp64."""
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    seg = np.ascontiguousarray(seg_offsets, dtype=np.int32)
    rs = np.ascontiguousarray(row_src, dtype=np.int32)
    gt = np.ascontiguousarray(gate, dtype=np.float64).reshape(-1)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    heads = np.ascontiguousarray(heads, dtype=np.int32)
    out = np.empty((len(rows), d), np.float64)
    pos = None if pos is None else np.ascontiguousarray(pos, dtype=np.int64)
    if pos is not None and pos.shape != (int(seg[-1]),):
        raise OracleError("pos must hold one position per packed row")
    rc = lib.oracle_prefill_rows(_ptr(q), _ptr(k), _ptr(v), len(seg) - 1, d, g, float(base), _ptr(seg),
                                 _ptr(rs), _ptr(gt), _ptr(rows), _ptr(heads), len(rows), _ptr(out),
                                 int(bool(interleaved)), _ptr(pos) if pos is not None else None)
    _check(rc, "prefill_rows")
    return out


def decode_step(topk_head, gate, q, k, v, Hr: int, d: int, g: int, base: float,
                k_cache: np.ndarray, v_cache: np.ndarray, seg_base: np.ndarray, seg_len: np.ndarray,
                seg_cap: np.ndarray, interleaved: bool = False, token_pos: np.ndarray | None = None,
                window: int = 0) -> np.ndarray:
    """One decode step.  k_cache/v_cache [cap_total, d] fp64 and seg_len are updated in place.

    topk_head/gate [B, Kr]; q [B, Kr*g, d], k/v [B, Kr, d] as bf16 bits.  Returns y [B, Kr*g, d].
    RoPE positions are the ranks, or token_pos [B] (the new tokens' indices) when given.
    window > 0 attends over the last `window` rows only (the new one included).
    """
    lib = _load()
    topk_head = np.ascontiguousarray(topk_head, dtype=np.int32)
    B, Kr = topk_head.shape
    gate = np.ascontiguousarray(gate, dtype=np.float64)
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    for name, arr, dt in (("k_cache", k_cache, np.float64), ("v_cache", v_cache, np.float64),
                          ("seg_base", seg_base, np.int64), ("seg_len", seg_len, np.int32),
                          ("seg_cap", seg_cap, np.int32)):
        if arr.dtype != dt or not arr.flags.c_contiguous:
            raise OracleError(f"{name} must be a contiguous {np.dtype(dt).name} array")
    y = np.zeros((B, Kr * g, d), np.float64)
    token_pos = None if token_pos is None else np.ascontiguousarray(token_pos, dtype=np.int64)
    rc = lib.oracle_decode_step(_ptr(topk_head), _ptr(gate), _ptr(q), _ptr(k), _ptr(v), B, Hr, Kr, d, g,
                                float(base), _ptr(k_cache), _ptr(v_cache), _ptr(seg_base), _ptr(seg_len),
                                _ptr(seg_cap), _ptr(y), int(bool(interleaved)),
                                _ptr(token_pos) if token_pos is not None else None, int(window))
    _check(rc, "decode_step")
    return y


def proj_qkv(x, w_qkv, seg_offsets, row_src, Hr: int, Kr: int, g: int, d: int, nthreads: int | None = None):
    """Eq. (namoh-qkv) in the packed layout: x [N, d_model] and w_qkv [Hr, (g+2) d, d_model] as
    bf16 bits.  Returns fp64 q [R g, d], k [R, d], v [R, d]."""
    lib = _load()
    x = np.ascontiguousarray(x, dtype=np.uint16)
    w = np.ascontiguousarray(w_qkv, dtype=np.uint16)
    seg = np.ascontiguousarray(seg_offsets, dtype=np.int32)
    rs = np.ascontiguousarray(row_src, dtype=np.int32)
    d_model = x.shape[1]
    if w.shape != (Hr, (g + 2) * d, d_model):
        raise OracleError("w_qkv must be [Hr, (g+2) d, d_model]")
    R = int(seg[-1])
    q = np.empty((R * g, d)); k = np.empty((R, d)); v = np.empty((R, d))
    nthreads = default_threads() if nthreads is None else int(nthreads)
    _check(lib.oracle_proj_qkv(_ptr(x), d_model, _ptr(w), Hr, Kr, g, d, _ptr(seg), len(seg) - 1, _ptr(rs), _ptr(q),
                               _ptr(k), _ptr(v), nthreads), "proj_qkv")
    return q, k, v


def proj_out(y, topk_head, w_o, g: int, d: int, nthreads: int | None = None):
    """Eq. (namoh-attention) output projection: y [N, Kr, g, d] (fp64 per-slot g h), topk_head
    [N, Kr], w_o [Hr, d_model, g d] bf16 bits.  Returns o [N, d_model] fp64."""
    lib = _load()
    topk = np.ascontiguousarray(topk_head, dtype=np.int32)
    N, Kr = topk.shape
    y = np.ascontiguousarray(y, dtype=np.float64).reshape(N, Kr, g * d)
    w = np.ascontiguousarray(w_o, dtype=np.uint16)
    Hr, d_model, gd = w.shape
    if gd != g * d:
        raise OracleError("w_o must be [Hr, d_model, g d]")
    o = np.empty((N, d_model))
    nthreads = default_threads() if nthreads is None else int(nthreads)
    _check(lib.oracle_proj_out(_ptr(y), _ptr(topk), N, Kr, g, d, _ptr(w), Hr, d_model, _ptr(o), nthreads),
           "proj_out")
    return o


def shared_prefill(q, k, v, window: int, base: float, interleaved: bool = False, nthreads: int | None = None):
    """Shared heads (Sec. 4.4): q, k, v [B, Hs, T, d] bf16 bits; full causal (window 0) or sliding
    window attention at global positions, no gate.  Returns y [B, T, Hs, d] fp64."""
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    B, Hs, T, d = q.shape
    y = np.empty((B, T, Hs, d))
    nthreads = default_threads() if nthreads is None else int(nthreads)
    _check(lib.oracle_shared_prefill(_ptr(q), _ptr(k), _ptr(v), B, Hs, T, d, int(window), float(base),
                                     int(bool(interleaved)), _ptr(y), nthreads), "shared_prefill")
    return y


def shared_decode_step(q, k, v, d: int, base: float, k_cache, v_cache, seg_base, seg_len, seg_cap, window: int):
    """One decode step of the shared heads: q, k, v [B, Hs, d] bf16 bits, every head active with
    gate 1 (decode_step with all heads selected).  Returns y [B, Hs, d] fp64."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    B, Hs = q.shape[0], q.shape[1]
    top = np.tile(np.arange(Hs, dtype=np.int32), (B, 1))
    return decode_step(top, np.ones((B, Hs)), q, k, v, Hs, d, 1, base, k_cache, v_cache, seg_base, seg_len,
                       seg_cap, window=window)


def sa_mask_words(n_max: int, block: int) -> int:
    """32-bit words per query of a kept-block mask for histories of at most n_max entries."""
    nblk = -(-int(n_max) // int(block))
    return max(1, -(-nblk // 32))


def sa_prefill(q, k, v, seg_offsets, row_src, gate, d: int, g: int, base: float, block: int,
               alpha_num: int, alpha_den: int, mask_in: np.ndarray | None = None, want_mask: bool = False,
               nthreads: int | None = None, interleaved: bool = False, pos: np.ndarray | None = None):
    """SA + NAMOH prefill over packed rows (App. B.8, selection model of App. B.3).

    alpha = alpha_num / alpha_den.  mask_in [R*g, W] uint32 (W >= sa_mask_words of the longest
    history) replaces the selection; want_mask also returns the blocks kept.  Returns y [R*g, d] fp64 (and the mask).
    """
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    seg = np.ascontiguousarray(seg_offsets, dtype=np.int32)
    rs = np.ascontiguousarray(row_src, dtype=np.int32)
    gt = np.ascontiguousarray(gate, dtype=np.float64).reshape(-1)
    R = int(seg[-1])
    n_max = int(np.max(np.diff(seg))) if len(seg) > 1 else 0
    W = sa_mask_words(n_max, block)
    if mask_in is not None:  # any width that holds the longest history's blocks
        mask_in = np.ascontiguousarray(mask_in, dtype=np.uint32)
        if mask_in.ndim != 2 or mask_in.shape[0] != R * g or mask_in.shape[1] < W:
            raise OracleError(f"mask_in must be [{R * g}, >= {W}]")
        W = mask_in.shape[1]
    mask_out = np.zeros((R * g, W), np.uint32) if want_mask else None
    y = np.zeros((R * g, d), np.float64)
    pos = None if pos is None else np.ascontiguousarray(pos, dtype=np.int64)
    nthreads = default_threads() if nthreads is None else int(nthreads)
    rc = lib.oracle_sa_prefill(_ptr(q), _ptr(k), _ptr(v), len(seg) - 1, d, g, float(base), _ptr(seg), _ptr(rs),
                               _ptr(gt), int(block), int(alpha_num), int(alpha_den),
                               _ptr(mask_in) if mask_in is not None else None,
                               _ptr(mask_out) if mask_out is not None else None, W, _ptr(y), nthreads,
                               int(bool(interleaved)), _ptr(pos) if pos is not None else None)
    _check(rc, "sa_prefill")
    return (y, mask_out) if want_mask else y


def sa_scores_rows(q, k, seg_offsets, d: int, g: int, base: float, block: int, rows, heads, nblk: int,
                   interleaved: bool = False, pos: np.ndarray | None = None) -> np.ndarray:
    """fp64 scores of the completed blocks (before the current one) for chosen queries: [len(rows), nblk],
    NaN where a block is not a completed block of that query's history."""
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    seg = np.ascontiguousarray(seg_offsets, dtype=np.int32)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    heads = np.ascontiguousarray(heads, dtype=np.int32)
    out = np.empty((len(rows), int(nblk)), np.float64)
    pos = None if pos is None else np.ascontiguousarray(pos, dtype=np.int64)
    rc = lib.oracle_sa_scores_rows(_ptr(q), _ptr(k), len(seg) - 1, d, g, float(base), _ptr(seg), int(block),
                                   _ptr(rows), _ptr(heads), len(rows), int(nblk), _ptr(out),
                                   int(bool(interleaved)), _ptr(pos) if pos is not None else None)
    _check(rc, "sa_scores_rows")
    return out
