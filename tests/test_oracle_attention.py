"""Pins of the oracle's RoPE, routed attention, combine and decode.

What the paper fixes, each checked by a formulation unlike the oracle's:
  * Sec. 3.2 Eq. (namoh-head-rope): R(p) is a rotation; RoPE written as complex
    multiplication; the dot product of rotated vectors depends only on p - s.
  * Sec. 3.2 (last sentence on RoPE) and Sec. 3.1: with K = H every rank equals t, so the
    method is dense causal MHA with standard RoPE -> torch scaled_dot_product_attention.
  * App. B (routing-induced attention structure): per-head weights alpha^{(i)}_{t,s}
    over the full T x T grid, zero outside routed causal pairs -> brute-force masks.
  * Sec. 3.1: each query attends only to earlier tokens (and itself) of the same head.
  * Sec. 3.1 (end): prefill and incremental decoding are the same causal computation.
  * App. B.5 Eq. (app-routed-kv): M_KV = T K after the prefix, + K per decode step.
  * App. B.7 "Adopted KV-group routing": g query heads share a group's keys, values,
    gate and rank.
  * Sec. 3.2 (end of "Head-relative positional encoding"): global RoPE replaces rho_i(t) by t
    -> the brute-force masks with t as the position, and prefill == decode at token index t.
  * Interleaved pairing (2j, 2j+1) is RoPE as complex multiplication on adjacent pairs, i.e.
    half-split RoPE conjugated by the pair permutation.
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni


def _widen(bits):
    return ni.bf16_to_f32(bits).astype(np.float64)


def _rope_complex(x, pos, base, interleaved=False):
    """RoPE as complex multiplication: (x_j + i x_{j+d/2}) * exp(i * pos * base^(-2j/d)),
    or (x_{2j} + i x_{2j+1}) for the interleaved pairing."""
    d = x.shape[-1]
    half = d // 2
    z = x[..., 0::2] + 1j * x[..., 1::2] if interleaved else x[..., :half] + 1j * x[..., half:]
    freq = np.exp(-np.log(base) * (2.0 * np.arange(half) / d))
    rot = z * np.exp(1j * np.asarray(pos, np.float64)[..., None] * freq)
    if interleaved:
        out = np.empty(rot.shape[:-1] + (d,))
        out[..., 0::2] = rot.real
        out[..., 1::2] = rot.imag
        return out
    return np.concatenate([rot.real, rot.imag], axis=-1)


def _topk_counting(s, K):
    H = s.shape[-1]
    pos = np.zeros(s.shape, np.int64)
    for h in range(H):
        pos[..., h] = (s > s[..., h:h + 1]).sum(-1) + (s[..., :h] == s[..., h:h + 1]).sum(-1)
    top = np.zeros(s.shape[:-1] + (K,), np.int64)
    for h in range(H):
        idx = np.nonzero(pos[..., h] < K)
        top[idx + (pos[..., h][idx],)] = h
    return top


def _softmax64(s):
    s = s.astype(np.float64)
    e = np.exp(s - s.max(-1, keepdims=True))
    return e / e.sum(-1, keepdims=True)


def _pack(top, B, T, Hr):
    """Test-side packing: segment (b, h) rows in t order; returns seg_offsets, row [B,T,K], row_src."""
    K = top.shape[-1]
    mask = np.zeros((B, T, Hr), np.int64)
    np.put_along_axis(mask, top, 1, axis=-1)
    n = mask.sum(1).reshape(-1)
    seg = np.concatenate([[0], np.cumsum(n)]).astype(np.int32)
    rho = np.cumsum(mask, axis=1) - 1
    row = seg[np.arange(B)[:, None, None] * Hr + top] + np.take_along_axis(rho, top, axis=-1)
    row_src = np.empty(B * T * K, np.int32)
    row_src[row.reshape(-1)] = np.arange(B * T * K)
    return seg, row.astype(np.int64), row_src, mask, rho


# --------------------------------------------------------------------------- RoPE
@pytest.mark.parametrize("d,base", [(64, 1e4), (128, 5e5), (8, 10.0)])
@pytest.mark.parametrize("interleaved", [False, True])
def test_rope_is_complex_rotation(oracle_mod, d, base, interleaved):
    rng = np.random.default_rng(0)
    x = ni.bf16_bits(rng.standard_normal((50, d)).astype(np.float32))
    pos = rng.integers(0, 40000, 50)
    pos[0] = 0
    out = oracle_mod.rope(x, pos, base, interleaved)
    np.testing.assert_allclose(out, _rope_complex(_widen(x), pos, base, interleaved), rtol=0, atol=1e-9)
    np.testing.assert_array_equal(out[0], _widen(x[0]))  # R(0) = I
    np.testing.assert_allclose(np.linalg.norm(out, axis=-1), np.linalg.norm(_widen(x), axis=-1), rtol=1e-12)
    if interleaved:  # half-split RoPE conjugated by the pair permutation (2j, 2j+1) <-> (j, j + d/2)
        perm = np.concatenate([np.arange(0, d, 2), np.arange(1, d, 2)])
        half_split = oracle_mod.rope(x[:, perm], pos, base)
        np.testing.assert_array_equal(out[:, perm], half_split)


def test_rope_relative_property(oracle_mod):
    rng = np.random.default_rng(1)
    d = 64
    q = ni.bf16_bits(rng.standard_normal((20, d)).astype(np.float32))
    k = ni.bf16_bits(rng.standard_normal((20, d)).astype(np.float32))
    p = rng.integers(0, 3000, 20)
    s = rng.integers(0, 3000, 20)
    lhs = np.sum(oracle_mod.rope(q, p, 1e4) * oracle_mod.rope(k, s, 1e4), -1)
    rhs = np.sum(oracle_mod.rope(q, p - s, 1e4) * _widen(k), -1)
    np.testing.assert_allclose(lhs, rhs, rtol=0, atol=1e-9)


# --------------------------------------------------------------------------- reductions
def _dense_causal_mha(qf, kf, vf, base):
    """qf/kf/vf [B, T, H, d] fp64 -> h [B, T, H, d] by torch SDPA with global-position RoPE."""
    B, T, H, d = qf.shape
    pos = np.arange(T)[None, :, None]
    qr = _rope_complex(qf, np.broadcast_to(pos, (B, T, H)), base)
    kr = _rope_complex(kf, np.broadcast_to(pos, (B, T, H)), base)
    tq = torch.from_numpy(qr).permute(0, 2, 1, 3)
    tk = torch.from_numpy(kr).permute(0, 2, 1, 3)
    tv = torch.from_numpy(vf).permute(0, 2, 1, 3)
    h = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True)
    return h.permute(0, 2, 1, 3).numpy()


@pytest.mark.parametrize("B,T,H,d", [(2, 33, 4, 16), (1, 70, 3, 64)])
def test_k_equals_h_is_dense_causal_mha(oracle_mod, B, T, H, d):
    rng = np.random.default_rng(2)
    s = ni.router_scores(4, B, T, H)
    qb, kb, vb = (ni.bf16_bits(rng.standard_normal((B, T, H, d)).astype(np.float32)) for _ in range(3))
    top = _topk_counting(s, H)
    seg, row, row_src, _, rho = _pack(top, B, T, H)
    np.testing.assert_array_equal(rho, np.broadcast_to(np.arange(T)[None, :, None], rho.shape))
    Rn = B * T * H
    qp = np.empty((Rn, d), np.uint16); kp = np.empty_like(qp); vp = np.empty_like(qp)
    b_i, t_i, k_i = np.meshgrid(np.arange(B), np.arange(T), np.arange(H), indexing="ij")
    hsel = top[b_i, t_i, k_i]
    qp[row] = qb[b_i, t_i, hsel]; kp[row] = kb[b_i, t_i, hsel]; vp[row] = vb[b_i, t_i, hsel]
    gate = np.take_along_axis(_softmax64(s), top, -1)
    y = oracle_mod.prefill(qp, kp, vp, seg, row_src, gate.reshape(-1), d, 1, 1e4).reshape(B, T, H, d)
    h = _dense_causal_mha(_widen(qb), _widen(kb), _widen(vb), 1e4)
    expect = gate[..., None] * np.take_along_axis(h, top[..., None], axis=2)
    np.testing.assert_allclose(y, expect, rtol=0, atol=1e-11)
    # with K = H every rank is t, so global RoPE changes nothing
    yg = oracle_mod.prefill(qp, kp, vp, seg, row_src, gate.reshape(-1), d, 1, 1e4,
                            pos=oracle_mod.global_positions(row_src, T, H))
    np.testing.assert_array_equal(yg.reshape(B, T, H, d), y)


def test_single_head_k1_is_single_head_attention(oracle_mod):
    B, T, H, d = 1, 90, 6, 32
    rng = np.random.default_rng(3)
    s = np.full((B, T, H), -1.0, np.float32)
    s[..., 2] = 3.0  # every token routes to head 2
    qb, kb, vb = (ni.bf16_bits(rng.standard_normal((B * T, d)).astype(np.float32)) for _ in range(3))
    top = _topk_counting(s, 1)
    seg, row, row_src, _, _ = _pack(top, B, T, H)
    gate = np.take_along_axis(_softmax64(s), top, -1).reshape(-1)
    y = oracle_mod.prefill(qb, kb, vb, seg, row_src, gate, d, 1, 1e4)
    h = _dense_causal_mha(_widen(qb).reshape(B, T, 1, d), _widen(kb).reshape(B, T, 1, d),
                          _widen(vb).reshape(B, T, 1, d), 1e4)
    np.testing.assert_allclose(y, gate[:, None] * h.reshape(B * T, d), rtol=0, atol=1e-11)


# --------------------------------------------------------------------------- brute force
def _brute_force(qf, kf, vf, s, Kr, g, base, interleaved=False, global_pos=False):
    """Full T x T per-query-head attention with routing masks (App. B definitions).

    qf [B, T, Hr*g, d], kf/vf [B, T, Hr, d] fp64; s [B, T, Hr] logits.  Returns y [B, T, Kr, g, d].
    global_pos encodes token t at position t instead of its rank.
    """
    B, T, Hr = s.shape
    d = qf.shape[-1]
    top = _topk_counting(s, Kr)
    mask = np.zeros((B, T, Hr), np.int64)
    np.put_along_axis(mask, top, 1, axis=-1)
    rho = np.cumsum(mask, axis=1) - 1
    if global_pos:
        rho = np.broadcast_to(np.arange(T)[None, :, None], (B, T, Hr))
    a = _softmax64(s)
    y = np.zeros((B, T, Kr, g, d))
    causal = np.tril(np.ones((T, T), bool))
    for b in range(B):
        for i in range(Hr):
            kr = _rope_complex(kf[b, :, i], rho[b, :, i], base, interleaved)
            for j in range(g):
                qr = _rope_complex(qf[b, :, i * g + j], rho[b, :, i], base, interleaved)
                logits = qr @ kr.T / np.sqrt(d)
                allowed = causal & (mask[b, :, i][:, None] == 1) & (mask[b, :, i][None, :] == 1)
                for t in range(T):
                    if not mask[b, t, i]:
                        continue
                    w = np.where(allowed[t], np.exp(logits[t] - logits[t][allowed[t]].max()), 0.0)
                    alpha = w / w.sum()
                    slot = list(top[b, t]).index(i)
                    y[b, t, slot, j] = a[b, t, i] * (alpha @ vf[b, :, i])
    return y, top


@pytest.mark.parametrize("variant", ["rank", "interleaved", "global", "global_interleaved"])
@pytest.mark.parametrize("B,T,Hr,Kr,g,d", [(2, 24, 4, 2, 1, 8), (1, 40, 6, 3, 1, 16), (2, 20, 4, 2, 3, 8)])
def test_prefill_matches_brute_force_masks(oracle_mod, B, T, Hr, Kr, g, d, variant):
    rng = np.random.default_rng(4)
    s = ni.router_scores(6, B, T, Hr)
    qb = ni.bf16_bits(rng.standard_normal((B, T, Hr * g, d)).astype(np.float32))
    kb = ni.bf16_bits(rng.standard_normal((B, T, Hr, d)).astype(np.float32))
    vb = ni.bf16_bits(rng.standard_normal((B, T, Hr, d)).astype(np.float32))
    il, gp = "interleaved" in variant, variant.startswith("global")
    expect, top = _brute_force(_widen(qb), _widen(kb), _widen(vb), s, Kr, g, 1e4, il, gp)
    seg, row, row_src, _, _ = _pack(top, B, T, Hr)
    R = B * T * Kr
    qp = np.empty((R, g, d), np.uint16); kp = np.empty((R, d), np.uint16); vp = np.empty_like(kp)
    for b in range(B):
        for t in range(T):
            for k in range(Kr):
                h = top[b, t, k]
                r = row[b, t, k]
                qp[r] = qb[b, t, h * g:(h + 1) * g]
                kp[r] = kb[b, t, h]
                vp[r] = vb[b, t, h]
    gate = np.take_along_axis(_softmax64(s), top, -1).reshape(-1)
    pos = oracle_mod.global_positions(row_src, T, Kr) if gp else None
    if gp:  # the packed row of (b, t, k) sits at position t
        expect_pos = np.empty(R, np.int64)
        expect_pos[row.reshape(-1)] = np.broadcast_to(np.arange(T)[None, :, None], (B, T, Kr)).reshape(-1)
        np.testing.assert_array_equal(pos, expect_pos)
    y = oracle_mod.prefill(qp.reshape(R * g, d), kp, vp, seg, row_src, gate, d, g, 1e4, interleaved=il, pos=pos)
    np.testing.assert_allclose(y.reshape(B, T, Kr, g, d), expect, rtol=0, atol=1e-11)
    # the row-subset entry point agrees with the full prefill
    pick = np.arange(0, R, 7)
    heads = (pick % g).astype(np.int32)
    out = oracle_mod.prefill_rows(qp.reshape(R * g, d), kp, vp, seg, row_src, gate, d, g, 1e4, pick, heads,
                                  interleaved=il, pos=pos)
    np.testing.assert_allclose(out, y[row_src[pick] * g + heads], rtol=0, atol=1e-13)


def test_causal_support_and_weights_sum_to_one(oracle_mod):
    wl = ni.PrefillWorkload("t", B=2, T=64, H=4, K=2, d=16)
    out = oracle_mod.route(wl.scores(), wl.K)
    q, k, v = wl.qkv()
    seg, rs = out["seg_offsets"], out["row_src"]
    y0 = oracle_mod.prefill(q, k, v, seg, rs, out["gate"], wl.d, 1, wl.base)
    # perturb V (and K) of later rows of segment 1 and of every other segment
    s_lo, s_hi = seg[1], seg[2]
    r_keep = s_lo + (s_hi - s_lo) // 2
    v2, k2 = v.copy(), k.copy()
    others = np.r_[0:s_lo, r_keep + 1:len(v)]
    v2[others] ^= 0x0055
    k2[others] ^= 0x0033
    y1 = oracle_mod.prefill(q, k2, v2, seg, rs, out["gate"], wl.d, 1, wl.base)
    keep = rs[s_lo:r_keep + 1]
    np.testing.assert_array_equal(y1[keep], y0[keep])
    # constant values: the weights sum to one, so h = 1 and y = gate
    ones = np.full_like(v, 0x3F80)
    y2 = oracle_mod.prefill(q, k, ones, seg, rs, out["gate"], wl.d, 1, wl.base)
    np.testing.assert_allclose(y2, np.repeat(out["gate"].reshape(-1, 1), wl.d, 1), rtol=1e-14, atol=0)


# --------------------------------------------------------------------------- decode
def _prefix_cache(oracle_mod, q, k, v, out, T, K, d, g, base, headroom, Hr, B, interleaved=False,
                  global_pos=False):
    """Prefill over the first T tokens; returns y and the fp64 caches with headroom."""
    seg = out["seg_offsets"]
    pos = oracle_mod.global_positions(out["row_src"], T, K) if global_pos else None
    y, krot = oracle_mod.prefill(q, k, v, seg, out["row_src"], out["gate"], d, g, base, return_krot=True,
                                 interleaved=interleaved, pos=pos)
    nseg = B * Hr
    n = (seg[1:] - seg[:-1]).astype(np.int32)
    seg_base = (seg[:-1] + np.arange(nseg) * headroom).astype(np.int64)
    cap = (n + headroom).astype(np.int32)
    kc = np.zeros((int(seg[-1]) + nseg * headroom, d))
    vc = np.zeros_like(kc)
    for s_ in range(nseg):
        kc[seg_base[s_]:seg_base[s_] + n[s_]] = krot[seg[s_]:seg[s_ + 1]]
        vc[seg_base[s_]:seg_base[s_] + n[s_]] = _widen(v[seg[s_]:seg[s_ + 1]])
    return y, kc, vc, seg_base, n.copy(), cap


@pytest.mark.parametrize("variant", ["rank", "interleaved", "global", "global_interleaved"])
@pytest.mark.parametrize("g", [1, 2])
def test_prefill_equals_incremental_decode(oracle_mod, g, variant):
    B, T, Hr, Kr, d, steps, base = 2, 40, 4, 2, 16, 3, 1e4
    il, gp = "interleaved" in variant, variant.startswith("global")
    Ttot = T + steps
    s = ni.router_scores(8, B, Ttot, Hr)
    full = oracle_mod.route(s, Kr)
    R = B * Ttot * Kr
    q, k, v = ni.qkv_rows(8, R, d, g)
    pos_full = oracle_mod.global_positions(full["row_src"], Ttot, Kr) if gp else None
    y_full = oracle_mod.prefill(q, k, v, full["seg_offsets"], full["row_src"], full["gate"], d, g, base,
                                interleaved=il, pos=pos_full)
    # the prefix: drop the rows of the last `steps` tokens (the last rows of their segments)
    tok = full["row_src"] // Kr % Ttot
    keep = np.nonzero(tok < T)[0]
    pre = oracle_mod.route(s[:, :T], Kr)
    np.testing.assert_array_equal(pre["row_src"], full["row_src"][keep] - (full["row_src"][keep] // (Ttot * Kr)) * (steps * Kr))
    qg = q.reshape(R, g, d)
    _, kc, vc, seg_base, n, cap = _prefix_cache(oracle_mod, qg[keep].reshape(-1, d), k[keep], v[keep], pre,
                                                T, Kr, d, g, base, steps, Hr, B, il, gp)
    # M_KV = T K after the prefix
    assert int(n.sum()) == B * T * Kr
    for st in range(steps):
        t = T + st
        top = full["topk_head"][:, t]
        rows = full["row"][:, t]
        yq = oracle_mod.decode_step(top, full["gate"][:, t], qg[rows].reshape(B, Kr * g, d), k[rows], v[rows],
                                    Hr, d, g, base, kc, vc, seg_base, n, cap, interleaved=il,
                                    token_pos=np.full(B, t, np.int64) if gp else None)
        idx = (np.arange(B)[:, None] * Ttot + t) * Kr + np.arange(Kr)[None, :]
        expect = y_full.reshape(B * Ttot * Kr, g, d)[idx.reshape(-1)].reshape(B, Kr * g, d)
        np.testing.assert_allclose(yq, expect, rtol=0, atol=1e-12)
        assert int(n.sum()) == B * (T + st + 1) * Kr  # + K per step


def test_decode_capacity_overflow_is_an_error(oracle_mod):
    B, Hr, Kr, d = 1, 2, 1, 8
    kc = np.zeros((4, d)); vc = np.zeros((4, d))
    seg_base = np.array([0, 2], np.int64)
    seg_len = np.array([2, 0], np.int32)
    cap = np.array([2, 2], np.int32)
    q = np.zeros((1, 1, d), np.uint16); k = q.copy(); v = q.copy()
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.decode_step(np.array([[0]]), np.array([[1.0]]), q, k, v, Hr, d, 1, 1e4, kc, vc, seg_base,
                               seg_len, cap)


# --------------------------------------------------------------------------- ragged batches
@pytest.mark.parametrize("global_pos", [False, True])
def test_varlen_prefill_equals_each_sequence_alone(oracle_mod, global_pos):
    """A ragged batch is independent sequences: prefill over the packed batch equals prefill
    of every sequence on its own (no attention across sequences, positions per sequence)."""
    lens, H, K, d, g, base = [37, 0, 130, 1, 64], 4, 2, 16, 2, 1e4
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    s = ni.router_scores(13, 1, N, H)[0]
    out = oracle_mod.route_varlen(s, cu, K)
    q, k, v = ni.qkv_rows(13, N * K, d, g)
    pos = oracle_mod.global_positions_varlen(out["row_src"], cu, K) if global_pos else None
    y = oracle_mod.prefill(q, k, v, out["seg_offsets"], out["row_src"], out["gate"], d, g, base, pos=pos)
    y = y.reshape(N, K, g, d)
    qg = q.reshape(N * K, g, d)
    for b, L in enumerate(lens):
        if L == 0:
            continue
        one = oracle_mod.route(s[None, cu[b]:cu[b + 1]], K)
        rows = out["row"][cu[b]:cu[b + 1]]  # this sequence's packed rows, in (t, slot) order
        # the same rows, re-packed in the single-sequence layout
        src = np.empty(L * K, np.int64)
        src[one["row"].reshape(-1)] = rows.reshape(-1)
        pos1 = oracle_mod.global_positions(one["row_src"], L, K) if global_pos else None
        y1 = oracle_mod.prefill(qg[src].reshape(-1, d), k[src], v[src], one["seg_offsets"], one["row_src"],
                                one["gate"], d, g, base, pos=pos1)
        np.testing.assert_array_equal(y[cu[b]:cu[b + 1]], y1.reshape(L, K, g, d))
    if global_pos:  # the position is the token's index in its own sequence
        tok = out["row_src"] // K
        for r in range(N * K):
            b = int(np.nonzero(cu[1:] > tok[r])[0][0])
            assert pos[r] == tok[r] - cu[b]
