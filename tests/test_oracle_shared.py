"""Pins of the oracle's shared heads (the paper's shared-head variant, Sec. 4.4 "Shared heads for
local context"): always-active heads attending to the full causal prefix or to the most recent
w tokens including the current one, with global RoPE and no gate.

Checked against torch scaled_dot_product_attention with RoPE written as complex multiplication:
causal for the full prefix, an explicit band mask for the window; w = 1 gives y = v; prefill and
incremental decoding agree for a window too.
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni


def _widen(bits):
    return ni.bf16_to_f32(bits).astype(np.float64)


def _rope_complex(x, pos, base):
    d = x.shape[-1]
    half = d // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = np.exp(-np.log(base) * (2.0 * np.arange(half) / d))
    rot = z * np.exp(1j * np.asarray(pos, np.float64)[..., None] * freq)
    return np.concatenate([rot.real, rot.imag], axis=-1)


def _qkv(seed, B, Hs, T, d):
    rng = np.random.default_rng(seed)
    return tuple(ni.bf16_bits(rng.standard_normal((B, Hs, T, d)).astype(np.float32)) for _ in range(3))


def _sdpa(q, k, v, base, window):
    B, Hs, T, d = q.shape
    pos = np.arange(T)
    qr = torch.from_numpy(_rope_complex(_widen(q), pos, base))
    kr = torch.from_numpy(_rope_complex(_widen(k), pos, base))
    vv = torch.from_numpy(_widen(v))
    t = torch.arange(T)
    allowed = t[None, :] <= t[:, None]
    if window > 0:
        allowed = allowed & (t[None, :] > t[:, None] - window)
    h = torch.nn.functional.scaled_dot_product_attention(qr, kr, vv, attn_mask=allowed)
    return h.numpy().transpose(0, 2, 1, 3)  # [B, T, Hs, d]


@pytest.mark.parametrize("window", [0, 1, 5, 16, 100])
def test_shared_heads_match_masked_sdpa(oracle_mod, window):
    B, Hs, T, d, base = 2, 3, 40, 16, 1e4
    q, k, v = _qkv(50, B, Hs, T, d)
    y = oracle_mod.shared_prefill(q, k, v, window, base)
    np.testing.assert_allclose(y, _sdpa(q, k, v, base, window), rtol=0, atol=1e-11)


def test_window_one_is_the_value(oracle_mod):
    q, k, v = _qkv(51, 1, 2, 30, 8)
    y = oracle_mod.shared_prefill(q, k, v, 1, 1e4)
    np.testing.assert_array_equal(y, _widen(v).transpose(0, 2, 1, 3))


def test_window_at_least_t_is_full_causal(oracle_mod):
    q, k, v = _qkv(52, 1, 2, 25, 8)
    np.testing.assert_array_equal(oracle_mod.shared_prefill(q, k, v, 25, 1e4), oracle_mod.shared_prefill(q, k, v, 0, 1e4))


@pytest.mark.parametrize("window", [0, 7])
def test_shared_prefill_equals_incremental_decode(oracle_mod, window):
    """Prefill over T + s tokens equals prefill over T (its rotated keys cached) plus s decode
    steps with every shared head active, gate 1, and the same window."""
    B, Hs, T, d, steps, base = 2, 2, 20, 8, 4, 1e4
    q, k, v = _qkv(53, B, Hs, T + steps, d)
    y_full = oracle_mod.shared_prefill(q, k, v, window, base)
    nseg = B * Hs
    cap = T + steps
    kc = np.zeros((nseg * cap, d)); vc = np.zeros_like(kc)
    for s in range(nseg):
        b, j = divmod(s, Hs)
        kc[s * cap:s * cap + T] = _rope_complex(_widen(k[b, j, :T]), np.arange(T), base)
        vc[s * cap:s * cap + T] = _widen(v[b, j, :T])
    seg_base = (np.arange(nseg) * cap).astype(np.int64)
    seg_len = np.full(nseg, T, np.int32)
    seg_cap = np.full(nseg, cap, np.int32)
    for st in range(steps):
        t = T + st
        y = oracle_mod.shared_decode_step(q[:, :, t], k[:, :, t], v[:, :, t], d, base, kc, vc, seg_base, seg_len,
                                          seg_cap, window)
        np.testing.assert_allclose(y, y_full[:, t], rtol=0, atol=1e-12)
