"""Pins of the oracle's projections around the routed-attention path.

Sec. 3.1 Eq. (namoh-qkv): only active token-head pairs project, q = x W_Q^(i), k = x W_K^(i),
v = x W_V^(i), W in R^{d_model x d_head}.  Eq. (namoh-attention): o_t = sum_{i in S_K(t)}
g_{t,i} h_{t,i} W_O^(i), W_O^(i) in R^{d_head x d_model}.  App. B.7: a KV group projects one key
and one value, and one query per query head.
Each check uses the paper's dense matrices and a formulation unlike the oracle's (dense
products over every head, then the active pairs; torch scaled_dot_product_attention for K = H).
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni


def _widen(bits):
    return ni.bf16_to_f32(bits).astype(np.float64)


def _weights(seed, Hr, g, d, d_model):
    """Dense per-head matrices as the paper writes them (bf16 bits), and the oracle's packed copies."""
    rng = np.random.default_rng(seed)
    sc = 1.0 / np.sqrt(d_model)
    wq = ni.bf16_bits((sc * rng.standard_normal((Hr * g, d_model, d))).astype(np.float32))  # W_Q^(i), query heads
    wk = ni.bf16_bits((sc * rng.standard_normal((Hr, d_model, d))).astype(np.float32))
    wv = ni.bf16_bits((sc * rng.standard_normal((Hr, d_model, d))).astype(np.float32))
    wo = ni.bf16_bits((rng.standard_normal((Hr * g, d, d_model)) / np.sqrt(d)).astype(np.float32))  # W_O^(i)
    w_qkv = np.concatenate([wq.reshape(Hr, g, d_model, d).transpose(0, 1, 3, 2).reshape(Hr, g * d, d_model),
                            wk.transpose(0, 2, 1), wv.transpose(0, 2, 1)], axis=1)
    w_o = wo.reshape(Hr, g, d, d_model).transpose(0, 3, 1, 2).reshape(Hr, d_model, g * d)
    return dict(wq=wq, wk=wk, wv=wv, wo=wo, w_qkv=np.ascontiguousarray(w_qkv), w_o=np.ascontiguousarray(w_o))


def _x(seed, N, d_model):
    return ni.bf16_bits(np.random.default_rng([seed, 9]).standard_normal((N, d_model)).astype(np.float32))


@pytest.mark.parametrize("B,T,Hr,Kr,g,d,d_model", [(2, 40, 4, 2, 1, 16, 64), (1, 33, 4, 2, 2, 8, 48)])
def test_proj_qkv_is_dense_projection_at_active_pairs(oracle_mod, B, T, Hr, Kr, g, d, d_model):
    s = ni.router_scores(30, B, T, Hr)
    out = oracle_mod.route(s, Kr)
    W = _weights(30, Hr, g, d, d_model)
    x = _x(30, B * T, d_model)
    q, k, v = oracle_mod.proj_qkv(x, W["w_qkv"], out["seg_offsets"], out["row_src"], Hr, Kr, g, d)
    xf = _widen(x)
    Q = np.einsum("nm,imc->nic", xf, _widen(W["wq"]))  # every token, every query head
    Kd = np.einsum("nm,imc->nic", xf, _widen(W["wk"]))
    V = np.einsum("nm,imc->nic", xf, _widen(W["wv"]))
    top = out["topk_head"].reshape(B * T, Kr)
    rows = out["row"].reshape(B * T, Kr)
    for tok in range(B * T):
        for slot in range(Kr):
            h, r = top[tok, slot], rows[tok, slot]
            np.testing.assert_allclose(k[r], Kd[tok, h], rtol=0, atol=1e-12)
            np.testing.assert_allclose(v[r], V[tok, h], rtol=0, atol=1e-12)
            for j in range(g):
                np.testing.assert_allclose(q[r * g + j], Q[tok, h * g + j], rtol=0, atol=1e-12)
    assert q.shape[0] == B * T * Kr * g and k.shape[0] == B * T * Kr  # inactive pairs project nothing


@pytest.mark.parametrize("g", [1, 2])
def test_proj_out_is_dense_sum_over_active_heads(oracle_mod, g):
    N, Hr, Kr, d, d_model = 50, 5, 3, 8, 40
    rng = np.random.default_rng(31)
    top = np.stack([rng.permutation(Hr)[:Kr] for _ in range(N)]).astype(np.int32)
    y = rng.standard_normal((N, Kr, g, d))
    W = _weights(31, Hr, g, d, d_model)
    o = oracle_mod.proj_out(y, top, W["w_o"], g, d)
    dense = np.zeros((N, Hr * g, d))  # g_{t,i} h_{t,i}, zero for inactive heads
    for t in range(N):
        for slot in range(Kr):
            dense[t, top[t, slot] * g:(top[t, slot] + 1) * g] = y[t, slot]
    expect = np.einsum("nic,icm->nm", dense, _widen(W["wo"]))
    np.testing.assert_allclose(o, expect, rtol=0, atol=1e-11)


def _rope_complex(x, pos, base):
    d = x.shape[-1]
    half = d // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = np.exp(-np.log(base) * (2.0 * np.arange(half) / d))
    rot = z * np.exp(1j * np.asarray(pos, np.float64)[..., None] * freq)
    return np.concatenate([rot.real, rot.imag], axis=-1)


@pytest.mark.parametrize("g", [1, 2])
def test_layer_with_k_equal_h_is_dense_gated_mha(oracle_mod, g):
    """K = H: every head is active and every rank is t, so the layer (projection, head-relative
    RoPE, routed attention, combine, output projection) is dense causal multi-head attention
    (grouped when g > 1) with standard RoPE, each head's output scaled by its softmax gate."""
    B, T, Hr, d, d_model, base = 2, 24, 3, 16, 32, 1e4
    s = ni.router_scores(32, B, T, Hr)
    out = oracle_mod.route(s, Hr)
    W = _weights(32, Hr, g, d, d_model)
    x = _x(32, B * T, d_model)
    q, k, v = oracle_mod.proj_qkv(x, W["w_qkv"], out["seg_offsets"], out["row_src"], Hr, Hr, g, d)
    qb, kb, vb = (ni.bf16_bits(a.astype(np.float32)) for a in (q, k, v))  # the path's bf16 inputs
    y = oracle_mod.prefill(qb, kb, vb, out["seg_offsets"], out["row_src"], out["gate"], d, g, base)
    o = oracle_mod.proj_out(y.reshape(B * T, Hr, g, d), out["topk_head"].reshape(B * T, Hr), W["w_o"], g, d)
    # dense reference from the same bf16 q, k, v (undo the packing with the row map)
    rows = out["row"].reshape(B * T, Hr)
    top = out["topk_head"].reshape(B * T, Hr)
    Qd = np.zeros((B * T, Hr * g, d)); Kd = np.zeros((B * T, Hr, d)); Vd = np.zeros((B * T, Hr, d))
    qf, kf, vf = _widen(qb).reshape(-1, g, d), _widen(kb), _widen(vb)
    for tok in range(B * T):
        for slot in range(Hr):
            h, r = top[tok, slot], rows[tok, slot]
            Qd[tok, h * g:(h + 1) * g] = qf[r]
            Kd[tok, h] = kf[r]
            Vd[tok, h] = vf[r]
    pos = np.arange(T)
    gate = np.zeros((B * T, Hr))
    np.put_along_axis(gate, top, out["gate"].reshape(B * T, Hr), axis=-1)
    expect = np.zeros((B * T, d_model))
    for b in range(B):
        sl = slice(b * T, (b + 1) * T)
        for i in range(Hr * g):
            qr = torch.from_numpy(_rope_complex(Qd[sl, i], pos, base))[None, None]
            kr = torch.from_numpy(_rope_complex(Kd[sl, i // g], pos, base))[None, None]
            vv = torch.from_numpy(Vd[sl, i // g])[None, None]
            h = torch.nn.functional.scaled_dot_product_attention(qr, kr, vv, is_causal=True)[0, 0].numpy()
            expect[sl] += (gate[sl, i // g][:, None] * h) @ _widen(W["wo"][i])
    np.testing.assert_allclose(o, expect, rtol=0, atol=1e-10)
