"""GPU parity of the projections around the path (the full attention layer).

Sec. 3.1 Eq. (namoh-qkv): q, k, v = x W^(i) for active token-head pairs only, in the packed
layout.  Eq. (namoh-attention): o_t = sum_i g h W_O^(i).  App. B.7: g queries per KV group.
Each stage is compared with the oracle on the same bf16 inputs: the projections' bf16 outputs
within half a bf16 ulp of the fp64 value (|err| <= 2^-8 |ref| + 1e-3); the fp32 o sums per-slot
products that were rounded to bf16, so |err| <= 2^-8 (sum of |y| |W_O| over its terms) + 1e-5.
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import bf16_to_f64, dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _weights(seed, Hr, g, d, d_model):
    rng = np.random.default_rng([seed, 7])
    w_qkv = ni.bf16_bits((rng.standard_normal((Hr, (g + 2) * d, d_model)) / np.sqrt(d_model)).astype(np.float32))
    w_o = ni.bf16_bits((rng.standard_normal((Hr, d_model, g * d)) / np.sqrt(g * d)).astype(np.float32))
    return w_qkv, w_o


def _x(seed, N, d_model):
    return ni.bf16_bits(np.random.default_rng([seed, 8]).standard_normal((N, d_model)).astype(np.float32))


def _check_proj(got, ref):
    err = np.abs(got - ref)
    bound = np.abs(ref) * 2.0 ** -8 + 1e-3
    assert np.all(err <= bound), f"max excess {float(np.max(err - bound)):.3g}"


def _sub_layout(seg, row_src, rows):
    """The packed layout restricted to `rows` (sorted): segment offsets over the kept rows."""
    rows = np.sort(rows)
    sidx = np.searchsorted(seg, rows, side="right") - 1
    counts = np.bincount(sidx, minlength=len(seg) - 1)
    return rows, np.concatenate([[0], np.cumsum(counts)]).astype(np.int32), row_src[rows]


def _run_qkv(namoh, oracle_mod, ro, ref, x, w_qkv, B, H, K, g, d, rows=None):
    Hr, Kr = H // g, K // g
    q, k, v = namoh.namoh_proj_qkv(dev_bf16(x), dev_bf16(w_qkv), ro.seg_offsets, ro.row_src, B=B, H=H, K=K,
                                   group=g, status=ro.status)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    seg, rs = ref["seg_offsets"], ref["row_src"]
    if rows is None:
        rows = np.arange(int(seg[-1]))
    rows, seg2, rs2 = _sub_layout(seg, rs, rows)
    qr, kr, vr = oracle_mod.proj_qkv(x, w_qkv, seg2, rs2, Hr, Kr, g, d)
    qg = bf16_to_f64(q).reshape(-1, g, d)
    _check_proj(qg[rows].reshape(-1, d), qr)
    _check_proj(bf16_to_f64(k)[rows], kr)
    _check_proj(bf16_to_f64(v)[rows], vr)
    return q, k, v


@pytest.mark.parametrize("B,T,H,K,d,g,d_model", [
    (2, 300, 8, 2, 128, 1, 512),    # (g+2) d = 384: two 192-column tiles
    (1, 500, 8, 4, 64, 2, 256),     # 256 columns: one tile
    (2, 130, 16, 8, 64, 4, 128),    # 384 columns, two k-blocks
    (1, 200, 64, 32, 128, 8, 64),   # 1280 columns in five 256-wide tiles, one k-block
    (3, 1, 8, 2, 128, 1, 192),      # one token per sequence: tiles of one row
    (72, 24, 16, 2, 128, 1, 128),   # 1152 segments: the tile list comes from the list kernels
])
def test_proj_qkv_matches_oracle(namoh, oracle_mod, B, T, H, K, d, g, d_model):
    Hr, Kr = H // g, K // g
    s = ni.router_scores(40, B, T, Hr)
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), Kr)
    ref = oracle_mod.route(s, Kr)
    np.testing.assert_array_equal(ro.row_src.cpu().numpy(), ref["row_src"])
    w_qkv, _ = _weights(40, Hr, g, d, d_model)
    _run_qkv(namoh, oracle_mod, ro, ref, _x(40, B * T, d_model), w_qkv, B, H, K, g, d)


def test_proj_qkv_empty_heads_and_ragged_batch(namoh, oracle_mod):
    """A ragged batch with empty sequences, and all tokens of one sequence on two heads."""
    lens, H, K, d, d_model = [0, 333, 1, 0, 129], 8, 2, 128, 256
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    s = ni.router_scores(41, 1, N, H)[0]
    s[cu[1]:cu[2], :2] += 10.0
    ro = namoh.namoh_route_varlen(torch.from_numpy(s).cuda(), torch.from_numpy(cu).cuda(), max(lens), K)
    ref = oracle_mod.route_varlen(s, cu, K)
    w_qkv, _ = _weights(41, H, 1, d, d_model)
    _run_qkv(namoh, oracle_mod, ro, ref, _x(41, N, d_model), w_qkv, len(lens), H, K, 1, d)


def _y(seed, N, Kr, g, d):
    """Seeded per-slot outputs y [N, Kr*g, d] (bf16 bits), of the size of g h for N(0, 1) values."""
    rng = np.random.default_rng([seed, 9])
    return ni.bf16_bits((0.3 * rng.standard_normal((N, Kr * g, d))).astype(np.float32))


def _check_out(oracle_mod, o, y_bits, top, w_o, g, d, base=None):
    """o against the oracle's sum over slots of y W_O for the same bf16 y (base: what accumulate added to)."""
    N = y_bits.shape[0]
    yf = ni.bf16_to_f32(y_bits).astype(np.float64).reshape(N, -1, g, d)
    ref = oracle_mod.proj_out(yf, top, w_o, g, d)
    scale = oracle_mod.proj_out(np.abs(yf), top, ni.bf16_bits(np.abs(ni.bf16_to_f32(w_o))), g, d)  # sum of |terms|
    got = o.cpu().numpy().astype(np.float64)
    if base is None:
        err = np.abs(got - ref)
        assert np.all(err <= 2.0 ** -8 * scale + 1e-5)
    else:
        err = np.abs(got - (ref + base))
        assert np.all(err <= 2.0 ** -8 * scale + 1e-6 * np.abs(base) + 1e-5)


@pytest.mark.parametrize("g,d_model", [
    (1, 512),   # two 256-column tiles
    (2, 512),
    (1, 192),   # one 192-column tile
])
def test_proj_out_matches_oracle(namoh, oracle_mod, g, d_model):
    """o = sum over slots of y W_O on a seeded y, and accumulate adds onto o."""
    B, T, H, K, d = 2, 400, 8 * g, 2 * g, 128
    Hr, Kr = H // g, K // g
    s = ni.router_scores(42, B, T, Hr)
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), Kr)
    ref = oracle_mod.route(s, Kr)
    y_bits = _y(42, B * T, Kr, g, d)
    y = dev_bf16(y_bits).view(B, T, K, d)
    _, w_o = _weights(42, Hr, g, d, d_model)
    o = namoh.namoh_proj_out(y, dev_bf16(w_o), ro.seg_offsets, ro.row_src, B=B, H=H, K=K, group=g, status=ro.status)
    base = torch.randn_like(o)
    o2 = namoh.namoh_proj_out(y, dev_bf16(w_o), ro.seg_offsets, ro.row_src, B=B, H=H, K=K, group=g,
                              o=base.clone(), accumulate=True, status=ro.status)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    top = ref["topk_head"].reshape(B * T, Kr)
    _check_out(oracle_mod, o, y_bits, top, w_o, g, d)
    _check_out(oracle_mod, o2, y_bits, top, w_o, g, d, base=base.cpu().numpy().astype(np.float64))


def test_proj_out_many_segments(namoh, oracle_mod):
    """1152 segments (more than a CTA's own tile table holds): the list kernels' tile list."""
    B, T, H, K, d, d_model = 72, 24, 16, 2, 128, 256
    s = ni.router_scores(44, B, T, H)
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), K)
    ref = oracle_mod.route(s, K)
    y_bits = _y(44, B * T, K, 1, d)
    _, w_o = _weights(44, H, 1, d, d_model)
    o = namoh.namoh_proj_out(dev_bf16(y_bits).view(B, T, K, d), dev_bf16(w_o), ro.seg_offsets, ro.row_src, B=B, H=H,
                             K=K, status=ro.status)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    _check_out(oracle_mod, o, y_bits, ref["topk_head"].reshape(B * T, K), w_o, 1, d)


def test_layer_full_size(namoh, oracle_mod):
    """The balanced workload's projections at d_model = 2048, in the launch configuration the
    benchmark times: the QKV projection of all 65536 packed rows and the output projection of all
    16384 tokens (on a seeded y), every element against the oracle."""
    wl = ni.BALANCED
    d_model = 2048
    B, T, H, K, d = wl.B, wl.T, wl.H, wl.K, wl.d
    s = wl.scores()
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), K)
    ref = oracle_mod.route(s, K)
    x = _x(43, B * T, d_model)
    w_qkv, w_o = _weights(43, H, 1, d, d_model)
    _run_qkv(namoh, oracle_mod, ro, ref, x, w_qkv, B, H, K, 1, d)
    y_bits = _y(43, B * T, K, 1, d)
    o = namoh.namoh_proj_out(dev_bf16(y_bits).view(B, T, K, d), dev_bf16(w_o), ro.seg_offsets, ro.row_src, B=B, H=H,
                             K=K, status=ro.status)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    _check_out(oracle_mod, o, y_bits, ref["topk_head"].reshape(B * T, K), w_o, 1, d)
