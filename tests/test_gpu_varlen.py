"""GPU parity of ragged batches (sequences of different lengths packed back to back).

Sec. 3.1 / Sec. 3.2 per sequence: index sets, ranks and segments restart at each sequence's
first token; prefill attends only within a sequence; global RoPE positions (Sec. 3.2) are the
token's index inside its own sequence.  Routing is bit-exact against the oracle; attention is
within the 2e-2 max / 2e-3 mean-abs tolerance.
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import GATE_RTOL, assert_close_attention, bf16_to_f64, dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _ragged(seed, lens, H):
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    s = ni.router_scores(seed, 1, int(cu[-1]), H)[0]
    return s, cu


def _route_gpu(namoh, s, cu, K, bias=None):
    out = namoh.namoh_route_varlen(torch.from_numpy(s).cuda(), torch.from_numpy(cu).cuda(), int(np.diff(cu).max()),
                                   K, bias=None if bias is None else torch.from_numpy(bias).cuda())
    torch.cuda.synchronize()
    return out


def _check_layout(out, ref):
    for key in ("topk_head", "rank", "row", "seg_offsets", "row_src"):
        np.testing.assert_array_equal(getattr(out, key).cpu().numpy(), ref[key], err_msg=key)


@pytest.mark.parametrize("lens,H,K", [
    ([5, 0, 300, 1, 256, 257], 8, 2),      # empty, one-token and chunk-boundary sequences
    ([1000, 3000, 17], 16, 4),
    ([40000, 123, 9000, 0], 32, 4),         # 157 chunks x 32 heads: the count table is scanned
    ([64] * 9 + [4096], 64, 8),
])
def test_route_varlen_matches_oracle(namoh, oracle_mod, lens, H, K):
    s, cu = _ragged(21, lens, H)
    out = _route_gpu(namoh, s, cu, K)
    ref = oracle_mod.route_varlen(s, cu, K)
    _check_layout(out, ref)
    np.testing.assert_allclose(out.gate.cpu().numpy(), ref["gate"], rtol=GATE_RTOL, atol=0)
    assert int(out.status.item()) == 0


def test_route_varlen_uniform_equals_fixed(namoh):
    """Equal lengths: the ragged entry point gives the fixed-length bytes."""
    B, T, H, K = 3, 1000, 16, 4
    s = ni.router_scores(22, B, T, H)
    fixed = namoh.namoh_route(torch.from_numpy(s).cuda(), K)
    var = _route_gpu(namoh, s.reshape(B * T, H), np.arange(B + 1, dtype=np.int32) * T, K)
    for key in ("topk_head", "gate", "rank", "row"):
        assert torch.equal(getattr(var, key), getattr(fixed, key).reshape(B * T, K)), key
    for key in ("seg_offsets", "row_src"):
        assert torch.equal(getattr(var, key), getattr(fixed, key)), key


def test_route_varlen_biased(namoh, oracle_mod):
    """Biased selection in a ragged batch: each sequence's picks equal the fixed-length biased
    routing of that sequence alone, and their dispatch is the oracle's, bit for bit."""
    lens, H, K = [700, 0, 33, 1500], 16, 4
    s, cu = _ragged(23, lens, H)
    bias = (0.05 * np.random.default_rng(23).standard_normal(H)).astype(np.float32)
    out = _route_gpu(namoh, s, cu, K, bias)
    top = out.topk_head.cpu().numpy()
    for b, L in enumerate(lens):
        if L == 0:
            continue
        one = namoh.namoh_route(torch.from_numpy(np.ascontiguousarray(s[None, cu[b]:cu[b + 1]])).cuda(), K,
                                bias=torch.from_numpy(bias).cuda())
        np.testing.assert_array_equal(top[cu[b]:cu[b + 1]], one.topk_head.cpu().numpy()[0])
        np.testing.assert_array_equal(out.gate.cpu().numpy()[cu[b]:cu[b + 1]], one.gate.cpu().numpy()[0])
    ref = oracle_mod.dispatch_varlen(top, cu, H)
    for key in ("rank", "row", "seg_offsets", "row_src"):
        np.testing.assert_array_equal(getattr(out, key).cpu().numpy(), ref[key], err_msg=key)
    assert int(out.status.item()) == 0


@pytest.mark.parametrize("cu,N,max_seqlen", [
    ([0, 300, 200, 600], 600, 400),   # decreasing
    ([0, 300, 500], 600, 300),        # does not end at N
    ([0, 100, 600], 600, 300),        # a sequence longer than max_seqlen
    ([5, 300, 600], 600, 300),        # does not start at 0
])
def test_route_varlen_bad_cu_seqlens_sets_status(namoh, cu, N, max_seqlen):
    """Malformed cu_seqlens (caught on the device): the status bit is set and every row the
    layout names stays below N*K (the kernels clamp each sequence into [0, N])."""
    H, K = 8, 2
    s = ni.router_scores(24, 1, N, H)[0]
    out = namoh.namoh_route_varlen(torch.from_numpy(s).cuda(), torch.tensor(cu, dtype=torch.int32, device="cuda"),
                                   max_seqlen, K)
    torch.cuda.synchronize()
    assert int(out.status.item()) & namoh.NAMOH_DEV_BAD_SEQLENS
    seg = out.seg_offsets.cpu().numpy()
    assert seg.min() >= 0 and seg.max() <= N * K


VARIANTS = ["rank", "global", "global_interleaved"]


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("lens,H,K,d,g", [
    ([37, 0, 700, 1, 129, 256], 8, 2, 128, 1),
    ([300, 1000, 5], 16, 8, 64, 2),
])
def test_prefill_varlen_matches_oracle(namoh, oracle_mod, lens, H, K, d, g, variant):
    Hr, Kr = H // g, K // g
    s, cu = _ragged(25, lens, Hr)
    N = int(cu[-1])
    ro = _route_gpu(namoh, s, cu, Kr)
    ref = oracle_mod.route_varlen(s, cu, Kr)
    _check_layout(ro, ref)
    q, k, v = ni.qkv_rows(25, N * Kr, d, g)
    il, gp = "interleaved" in variant, variant.startswith("global")
    y, kc, _ = namoh.namoh_prefill_varlen(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets.new_tensor(cu),
                                          int(max(lens)), ro.seg_offsets, ro.row_src, ro.gate, H=H, K=K, group=g,
                                          interleaved=il, global_positions=gp, status=ro.status)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    pos = oracle_mod.global_positions_varlen(ref["row_src"], cu, Kr) if gp else None
    y_ref, krot = oracle_mod.prefill(q, k, v, ref["seg_offsets"], ref["row_src"], ref["gate"], d, g, 1e4,
                                     return_krot=True, interleaved=il, pos=pos)
    assert_close_attention(bf16_to_f64(y).reshape(-1, d), y_ref, np.repeat(ref["gate"].reshape(-1), g))
    kc_got = bf16_to_f64(kc)
    assert np.all(np.abs(kc_got - krot) <= np.abs(krot) * 2.0 ** -7 + 1e-6)


def test_prefill_varlen_uniform_equals_fixed(namoh):
    """Equal lengths: namoh_prefill_varlen writes the bytes namoh_prefill writes."""
    wl = ni.PrefillWorkload("uniform", B=3, T=700, H=8, K=2, d=128, seed=26)
    s = wl.scores()
    q, k, v = (dev_bf16(a) for a in wl.qkv())
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), wl.Kr)
    y0, kc0, _ = namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, B=wl.B, T=wl.T, H=wl.H, K=wl.K,
                                     global_positions=True)
    cu = torch.arange(wl.B + 1, dtype=torch.int32, device="cuda") * wl.T
    y1, kc1, _ = namoh.namoh_prefill_varlen(q, k, v, cu, wl.T, ro.seg_offsets, ro.row_src, ro.gate.reshape(-1, wl.K),
                                            H=wl.H, K=wl.K, global_positions=True)
    torch.cuda.synchronize()
    assert torch.equal(y0.view(torch.int16).reshape(-1), y1.view(torch.int16).reshape(-1))
    assert torch.equal(kc0.view(torch.int16), kc1.view(torch.int16))
