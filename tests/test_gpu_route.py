"""GPU parity of routing and dispatch against the oracle (bit-exact integers, fp32 gates).

Sec. 3.1 Eq. (namoh-gates), the ordered index sets I_i, and Sec. 3.2 Eq. (namoh-head-rope).
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import GATE_RTOL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _check_route(namoh, oracle_mod, s: np.ndarray, K: int):
    B, T, H = s.shape
    out = namoh.namoh_route(torch.from_numpy(s).cuda(), K)
    torch.cuda.synchronize()
    ref = oracle_mod.route(s, K)
    np.testing.assert_array_equal(out.topk_head.cpu().numpy(), ref["topk_head"])
    np.testing.assert_array_equal(out.rank.cpu().numpy(), ref["rank"])
    np.testing.assert_array_equal(out.row.cpu().numpy(), ref["row"])
    np.testing.assert_array_equal(out.seg_offsets.cpu().numpy(), ref["seg_offsets"])
    np.testing.assert_array_equal(out.row_src.cpu().numpy(), ref["row_src"])
    np.testing.assert_allclose(out.gate.cpu().numpy(), ref["gate"], rtol=GATE_RTOL, atol=0)
    assert int(out.status.item()) == 0
    return out


@pytest.mark.parametrize("B,T,H,K", [
    (1, 512, 8, 2),      # PR1 routing
    (2, 1000, 16, 4),    # ragged last chunk
    (3, 257, 5, 3),      # H not a power of two, one token past a chunk
    (1, 40, 64, 64),     # K = H = the limit
    (2, 300, 64, 1),     # K = 1 with the widest router
    (1, 1, 8, 2),        # one token
    (4, 4096, 16, 4),    # balanced routing at full size
    (1, 65536, 16, 4),   # 256 chunks x 16 heads = 4096 table entries: the largest summed per block
    (1, 65537, 16, 4),   # one token more: 4112 entries, the count table is scanned once instead
    (2, 19200, 64, 8),   # 75 chunks of the widest router (4800 entries): scanned
    (3, 70000, 16, 4),   # 274 chunks per sequence: scanned
])
def test_route_matches_oracle(namoh, oracle_mod, B, T, H, K):
    _check_route(namoh, oracle_mod, ni.router_scores(0, B, T, H), K)


def test_route_ties_and_signed_zeros(namoh, oracle_mod):
    rng = np.random.default_rng(5)
    s = (np.round(2 * rng.standard_normal((2, 700, 16))) / 2).astype(np.float32)
    s[0, :50] = 0.0
    s[0, :50, ::3] = -0.0
    _check_route(namoh, oracle_mod, s, 4)


def test_route_all_tokens_same_heads(namoh, oracle_mod):
    s = np.tile(np.linspace(1, -1, 32, dtype=np.float32), (1, 3000, 1))
    out = _check_route(namoh, oracle_mod, s, 4)
    n = np.diff(out.seg_offsets.cpu().numpy())
    assert list(n[:4]) == [3000] * 4 and n[4:].sum() == 0


def test_route_skewed_full_size(namoh, oracle_mod):
    wl = ni.SKEWED
    _check_route(namoh, oracle_mod, wl.scores(), wl.K)


@pytest.mark.parametrize("H", [8, 16, 32, 64])
def test_route_h_sweep_full_size(namoh, oracle_mod, H):
    _check_route(namoh, oracle_mod, ni.router_scores(0, 1, 16384, H), 4)


def test_route_decode_prefix_full_size(namoh, oracle_mod):
    """64 x 131072 tokens, H = 32, K = 4: 1.07 GB of logits; every sequence checked."""
    wl = ni.DECODE
    s = ni.router_scores(wl.seed, wl.B, wl.prefix, wl.Hr)
    out = namoh.namoh_route(torch.from_numpy(s).cuda(), wl.Kr)
    torch.cuda.synchronize()
    ref = oracle_mod.route(s, wl.Kr)
    np.testing.assert_array_equal(out.topk_head.cpu().numpy(), ref["topk_head"])
    np.testing.assert_array_equal(out.rank.cpu().numpy(), ref["rank"])
    np.testing.assert_array_equal(out.seg_offsets.cpu().numpy(), ref["seg_offsets"])
    np.testing.assert_array_equal(out.row_src.cpu().numpy(), ref["row_src"])
    np.testing.assert_array_equal(out.row.cpu().numpy(), ref["row"])
    np.testing.assert_allclose(out.gate.cpu().numpy(), ref["gate"], rtol=GATE_RTOL, atol=0)


def test_route_single_token_without_packing(namoh, oracle_mod):
    s = ni.router_scores(1, 64, 1, 32)
    out = namoh.namoh_route(torch.from_numpy(s).cuda(), 4, compact=False)
    torch.cuda.synchronize()
    ref = oracle_mod.route(s, 4)
    np.testing.assert_array_equal(out.topk_head.cpu().numpy(), ref["topk_head"])
    np.testing.assert_allclose(out.gate.cpu().numpy(), ref["gate"], rtol=GATE_RTOL, atol=0)


def test_route_nonfinite_sets_status(namoh):
    s = ni.router_scores(2, 1, 300, 8)
    s[0, 7, 3] = np.nan
    s[0, 200, 1] = -np.inf
    out = namoh.namoh_route(torch.from_numpy(s).cuda(), 2)
    torch.cuda.synchronize()
    assert int(out.status.item()) & namoh.NAMOH_DEV_NONFINITE_SCORE
    top = out.topk_head.cpu().numpy()
    assert top.min() >= 0 and top.max() < 8  # still in range
    assert int(out.seg_offsets[-1].item()) == 300 * 2


def test_route_repeated_calls_reuse_workspace(namoh, oracle_mod):
    """Back-to-back calls on one workspace: nothing carries over from one call to the next."""
    ws = namoh.Workspace()
    for seed in (3, 4, 3):
        s = ni.router_scores(seed, 2, 3000, 16)
        out = namoh.namoh_route(torch.from_numpy(s).cuda(), 4, workspace=ws)
        torch.cuda.synchronize()
        r = oracle_mod.route(s, 4)
        np.testing.assert_array_equal(out.row_src.cpu().numpy(), r["row_src"])
        np.testing.assert_array_equal(out.seg_offsets.cpu().numpy(), r["seg_offsets"])
        assert int(out.status.item()) == 0


# --------------------------------------------------------------------------- biased selection
# App. A.3, Eq. (namoh-biased-routing).  The GPU ranks fp32 affinities (exp2 of pre-scaled logit
# differences) plus the bias; the oracle ranks the same sums in fp64.  Where two sums lie
# within the fp32 error bound of each other either order is correct, so the selection is
# checked for validity within that bound, and for equality with the oracle wherever the
# margins are larger; the dispatch of the GPU's own picks must then be bit-exact.
BIAS_EPS = 4e-6


def _check_biased(namoh, oracle_mod, scores, K, bias, compact=True):
    import scipy.special
    H = scores.shape[-1]
    dev = torch.device("cuda")
    out = namoh.namoh_route(torch.from_numpy(scores).to(dev), K, compact=compact,
                            bias=torch.from_numpy(bias).to(dev))
    torch.cuda.synchronize()
    ref = oracle_mod.route_biased(scores, K, bias)
    top = out.topk_head.cpu().numpy().astype(np.int64)
    key = ref["key"]
    sel = np.take_along_axis(key, top, -1)
    mask = np.zeros(key.shape, bool)
    np.put_along_axis(mask, top, True, -1)
    assert (mask.sum(-1) == K).all(), "picks are not K distinct heads"
    if K < H:
        assert (sel.min(-1) >= np.where(mask, -np.inf, key).max(-1) - BIAS_EPS).all()
    assert (np.diff(sel, axis=-1) <= BIAS_EPS).all()
    ordered = -np.sort(-key, axis=-1)[..., :min(K + 1, H)]
    clear = (-np.diff(ordered, axis=-1) > BIAS_EPS).all(-1)
    np.testing.assert_array_equal(top[clear], ref["topk_head"][clear])
    assert clear.mean() > 0.9  # most tokens are compared exactly
    a = scipy.special.softmax(scores.astype(np.float64), axis=-1)
    np.testing.assert_allclose(out.gate.cpu().numpy(), np.take_along_axis(a, top, -1), rtol=GATE_RTOL, atol=0)
    if compact:
        d = oracle_mod.dispatch(top, H)
        np.testing.assert_array_equal(out.rank.cpu().numpy(), d["rank"])
        np.testing.assert_array_equal(out.row.cpu().numpy(), d["row"])
        np.testing.assert_array_equal(out.seg_offsets.cpu().numpy(), d["seg_offsets"])
        np.testing.assert_array_equal(out.row_src.cpu().numpy(), d["row_src"])
    assert int(out.status.item()) == 0


@pytest.mark.parametrize("B,T,H,K", [
    (4, 4096, 16, 4),    # balanced routing
    (1, 8192, 32, 4),    # the decode prefix's router
    (2, 777, 64, 8),     # K = 8 (picks in registers)
    (1, 300, 64, 16),    # K > 8 (K passes over the logits)
    (3, 257, 5, 3),      # H not a power of two
])
@pytest.mark.parametrize("spread", [0.02, 0.5])
def test_route_biased_matches_oracle(namoh, oracle_mod, B, T, H, K, spread):
    bias = (np.random.default_rng(H * 31 + K).standard_normal(H) * spread / H).astype(np.float32)
    _check_biased(namoh, oracle_mod, ni.router_scores(7, B, T, H), K, bias)


def test_route_biased_single_token_without_packing(namoh, oracle_mod):
    bias = (np.random.default_rng(4).standard_normal(32) * 0.01).astype(np.float32)
    _check_biased(namoh, oracle_mod, ni.router_scores(9, 64, 1, 32), 4, bias, compact=False)


def test_route_biased_dominant_head(namoh, oracle_mod):
    bias = np.zeros(16, np.float32)
    bias[11] = 3.0
    s = ni.router_scores(12, 2, 1000, 16)
    _check_biased(namoh, oracle_mod, s, 4, bias)
