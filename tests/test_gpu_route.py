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
