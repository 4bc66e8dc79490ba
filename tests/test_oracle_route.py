"""Pins of the oracle's routing and dispatch against what the paper fixes.

Sec. 3.1 Eq. (namoh-gates): TopK over affinities, mask, gates (not renormalised).
Sec. 3.1: ordered index sets I_i; App. B.5 Eq. (app-assignment-count): sum_i n_i = T K.
Sec. 3.2 Eq. (namoh-head-rope): rho_i(t) = sum_{s<=t} m_{s,i} - 1.
Each test uses a formulation that differs from the oracle's (counting ranks instead of
sorting, cumulative sums of the mask instead of appending, library softmax / topk).
"""
import os

import numpy as np
import pytest
import scipy.special
import torch

import namoh_inputs as ni

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "fig2_head_relative_ranks.txt")


def _rank_by_counting(s: np.ndarray) -> np.ndarray:
    """Position of each head in the order (score desc, index asc), by counting the heads ahead."""
    H = s.shape[-1]
    out = np.zeros(s.shape, np.int64)
    for h in range(H):
        ahead = (s > s[..., h:h + 1]).sum(-1) + (s[..., :h] == s[..., h:h + 1]).sum(-1)
        out[..., h] = ahead
    return out


def _topk_by_counting(s: np.ndarray, K: int) -> np.ndarray:
    pos = _rank_by_counting(s)
    B, T, H = s.shape
    top = np.full((B, T, K), -1, np.int64)
    for h in range(H):
        sel = pos[..., h] < K
        bb, tt = np.nonzero(sel)
        top[bb, tt, pos[bb, tt, h]] = h
    return top


@pytest.mark.parametrize("B,T,H,K", [(1, 64, 8, 2), (2, 37, 16, 4), (3, 20, 5, 5), (1, 50, 64, 7), (2, 9, 3, 1)])
def test_topk_matches_counting_with_ties(oracle_mod, B, T, H, K):
    rng = np.random.default_rng(11 + H)
    # quantised logits force many exact ties; include both signed zeros
    s = (np.round(4 * rng.standard_normal((B, T, H))) / 4).astype(np.float32)
    s[0, 0, :] = 0.0
    s[0, 0, ::2] = -0.0
    out = oracle_mod.route(s, K)
    np.testing.assert_array_equal(out["topk_head"], _topk_by_counting(s, K))


def test_topk_matches_torch_on_distinct_scores(oracle_mod):
    s = ni.router_scores(3, 2, 300, 32)
    out = oracle_mod.route(s, 4)
    vals, idx = torch.topk(torch.from_numpy(s).double(), 4, dim=-1, sorted=True)
    np.testing.assert_array_equal(out["topk_head"], idx.numpy())


@pytest.mark.parametrize("H,K", [(8, 2), (16, 4), (32, 32), (5, 1)])
def test_gates_are_softmax_over_all_heads(oracle_mod, H, K):
    s = ni.router_scores(5, 2, 40, H)
    out = oracle_mod.route(s, K)
    a = scipy.special.softmax(s.astype(np.float64), axis=-1)
    expect = np.take_along_axis(a, out["topk_head"].astype(np.int64), axis=-1)
    np.testing.assert_allclose(out["gate"], expect, rtol=1e-13, atol=0)
    tot = out["gate"].sum(-1)
    if K == H:
        np.testing.assert_allclose(tot, 1.0, rtol=1e-13)
    else:
        assert np.all(tot < 1.0)  # not renormalised over the selected heads
    # slots follow descending score
    sel = np.take_along_axis(s, out["topk_head"].astype(np.int64), axis=-1)
    assert np.all(np.diff(sel, axis=-1) <= 0)


@pytest.mark.parametrize("B,T,H,K", [(1, 512, 8, 2), (3, 100, 16, 4), (2, 33, 4, 4), (4, 7, 9, 1)])
def test_dispatch_matches_mask_cumsum(oracle_mod, B, T, H, K):
    s = ni.router_scores(7, B, T, H)
    out = oracle_mod.route(s, K)
    top = out["topk_head"].astype(np.int64)
    mask = np.zeros((B, T, H), np.int64)
    np.put_along_axis(mask, top, 1, axis=-1)
    # Eq. (namoh-head-rope): rho_i(t) = sum_{s<=t} m_{s,i} - 1
    rho = np.cumsum(mask, axis=1) - 1
    np.testing.assert_array_equal(out["rank"], np.take_along_axis(rho, top, axis=-1))
    n = mask.sum(axis=1)
    np.testing.assert_array_equal(out["n"], n)
    # App. B.5 Eq. (app-assignment-count): sum_i n_i = T K for every sequence
    np.testing.assert_array_equal(n.sum(-1), T * K)
    seg = np.concatenate([[0], np.cumsum(n.reshape(-1))])
    np.testing.assert_array_equal(out["seg_offsets"], seg)
    assert out["seg_offsets"][-1] == B * T * K
    b_idx = np.arange(B)[:, None, None]
    np.testing.assert_array_equal(out["row"], seg[b_idx * H + top] + out["rank"])
    # row_src inverts row, and rows within a segment ascend in t
    flat = out["row"].reshape(-1)
    np.testing.assert_array_equal(out["row_src"][flat], np.arange(B * T * K))
    tok = out["row_src"] // K
    for sgi in range(B * H):
        r = tok[seg[sgi]:seg[sgi + 1]]
        assert np.all(np.diff(r) > 0)


def test_all_tokens_same_heads(oracle_mod):
    # App. B.5 after Eq. (app-interaction-bounds): every token selecting the same K heads
    B, T, H, K = 2, 50, 8, 3
    s = np.tile(np.linspace(1.0, -1.0, H, dtype=np.float32), (B, T, 1))
    out = oracle_mod.route(s, K)
    expect = np.zeros((B, H), np.int32)
    expect[:, :K] = T
    np.testing.assert_array_equal(out["n"], expect)
    np.testing.assert_array_equal(out["rank"][0, :, 0], np.arange(T))


def _read_golden():
    vals = {}
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        key, *rest = line.split()
        vals[key] = [int(x) for x in rest]
    return vals


def test_fig2_worked_example(oracle_mod):
    gold = _read_golden()
    H, K = gold["H"][0], gold["K"][0]
    T = 10
    # logits realising the example: head 0 active at tokens 0, 2, 5, 6 and 8;
    # token 8 selects {0, 3}, token 9 selects {2, 3}; the others pick heads 1 and 2 or 3
    s = np.full((1, T, H), -1.0, np.float32)
    for t in range(T):
        if t in gold["head0_tokens"] or t == gold["next_head0_token"][0]:
            s[0, t, 0] = 2.0
            s[0, t, 1 + (t % 3)] = 1.0
        else:
            s[0, t, 1] = 1.0
            s[0, t, 2 + (t % 2)] = 0.5
    s[0, 8, :] = [2.0, -1.0, -1.0, 1.0]
    s[0, 9, :] = [-1.0, -1.0, 1.0, 2.0]
    out = oracle_mod.route(s, K)
    top = out["topk_head"][0]
    assert sorted(top[8].tolist()) == gold["decode_token8_heads"]
    assert sorted(top[9].tolist()) == gold["decode_token9_heads"]
    ranks0 = [int(out["rank"][0, t, list(top[t]).index(0)]) for t in gold["head0_tokens"]]
    assert ranks0 == gold["head0_ranks"]
    t8 = gold["next_head0_token"][0]
    assert int(out["rank"][0, t8, list(top[t8]).index(0)]) == gold["next_head0_rank"][0]
    # head 0's packed rows are exactly its tokens, in order (the ordered index set I_0)
    seg = out["seg_offsets"]
    toks = (out["row_src"][seg[0]:seg[1]] // K).tolist()
    assert toks == gold["head0_tokens"] + [t8]


def test_nonfinite_scores_rejected(oracle_mod):
    s = ni.router_scores(1, 1, 8, 8)
    s[0, 3, 2] = np.nan
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.route(s, 2)
    s[0, 3, 2] = np.inf
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.route(s, 2)


# --------------------------------------------------------------------------- biased selection
# App. A.3, Eq. (namoh-biased-routing): S_K(t) = TopK_i(a_{t,i} + b_i), g_{t,i} = m_{t,i} a_{t,i}.

def _affinity(scores: np.ndarray) -> np.ndarray:
    return scipy.special.softmax(scores.astype(np.float64), axis=-1)


def test_biased_zero_bias_is_plain_routing(oracle_mod):
    s = ni.router_scores(3, 2, 257, 16)
    r0 = oracle_mod.route(s, 4)
    rb = oracle_mod.route_biased(s, 4, np.zeros(16, np.float32))
    for key in ("topk_head", "rank", "row", "seg_offsets", "row_src"):
        np.testing.assert_array_equal(rb[key], r0[key])
    np.testing.assert_allclose(rb["gate"], r0["gate"], rtol=1e-15, atol=0)


def test_biased_dominant_bias_takes_slot_zero(oracle_mod):
    """A bias larger than any affinity difference puts its head first for every token; the
    other slots are the unbiased TopK of the remaining heads; the gates stay the softmax."""
    B, T, H, K, hb = 2, 200, 12, 3, 7
    s = ni.router_scores(5, B, T, H)
    bias = np.zeros(H, np.float32)
    bias[hb] = 2.0
    rb = oracle_mod.route_biased(s, K, bias)
    assert (rb["topk_head"][..., 0] == hb).all()
    others = [h for h in range(H) if h != hb]
    rest = _topk_by_counting(s[..., others], K - 1)
    np.testing.assert_array_equal(rb["topk_head"][..., 1:], np.array(others)[rest])
    a = _affinity(s)
    np.testing.assert_allclose(rb["gate"], np.take_along_axis(a, rb["topk_head"].astype(np.int64), -1),
                               rtol=1e-12, atol=0)


def test_biased_brute_force_subsets(oracle_mod):
    """On tiny routers the selected set is the K-subset with the largest sum of a + b
    (enumerated), and the slots come in decreasing a + b."""
    import itertools
    rng = np.random.default_rng(11)
    for H, K in ((5, 2), (6, 3), (7, 4)):
        s = ni.router_scores(int(rng.integers(1 << 20)), 1, 40, H)
        bias = (rng.standard_normal(H) * 0.2).astype(np.float32)
        rb = oracle_mod.route_biased(s, K, bias)
        key = _affinity(s) + bias.astype(np.float64)
        for t in range(40):
            best = max(itertools.combinations(range(H), K), key=lambda c: sum(key[0, t, list(c)]))
            assert set(rb["topk_head"][0, t].tolist()) == set(best)
            sel = key[0, t, rb["topk_head"][0, t]]
            assert (np.diff(sel) <= 0).all()


def test_biased_gates_exclude_bias(oracle_mod):
    s = ni.router_scores(8, 1, 300, 32)
    bias = (np.random.default_rng(2).standard_normal(32) * 0.05).astype(np.float32)
    rb = oracle_mod.route_biased(s, 4, bias)
    a = _affinity(s)
    np.testing.assert_allclose(rb["gate"], np.take_along_axis(a, rb["topk_head"].astype(np.int64), -1),
                               rtol=1e-12, atol=0)
    assert (rb["gate"].sum(-1) < 1.0).all()


def test_biased_ties_go_to_lower_index(oracle_mod):
    """Equal logits and equal biases give equal a + b: the lower head index comes first."""
    s = np.zeros((1, 3, 8), np.float32)
    s[0, 1, [2, 5]] = 1.0
    bias = np.zeros(8, np.float32)
    bias[[1, 6]] = 0.5
    rb = oracle_mod.route_biased(s, 3, bias)
    np.testing.assert_array_equal(rb["topk_head"][0, 0], [1, 6, 0])
    np.testing.assert_array_equal(rb["topk_head"][0, 1], [1, 6, 2])


# --------------------------------------------------------------------------- ragged batches
def _ragged_scores(seed, lens, H):
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    s = ni.router_scores(seed, 1, int(cu[-1]), H)[0] if cu[-1] > 0 else np.zeros((0, H), np.float32)
    return s, cu


@pytest.mark.parametrize("lens,H,K", [([5, 0, 300, 1, 256, 257], 8, 2), ([40, 41], 16, 4), ([0], 4, 1), ([9], 3, 3)])
def test_varlen_dispatch_matches_mask_cumsum(oracle_mod, lens, H, K):
    """Sec. 3.1 / Eq. (namoh-head-rope) per sequence of a ragged batch: ranks restart at each
    sequence's first token; n_{b,i} sums to len_b K (Eq. app-assignment-count)."""
    s, cu = _ragged_scores(11, lens, H)
    out = oracle_mod.route_varlen(s, cu, K)
    B, N = len(lens), int(cu[-1])
    top = out["topk_head"].astype(np.int64)
    mask = np.zeros((N, H), np.int64)
    if N:
        np.put_along_axis(mask, top, 1, axis=-1)
    seg = [0]
    for b in range(B):
        m = mask[cu[b]:cu[b + 1]]
        rho = np.cumsum(m, axis=0) - 1
        np.testing.assert_array_equal(out["rank"][cu[b]:cu[b + 1]], np.take_along_axis(rho, top[cu[b]:cu[b + 1]], -1))
        np.testing.assert_array_equal(out["n"][b], m.sum(0))
        assert m.sum() == lens[b] * K
        seg += list(seg[-1] + np.cumsum(m.sum(0)))
    np.testing.assert_array_equal(out["seg_offsets"], seg)
    flat = out["row"].reshape(-1)
    np.testing.assert_array_equal(out["row_src"][flat], np.arange(N * K))
    tok = out["row_src"] // K
    for sgi in range(B * H):
        r = tok[seg[sgi]:seg[sgi + 1]]
        b = sgi // H
        assert np.all(np.diff(r) > 0) and np.all((r >= cu[b]) & (r < cu[b + 1]))


def test_varlen_uniform_lengths_equal_fixed(oracle_mod):
    B, T, H, K = 3, 70, 8, 3
    s = ni.router_scores(12, B, T, H)
    fixed = oracle_mod.route(s, K)
    var = oracle_mod.route_varlen(s.reshape(B * T, H), np.arange(B + 1) * T, K)
    for key in ("topk_head", "gate", "rank", "row"):
        np.testing.assert_array_equal(var[key], fixed[key].reshape(B * T, K))
    for key in ("n", "seg_offsets", "row_src"):
        np.testing.assert_array_equal(var[key], fixed[key])


def test_varlen_rejects_bad_cu_seqlens(oracle_mod):
    s = np.zeros((10, 4), np.float32)
    for cu in ([1, 10], [0, 6, 4, 10], [0, 9]):
        with pytest.raises(oracle_mod.OracleError):
            oracle_mod.route_varlen(s, np.array(cu), 2)
