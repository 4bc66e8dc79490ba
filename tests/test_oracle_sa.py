"""Pins of the oracle's SA + NAMOH block selection (App. B.8 with the selection model of App. B.3).

What the paper fixes, each checked by a formulation unlike the oracle's:
  * Eq. (app-block-budget): N_B(r) = ceil(r / B) blocks, R(r) = ceil(alpha N_B(r)) kept, the current
    block always among them -> the kept-block count per query, computed here with exact fractions.
  * Eq. (app-selected-entries): a(r) = r - B [N_B(r) - R(r)] entries attended; Eq.
    (app-block-rounding): |a(r) - alpha r| <= B; Eq. (app-fractional-causal-sum): their sum Phi.
  * App. B.3 (end of the selection model): alpha = 1 restores dense attention within the local
    history, and a history inside one block is attended densely -> the pinned dense oracle.
  * App. B.3: MoBA scores mean-pooled keys -> the kept blocks are the top scorers by an
    independent per-query scoring routine; planted block orders whose selection and output have
    closed forms.
  * Future blocks are excluded: outputs never depend on later keys or values.
  * App. B.7 "Adopted KV-group routing": the g query heads of a group select independently over
    shared keys -> equal to g separate single-head runs.
"""
from fractions import Fraction
import math

import numpy as np
import pytest

import namoh_inputs as ni


def _case(oracle_mod, B=2, T=96, H=4, K=2, d=16, g=1, seed=3):
    wl = ni.PrefillWorkload("sa", B=B, T=T, H=H * g, K=K * g, d=d, g=g, seed=seed)
    rt = oracle_mod.route(wl.scores(), wl.Kr)
    q, k, v = wl.qkv()
    return wl, rt, q, k, v


def _kept_formula(r1, Bk, num, den):
    nb = math.ceil(Fraction(r1, Bk))
    return math.ceil(Fraction(num, den) * nb), nb


def _popcount(words):
    return np.array([sum(bin(int(w)).count("1") for w in row) for row in words])


def test_alpha_one_is_dense(oracle_mod):
    wl, rt, q, k, v = _case(oracle_mod)
    dense = oracle_mod.prefill(q, k, v, rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d, wl.g, wl.base)
    for Bk in (1, 4, 16):
        y = oracle_mod.sa_prefill(q, k, v, rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d, wl.g, wl.base,
                                  Bk, 7, 7)
        np.testing.assert_allclose(y, dense, rtol=0, atol=1e-13)


def test_history_in_one_block_is_dense(oracle_mod):
    wl, rt, q, k, v = _case(oracle_mod)
    n_max = int(np.diff(rt["seg_offsets"]).max())
    dense = oracle_mod.prefill(q, k, v, rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d, wl.g, wl.base)
    y = oracle_mod.sa_prefill(q, k, v, rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d, wl.g, wl.base,
                              n_max, 1, 5)
    np.testing.assert_allclose(y, dense, rtol=0, atol=1e-13)


@pytest.mark.parametrize("Bk,num,den", [(4, 1, 5), (8, 1, 3), (4, 2, 3), (16, 1, 4), (1, 1, 2)])
def test_kept_blocks_and_entry_count(oracle_mod, Bk, num, den):
    wl, rt, q, k, v = _case(oracle_mod, T=128)
    seg = rt["seg_offsets"]
    _, mask = oracle_mod.sa_prefill(q, k, v, seg, rt["row_src"], rt["gate"], wl.d, wl.g, wl.base, Bk, num, den,
                                    want_mask=True)
    kept = _popcount(mask)
    alpha = Fraction(num, den)
    for s in range(len(seg) - 1):
        n = int(seg[s + 1] - seg[s])
        phi = 0
        for r0 in range(n):
            r1 = r0 + 1
            R_r, nb = _kept_formula(r1, Bk, num, den)
            assert 1 <= R_r <= nb
            assert kept[seg[s] + r0] == R_r - 1
            # no block at or after the current one is marked
            cur = r0 // Bk
            for b in range(cur, 32 * mask.shape[1]):
                assert not (int(mask[seg[s] + r0, b // 32]) >> (b % 32)) & 1
            entries = Bk * (kept[seg[s] + r0]) + (r1 - Bk * (nb - 1))
            assert entries == r1 - Bk * (nb - R_r)          # Eq. (app-selected-entries)
            assert abs(entries - alpha * r1) <= Bk           # Eq. (app-block-rounding)
            phi += entries
        # Eq. (app-fractional-causal-sum): Phi = alpha n (n + 1) / 2 + sum of the rounding errors
        assert abs(phi - alpha * n * (n + 1) / 2) <= Bk * n


@pytest.mark.parametrize("g", [1, 2])
def test_kept_blocks_score_highest(oracle_mod, g):
    wl, rt, q, k, v = _case(oracle_mod, T=160, g=g, seed=5)
    seg, Bk = rt["seg_offsets"], 8
    _, mask = oracle_mod.sa_prefill(q, k, v, seg, rt["row_src"], rt["gate"], wl.d, wl.g, wl.base, Bk, 1, 4,
                                    want_mask=True)
    R = int(seg[-1])
    rows = np.repeat(np.arange(R), g)
    heads = np.tile(np.arange(g), R).astype(np.int32)
    nblk = -(-int(np.diff(seg).max()) // Bk)
    sc = oracle_mod.sa_scores_rows(q, k, seg, wl.d, g, wl.base, Bk, rows, heads, nblk)
    checked = 0
    for i in range(R * g):
        valid = ~np.isnan(sc[i])
        if not valid.any():
            continue
        bits = np.array([(int(mask[i, b // 32]) >> (b % 32)) & 1 for b in range(nblk)], bool)
        assert not (bits & ~valid).any()
        if bits.any() and (valid & ~bits).any():
            assert sc[i][bits].min() >= sc[i][valid & ~bits].max()
            checked += 1
    assert checked > 100


def test_planted_block_order(oracle_mod):
    """d = 4, RoPE off (every position 0), one head: all queries = e0, every key of block b =
    s_b e0, every value of block b = u_b e1.  Kept = the R - 1 largest s_b before the current block;
    y = gate * sum_b n_b exp(s_b / 2) u_b / sum_b n_b exp(s_b / 2) e1 (scale 1/sqrt(4))."""
    Bk, num, den, n, d = 4, 1, 3, 40, 4
    nblk = n // Bk
    s_blk = np.array([0.5, 2.0, -1.0, 1.5, 3.0, -0.5, 1.0, 2.5, 0.0, -2.0])
    u_blk = np.arange(1.0, nblk + 1.0)
    assert len(s_blk) == nblk
    q = np.zeros((n, d), np.float32); q[:, 0] = 1.0
    k = np.zeros((n, d), np.float32); k[:, 0] = np.repeat(s_blk, Bk)
    v = np.zeros((n, d), np.float32); v[:, 1] = np.repeat(u_blk, Bk)
    seg = np.array([0, n], np.int32)
    row_src = np.arange(n, dtype=np.int32)
    gate = np.linspace(0.5, 1.0, n)
    y, mask = oracle_mod.sa_prefill(ni.bf16_bits(q), ni.bf16_bits(k), ni.bf16_bits(v), seg, row_src, gate, d, 1,
                                    1e4, Bk, num, den, want_mask=True, pos=np.zeros(n, np.int64))
    for r0 in range(n):
        cur = r0 // Bk
        R_r, _ = _kept_formula(r0 + 1, Bk, num, den)
        order = sorted(range(cur), key=lambda b: -s_blk[b])[:R_r - 1]
        bits = {b for b in range(cur) if (int(mask[r0, 0]) >> b) & 1}
        assert bits == set(order)
        cnt = {b: Bk for b in order}
        cnt[cur] = r0 - cur * Bk + 1
        wts = {b: c * np.exp(s_blk[b] / 2.0) for b, c in cnt.items()}
        expect = gate[r0] * sum(wts[b] * u_blk[b] for b in wts) / sum(wts.values())
        np.testing.assert_allclose(y[r0], [0.0, expect, 0.0, 0.0], rtol=0, atol=1e-12)


def test_mask_in_reproduces_selection(oracle_mod):
    wl, rt, q, k, v = _case(oracle_mod, seed=9)
    args = (q, k, v, rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d, wl.g, wl.base, 4, 1, 3)
    y, mask = oracle_mod.sa_prefill(*args, want_mask=True)
    np.testing.assert_array_equal(oracle_mod.sa_prefill(*args, mask_in=mask), y)
    # another admissible choice changes the result: keep block 0 wherever a block is kept
    alt = mask.copy()
    alt[:, 0] |= np.where(alt[:, 0] != 0, 1, 0).astype(np.uint32)
    changed = np.abs(oracle_mod.sa_prefill(*args, mask_in=alt) - y).max(axis=1) > 0
    assert changed.any()


def test_no_dependence_on_later_entries(oracle_mod):
    wl, rt, q, k, v = _case(oracle_mod, T=64, seed=11)
    seg = rt["seg_offsets"]
    args = lambda kk, vv: (q, kk, vv, seg, rt["row_src"], rt["gate"], wl.d, wl.g, wl.base, 4, 1, 2)
    y = oracle_mod.sa_prefill(*args(k, v))
    cut = 20  # change every entry at local rank >= cut of every head
    k2, v2 = k.copy(), v.copy()
    for s in range(len(seg) - 1):
        k2[seg[s] + cut:seg[s + 1]] ^= np.uint16(0x0040)
        v2[seg[s] + cut:seg[s + 1]] ^= np.uint16(0x0040)
    y2 = oracle_mod.sa_prefill(*args(k2, v2))
    early = np.concatenate([np.arange(seg[s], min(seg[s] + cut, seg[s + 1])) for s in range(len(seg) - 1)])
    dst = rt["row_src"][early]
    np.testing.assert_array_equal(y2[dst], y[dst])
    assert np.abs(y2 - y).max() > 0


def test_groups_select_independently(oracle_mod):
    g = 2
    wl, rt, q, k, v = _case(oracle_mod, g=g, seed=13)
    args = (rt["seg_offsets"], rt["row_src"], rt["gate"], wl.d)
    y = oracle_mod.sa_prefill(q, k, v, *args, g, wl.base, 4, 1, 3).reshape(-1, g, wl.d)
    qg = q.reshape(-1, g, wl.d)
    for j in range(g):
        yj = oracle_mod.sa_prefill(np.ascontiguousarray(qg[:, j]), k, v, *args, 1, wl.base, 4, 1, 3)
        np.testing.assert_array_equal(y[:, j], yj)
