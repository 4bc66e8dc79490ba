"""GPU parity of SA + NAMOH (App. B.8 with the selection model of App. B.3).

The kept blocks decide which keys each query sees, and they are decided by fp32 scores of
bf16-rounded rotated queries and pooled keys.  So the test checks what is unique and that the rest
is valid:
  * the number of kept blocks of every query is the paper's R(r) - 1 (Eq. app-block-budget), and no
    block at or after the current one is marked;
  * every kept block scores at least as high, in the oracle's fp64 scores, as every dropped one,
    up to the bound that bf16 rounding of q~ and k~ puts on a score;
  * y equals the oracle's y computed with the GPU's kept blocks, element by element, within the
    attention tolerance; and alpha = 1 reproduces namoh_prefill bit for bit.
"""
from fractions import Fraction
import math

import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import assert_close_attention, bf16_to_f64, dev_bf16, sample_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _run(namoh, wl, block, num, den, scores=None, **rope):
    scores = wl.scores() if scores is None else scores
    q, k, v = wl.qkv()
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    y, mask, kc, _ = namoh.namoh_sa_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src,
                                            ro.gate, B=wl.B, T=wl.T, H=wl.H, K=wl.K, group=wl.g, block=block,
                                            alpha_num=num, alpha_den=den, rope_base=wl.base, status=ro.status,
                                            **rope)
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    return scores, (q, k, v), ro, y, mask.cpu().numpy().view(np.uint32), kc


def _bits(mask_row, nblk):
    return np.array([(int(mask_row[b // 32]) >> (b % 32)) & 1 for b in range(nblk)], bool)


def _check_counts(mask, seg, g, block, num, den):
    words = mask.shape[1]
    for s in range(len(seg) - 1):
        for r in range(int(seg[s + 1] - seg[s])):
            row = int(seg[s]) + r
            nb = math.ceil(Fraction(r + 1, block))
            keep = math.ceil(Fraction(num, den) * nb) - 1
            for j in range(g):
                m = mask[row * g + j]
                assert sum(bin(int(w)).count("1") for w in m) == keep, (row, j)
                cur = r // block
                for b in range(cur, 32 * words):
                    assert not (int(m[b // 32]) >> (b % 32)) & 1, (row, j, b)


def _check_scores(oracle_mod, wl, q, k, seg, mask, block, rows, interleaved=False, pos=None):
    """pos: the RoPE position of every packed row (global positions), else the local ranks."""
    g, d = wl.g, wl.d
    rows = np.repeat(np.asarray(rows, np.int64), g)
    heads = np.tile(np.arange(g, dtype=np.int32), len(rows) // g)
    nblk = -(-int(np.diff(seg).max()) // block)
    sc = oracle_mod.sa_scores_rows(q, k, seg, d, g, wl.base, block, rows, heads, nblk, interleaved=interleaved,
                                   pos=pos)
    # |q~ . mean k~ - bf16(q~) . mean bf16(k~)| <= u sum_c |q~_c| (|mean k~_c| + mean |k~_c|), u = 2^-8 for the
    # bf16 rounding; u = 2^-7 covers the fp32 rotation before it as well (+ a floor for the fp32 sums)
    seg_of = np.searchsorted(seg, rows, side="right") - 1
    local = rows - seg[seg_of]
    qrot = oracle_mod.rope(q.reshape(-1, d)[rows * g + heads], local if pos is None else pos[rows], wl.base,
                           interleaved)
    compared = 0
    for i in range(len(rows)):
        valid = ~np.isnan(sc[i])
        if not valid.any():
            continue
        kept = _bits(mask[rows[i] * g + heads[i]], nblk)
        assert not (kept & ~valid).any()
        if not kept.any() or not (valid & ~kept).any():
            continue
        s0 = int(seg[seg_of[i]])
        nb = int(valid.sum())
        kpos = np.arange(nb * block) if pos is None else pos[s0:s0 + nb * block]
        krot = oracle_mod.rope(k[s0:s0 + nb * block], kpos, wl.base, interleaved).reshape(nb, block, d)
        bound = 2.0 ** -7 * (np.abs(qrot[i]) * (np.abs(krot.mean(1)) + np.abs(krot).mean(1))).sum(1) + 1e-4
        kept_v, drop_v = kept[:nb], ~kept[:nb]
        worst_kept = np.min(sc[i][:nb][kept_v] + bound[kept_v])
        best_drop = np.max(sc[i][:nb][drop_v] - bound[drop_v])
        assert worst_kept >= best_drop, (rows[i], heads[i])
        compared += 1
    return compared


def _check_y(oracle_mod, wl, qkv, ro, y, mask, block, num, den, interleaved=False, pos=None):
    q, k, v = qkv
    seg = ro.seg_offsets.cpu().numpy()
    row_src = ro.row_src.cpu().numpy()
    gate = ro.gate.cpu().numpy().astype(np.float64)
    y_ref = oracle_mod.sa_prefill(q, k, v, seg, row_src, gate, wl.d, wl.g, wl.base, block, num, den, mask_in=mask,
                                  interleaved=interleaved, pos=pos)
    got = bf16_to_f64(y).reshape(-1, wl.d)
    assert_close_attention(got, y_ref, np.repeat(gate.reshape(-1), wl.g))
    return seg


@pytest.mark.parametrize("wl,block,num,den", [
    (ni.PrefillWorkload("sa_small", B=2, T=700, H=8, K=2, d=128, seed=21), 32, 1, 5),
    (ni.PrefillWorkload("sa_gqa_d64", B=1, T=1000, H=8, K=4, d=64, g=2, seed=22), 32, 1, 3),
    (ni.PrefillWorkload("sa_block64", B=2, T=900, H=4, K=2, d=128, seed=23), 64, 2, 5),
    (ni.PrefillWorkload("sa_block128", B=1, T=1200, H=4, K=1, d=128, seed=24), 128, 1, 2),
], ids=lambda x: getattr(x, "name", str(x)))
def test_sa_prefill_matches_oracle(namoh, oracle_mod, wl, block, num, den):
    _, qkv, ro, y, mask, _ = _run(namoh, wl, block, num, den)
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, block, num, den)
    _check_counts(mask, seg, wl.g, block, num, den)
    assert _check_scores(oracle_mod, wl, qkv[0], qkv[1], seg, mask, block, np.arange(int(seg[-1]))) > 50


@pytest.mark.parametrize("wl,block,il,gp", [
    (ni.PrefillWorkload("sa_interleaved", B=2, T=700, H=8, K=2, d=128, seed=31), 32, True, False),
    (ni.PrefillWorkload("sa_global", B=2, T=700, H=8, K=2, d=128, seed=32), 32, False, True),
    (ni.PrefillWorkload("sa_d64_block64_both", B=1, T=1500, H=4, K=2, d=64, seed=33), 64, True, True),
    (ni.PrefillWorkload("sa_d64_g4", B=1, T=900, H=8, K=4, d=64, g=4, seed=34), 32, False, False),
    (ni.PrefillWorkload("sa_g2_global", B=2, T=500, H=8, K=2, d=128, g=2, seed=35), 32, False, True),
], ids=lambda x: getattr(x, "name", str(x)))
def test_sa_rope_variants(namoh, oracle_mod, wl, block, il, gp):
    """The RoPE variants (interleaved pairs, global positions) and the head sizes and groups whose
    blocks the RoPE pass pools itself (blocks no taller than its chunks of packed rows)."""
    _, qkv, ro, y, mask, _ = _run(namoh, wl, block, 1, 4, interleaved=il, global_positions=gp)
    pos = oracle_mod.global_positions(ro.row_src.cpu().numpy(), wl.T, wl.Kr) if gp else None
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, block, 1, 4, interleaved=il, pos=pos)
    _check_counts(mask, seg, wl.g, block, 1, 4)
    assert _check_scores(oracle_mod, wl, qkv[0], qkv[1], seg, mask, block, np.arange(int(seg[-1])),
                         interleaved=il, pos=pos) > 50


def test_sa_alpha_one_is_prefill(namoh):
    wl = ni.PrefillWorkload("sa_dense", B=2, T=640, H=8, K=2, d=128, seed=25)
    _, qkv, ro, y, mask, _ = _run(namoh, wl, 32, 1, 1)
    q, k, v = qkv
    y2, _, _ = namoh.namoh_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src, ro.gate,
                                   B=wl.B, T=wl.T, H=wl.H, K=wl.K, rope_base=wl.base)
    torch.cuda.synchronize()
    assert torch.equal(y, y2)


def test_sa_short_and_empty_histories(namoh, oracle_mod):
    """Zipf-biased routing with planted logits: head 15 never wins (an empty history), head 14 wins
    20 tokens (a history shorter than one block), head 13 wins 40 (one complete block and a tail)."""
    wl = ni.PrefillWorkload("sa_skew", B=1, T=600, H=16, K=2, d=128, zipf_bias=True, seed=26)
    scores = wl.scores().copy()
    scores[..., 13:] = -30.0
    scores[0, 100:120, 14] = 30.0
    scores[0, 300:340, 13] = 30.0
    _, qkv, ro, y, mask, _ = _run(namoh, wl, 32, 1, 4, scores=scores)
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, 32, 1, 4)
    n = np.diff(seg)
    assert (n == 0).any() and ((n > 0) & (n < 32)).any()
    _check_counts(mask, seg, wl.g, 32, 1, 4)


def test_sa_full_size_balanced(namoh, oracle_mod):
    """The balanced workload (B4 T4096 H16 K4 d128) at alpha = 1/5, 32-key blocks: every output
    against the oracle with the GPU's kept blocks; counts everywhere; scores on sampled rows."""
    wl = ni.BALANCED
    _, qkv, ro, y, mask, _ = _run(namoh, wl, 32, 1, 5)
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, 32, 1, 5)
    rows = sample_rows(seg, 300, seed=3)
    words = mask.shape[1]
    for row in rows:
        s = int(np.searchsorted(seg, row, side="right") - 1)
        r = int(row - seg[s])
        keep = math.ceil(Fraction(1, 5) * math.ceil(Fraction(r + 1, 32))) - 1
        assert sum(bin(int(w)).count("1") for w in mask[row]) == keep
        for b in range(r // 32, 32 * words):
            assert not (int(mask[row, b // 32]) >> (b % 32)) & 1
    assert _check_scores(oracle_mod, wl, qkv[0], qkv[1], seg, mask, 32, rows) > 100


def test_sa_rejects_bad_arguments(namoh):
    wl = ni.PrefillWorkload("sa_args", B=1, T=256, H=4, K=1, d=128, seed=27)
    q, k, v = wl.qkv()
    ro = namoh.namoh_route(torch.from_numpy(wl.scores()).cuda(), wl.Kr)
    args = (dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src, ro.gate)
    for kw in (dict(block=48), dict(block=16), dict(alpha_num=0), dict(alpha_num=3, alpha_den=2)):
        with pytest.raises(namoh.NamohError):
            namoh.namoh_sa_prefill(*args, B=wl.B, T=wl.T, H=wl.H, K=wl.K, **kw)


def test_sa_segment_over_capacity(namoh, oracle_mod):
    """Caches at seg_base with one segment one row too small: the status reports it, that segment's
    rows are neither pooled nor attended, and every other segment matches the oracle."""
    wl = ni.PrefillWorkload("sa_capacity", B=2, T=600, H=4, K=2, d=128, seed=28)
    block, num, den = 32, 1, 4
    scores = wl.scores()
    q, k, v = wl.qkv()
    ref = oracle_mod.route(scores, wl.Kr)
    seg = ref["seg_offsets"].astype(np.int64)
    nseg = len(seg) - 1
    n = seg[1:] - seg[:-1]
    head = 40
    seg_base = seg[:-1] + np.arange(nseg) * head
    cap = (n + head).astype(np.int32)
    over = int(np.argmax(n))
    cap[over] = n[over] - 1
    rows = int(seg[-1] + nseg * head)
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    kc = torch.zeros((rows, wl.d), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    y, mask, _, _ = namoh.namoh_sa_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src,
                                           ro.gate, B=wl.B, T=wl.T, H=wl.H, K=wl.K, block=block, alpha_num=num,
                                           alpha_den=den, rope_base=wl.base, k_cache=kc, v_cache=vc,
                                           seg_base=torch.from_numpy(seg_base).cuda(),
                                           seg_cap=torch.from_numpy(cap).cuda(), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & namoh.NAMOH_DEV_CAPACITY
    mask = mask.cpu().numpy().view(np.uint32)
    assert not mask[seg[over]:seg[over + 1]].any()  # nothing selected in the skipped history
    gate = ref["gate"].astype(np.float64)
    y_ref = oracle_mod.sa_prefill(q, k, v, seg, ref["row_src"], gate, wl.d, 1, wl.base, block, num, den,
                                  mask_in=mask)
    keep = np.concatenate([np.arange(seg[s_], seg[s_ + 1]) for s_ in range(nseg) if s_ != over])
    dst = ref["row_src"][keep]
    assert_close_attention(bf16_to_f64(y).reshape(-1, wl.d)[dst], y_ref[dst], gate.reshape(-1)[dst])
    keep_mask = np.concatenate([np.arange(seg[s_], seg[s_ + 1]) for s_ in range(nseg) if s_ != over])
    _check_counts_rows(mask, seg, keep_mask, block, num, den)


def _check_counts_rows(mask, seg, rows, block, num, den):
    for row in rows:
        s = int(np.searchsorted(seg, row, side="right") - 1)
        r = int(row - seg[s])
        keep = math.ceil(Fraction(num, den) * math.ceil(Fraction(r + 1, block))) - 1
        assert sum(bin(int(w)).count("1") for w in mask[row]) == keep, row


@pytest.mark.parametrize("num,den", [(1, 2), (3, 4)], ids=["alpha_1_2", "alpha_3_4"])
def test_sa_long_histories_many_kept(namoh, oracle_mod, num, den):
    """Histories of about 2048 rows (64 blocks of 32): a query keeps up to 31 blocks (alpha 1/2), or
    drops up to 16 (alpha 3/4), more than the selector's 8-entry register list, so the kept set is
    found by bisection over the selection keys."""
    wl = ni.PrefillWorkload("sa_long", B=1, T=4096, H=2, K=1, d=128, seed=29)
    _, qkv, ro, y, mask, _ = _run(namoh, wl, 32, num, den)
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, 32, num, den)
    _check_counts(mask, seg, wl.g, 32, num, den)
    rows = sample_rows(seg, 200, seed=5)
    assert _check_scores(oracle_mod, wl, qkv[0], qkv[1], seg, mask, 32, rows) > 100


def test_sa_history_longer_than_the_tmem_scores(namoh, oracle_mod):
    """One history of 17000 rows (532 blocks of 32): rows whose current block is past the 512 block
    scores one selection CTA holds in TMEM take the per-query selector; both meet at block 512."""
    wl = ni.PrefillWorkload("sa_very_long", B=1, T=17000, H=1, K=1, d=64, seed=30)
    _, qkv, ro, y, mask, _ = _run(namoh, wl, 32, 1, 5)
    seg = _check_y(oracle_mod, wl, qkv, ro, y, mask, 32, 1, 5)
    _check_counts(mask, seg, wl.g, 32, 1, 5)
    rows = np.concatenate([sample_rows(seg, 100, seed=6), np.arange(512 * 32 - 40, 513 * 32 + 40)])
    assert _check_scores(oracle_mod, wl, qkv[0], qkv[1], seg, np.asarray(mask), 32, np.unique(rows)) > 100
