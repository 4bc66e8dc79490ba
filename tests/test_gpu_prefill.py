"""GPU parity of prefill (RoPE at rank, routed causal attention, gate-weighted combine).

Sec. 3.2 Eq. (namoh-head-rope); Sec. 3.1 Eq. (namoh-attention); App. B.7 KV-group routing.
Every case, the full-size workloads included, compares every output element (and every
rotated key written to the cache) with the oracle.
"""
import numpy as np
import pytest
import torch

import namoh_inputs as ni
from _gpu_helpers import assert_close_attention, bf16_to_f64, dev_bf16, host_bf16_bits

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _run_gpu(namoh, wl: ni.PrefillWorkload, scores, q, k, v, **kw):
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    y, kc, vc = namoh.namoh_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src, ro.gate,
                                    B=wl.B, T=wl.T, H=wl.H, K=wl.K, group=wl.g, rope_base=wl.base,
                                    status=ro.status, **kw)
    torch.cuda.synchronize()
    return ro, y, kc, vc


def _variant(name: str) -> dict:
    """RoPE variant keywords of namoh_prefill (Sec. 3.2: global positions replace the rank)."""
    return dict(interleaved="interleaved" in name, global_positions=name.startswith("global"))


def _full_check(namoh, oracle_mod, wl: ni.PrefillWorkload, scores=None, variant: str = "rank"):
    scores = wl.scores() if scores is None else scores
    q, k, v = wl.qkv()
    kw = _variant(variant)
    ro, y, kc, _ = _run_gpu(namoh, wl, scores, q, k, v, **kw)
    assert int(ro.status.item()) == 0
    ref = oracle_mod.route(scores, wl.Kr)
    np.testing.assert_array_equal(ro.seg_offsets.cpu().numpy(), ref["seg_offsets"])
    pos = oracle_mod.global_positions(ref["row_src"], wl.T, wl.Kr) if kw["global_positions"] else None
    y_ref, krot = oracle_mod.prefill(q, k, v, ref["seg_offsets"], ref["row_src"], ref["gate"], wl.d, wl.g, wl.base,
                                     return_krot=True, interleaved=kw["interleaved"], pos=pos)
    got = bf16_to_f64(y).reshape(-1, wl.d)
    gate = np.repeat(ref["gate"].reshape(-1), wl.g)
    assert_close_attention(got, y_ref, gate)
    # rotated keys in the cache: bf16 rounding of the rotation (within one bf16 ulp of the
    # fp64 value, plus the fp32 rotation's absolute error where x cos - y sin cancels)
    kc_got = bf16_to_f64(kc)
    assert np.all(np.abs(kc_got - krot) <= np.abs(krot) * 2.0 ** -7 + 1e-6)
    return got, y_ref


@pytest.mark.parametrize("wl", [
    ni.PR1,
    ni.PrefillWorkload("small_d128", B=2, T=700, H=4, K=2, d=128),
    ni.PrefillWorkload("small_d64_ragged", B=3, T=333, H=6, K=3, d=64, seed=3),
    ni.PrefillWorkload("dense_k_eq_h", B=1, T=300, H=4, K=4, d=128, seed=4),
    ni.PrefillWorkload("one_token", B=2, T=1, H=8, K=2, d=128, seed=5),
    ni.PrefillWorkload("gqa_g2", B=1, T=500, H=8, K=4, d=128, g=2, seed=6),
    ni.PrefillWorkload("gqa_g8", B=1, T=400, H=64, K=32, d=128, g=8, seed=7),
    ni.PrefillWorkload("gqa_g4_d64", B=2, T=260, H=16, K=8, d=64, g=4, seed=8),
    ni.PrefillWorkload("base5e5_long_segment", B=1, T=2500, H=4, K=1, d=128, base=500000.0, seed=9),
], ids=lambda w: w.name)
def test_prefill_matches_oracle(namoh, oracle_mod, wl):
    _full_check(namoh, oracle_mod, wl)


def test_prefill_empty_heads_and_one_long_segment(namoh, oracle_mod):
    """All tokens on head 2 (n = T there, n = 0 elsewhere): empty segments have no work."""
    wl = ni.PrefillWorkload("single_head", B=2, T=1100, H=8, K=1, d=128, seed=10)
    s = np.full((2, 1100, 8), -1.0, np.float32)
    s[..., 2] = 1.0
    _full_check(namoh, oracle_mod, wl, scores=s)


def test_prefill_cache_layout_with_headroom_and_capacity(namoh, oracle_mod):
    """Caches at seg_base with headroom; unwritten rows hold NaN patterns that must not leak."""
    wl = ni.PrefillWorkload("cache_layout", B=2, T=600, H=4, K=2, d=128, seed=11)
    scores = wl.scores()
    q, k, v = wl.qkv()
    ref = oracle_mod.route(scores, wl.Kr)
    seg = ref["seg_offsets"].astype(np.int64)
    nseg = len(seg) - 1
    head = 37
    n = seg[1:] - seg[:-1]
    seg_base = seg[:-1] + np.arange(nseg) * head
    cap = (n + head).astype(np.int32)
    rows = int(seg[-1] + nseg * head)
    nan_bits = torch.full((rows, wl.d), -1, dtype=torch.int16, device="cuda").view(torch.bfloat16)  # 0xFFFF = NaN
    kc, vc = nan_bits.clone(), nan_bits.clone()
    seg_len = torch.zeros(nseg, dtype=torch.int32, device="cuda")
    ro, y, _, _ = _run_gpu(namoh, wl, scores, q, k, v, k_cache=kc, v_cache=vc,
                           seg_base=torch.from_numpy(seg_base).cuda(), seg_cap=torch.from_numpy(cap).cuda(),
                           seg_len=seg_len)
    assert int(ro.status.item()) == 0
    np.testing.assert_array_equal(seg_len.cpu().numpy(), n)
    y_ref = oracle_mod.prefill(q, k, v, ref["seg_offsets"], ref["row_src"], ref["gate"], wl.d, 1, wl.base)
    assert_close_attention(bf16_to_f64(y).reshape(-1, wl.d), y_ref, ref["gate"].reshape(-1))
    vc_bits = host_bf16_bits(vc)
    for s_ in range(nseg):
        np.testing.assert_array_equal(vc_bits[seg_base[s_]:seg_base[s_] + n[s_]], v[seg[s_]:seg[s_ + 1]])
    # one segment too small: the status reports it, the other segments are unaffected
    cap2 = cap.copy()
    cap2[1] = n[1] - 1
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ro2 = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    y2, _, _ = namoh.namoh_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro2.seg_offsets, ro2.row_src, ro2.gate,
                                   B=wl.B, T=wl.T, H=wl.H, K=wl.K, rope_base=wl.base, k_cache=nan_bits.clone(),
                                   v_cache=nan_bits.clone(), seg_base=torch.from_numpy(seg_base).cuda(),
                                   seg_cap=torch.from_numpy(cap2).cuda(), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & namoh.NAMOH_DEV_CAPACITY
    keep = np.concatenate([ref["row_src"][seg[s_]:seg[s_ + 1]] for s_ in range(nseg) if s_ != 1])
    got = bf16_to_f64(y2).reshape(-1, wl.d)[keep]
    assert_close_attention(got, y_ref[keep], ref["gate"].reshape(-1)[keep])


@pytest.mark.parametrize("wl", [ni.BALANCED, ni.SKEWED, *ni.H_SWEEP, ni.GQA], ids=lambda w: w.name)
def test_prefill_full_size(namoh, oracle_mod, wl):
    """The full-size workloads in the launch configuration the benchmark times: every output
    element against the oracle (long items, several items per CTA, TMEM and ring reuse across
    items only happen at these sizes), and every rotated key in the cache."""
    _full_check(namoh, oracle_mod, wl)


VARIANTS = ["interleaved", "global", "global_interleaved"]


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("wl", [
    ni.PrefillWorkload("small_d128", B=2, T=700, H=4, K=2, d=128),
    ni.PrefillWorkload("small_d64_ragged", B=3, T=333, H=6, K=3, d=64, seed=3),
    ni.PrefillWorkload("gqa_g4_d64", B=2, T=260, H=16, K=8, d=64, g=4, seed=8),
    ni.PrefillWorkload("base5e5_long_segment", B=1, T=2500, H=4, K=1, d=128, base=500000.0, seed=9),
], ids=lambda w: w.name)
def test_prefill_rope_variants_match_oracle(namoh, oracle_mod, wl, variant):
    """Interleaved pairing and global positions (t instead of rho), against the oracle in the
    same variant: outputs and the rotated keys in the cache."""
    _full_check(namoh, oracle_mod, wl, variant=variant)


def test_prefill_k_equals_h_global_is_rank(namoh):
    """K = H: every rank is t, so global positions give the same bytes."""
    wl = ni.PrefillWorkload("dense_k_eq_h", B=1, T=300, H=4, K=4, d=128, seed=4)
    scores = wl.scores()
    q, k, v = wl.qkv()
    _, y0, kc0, _ = _run_gpu(namoh, wl, scores, q, k, v)
    _, y1, kc1, _ = _run_gpu(namoh, wl, scores, q, k, v, global_positions=True)
    assert torch.equal(y0.view(torch.int16), y1.view(torch.int16))
    assert torch.equal(kc0.view(torch.int16), kc1.view(torch.int16))


@pytest.mark.parametrize("variant", ["interleaved", "global", "global_interleaved"])
def test_prefill_full_size_variants(namoh, oracle_mod, variant):
    """Global positions reach T - 1 (32767 here, base 5e5) instead of about T K / H; every
    output of the skewed workload against the oracle in the same variant."""
    _full_check(namoh, oracle_mod, ni.SKEWED, variant=variant)


def test_prefill_many_segments_unstaged(namoh, oracle_mod):
    """B*H = 8320 segments: more offsets than the RoPE kernel stages in shared memory and a
    plan too large to build inside the RoPE launch (separate plan kernel)."""
    _full_check(namoh, oracle_mod, ni.PrefillWorkload("many_segments", B=130, T=64, H=64, K=2, d=64, seed=11))


@pytest.mark.parametrize("wl", [ni.PR1, ni.PrefillWorkload("gqa_g4_staged", B=2, T=900, H=16, K=8, d=128, g=4, seed=12)],
                         ids=lambda w: w.name)
@pytest.mark.parametrize("variant", ["rank", "global_interleaved"])
def test_staged_calls_match_prefill(namoh, wl, variant):
    """namoh_rope_pack (building the plan in the same launch, or not) + namoh_attention give
    the bytes namoh_prefill gives."""
    scores = wl.scores()
    q, k, v = (dev_bf16(a) for a in wl.qkv())
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    vkw = _variant(variant)
    y_ref, _, _ = namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, B=wl.B, T=wl.T, H=wl.H, K=wl.K,
                                      group=wl.g, rope_base=wl.base, status=ro.status, **vkw)
    kw = dict(B=wl.B, T=wl.T, H=wl.H, K=wl.K, group=wl.g)
    rkw = dict(interleaved=vkw["interleaved"], row_src=ro.row_src if vkw["global_positions"] else None)
    for fused in (True, False):
        plan = namoh.namoh_attention_plan(ro.seg_offsets, **kw)
        plan.fill_(0xAB)  # stale bytes: the fused launch must rebuild every word it uses
        if fused:
            q_rot, kc, vc = namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, rope_base=wl.base, status=ro.status,
                                                  plan=plan, **kw, **rkw)
        else:
            q_rot, kc, vc = namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, rope_base=wl.base, status=ro.status,
                                                  **kw, **rkw)
            namoh.namoh_attention_plan(ro.seg_offsets, plan=plan, **kw)
        y = namoh.namoh_attention(q_rot, kc, vc, ro.seg_offsets, ro.row_src, ro.gate, plan, status=ro.status, **kw)
        torch.cuda.synchronize()
        assert torch.equal(y.view(torch.int16), y_ref.view(torch.int16)), f"fused plan = {fused}"
    assert int(ro.status.item()) == 0


def test_attention_output_not_sector_aligned(namoh):
    """y only 16-byte aligned (not 32): rows take the 16-byte store path, same bytes."""
    wl = ni.PrefillWorkload("y_offset", B=2, T=600, H=8, K=2, d=128, seed=13)
    scores = wl.scores()
    q, k, v = (dev_bf16(a) for a in wl.qkv())
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), wl.Kr)
    kw = dict(B=wl.B, T=wl.T, H=wl.H, K=wl.K, group=wl.g)
    y_ref, _, _ = namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, rope_base=wl.base,
                                      status=ro.status, **kw)
    numel = wl.B * wl.T * wl.K * wl.d
    big = torch.empty(numel + 8, dtype=torch.bfloat16, device="cuda")
    y_off = big[8:].view(wl.B, wl.T, wl.K, wl.d)
    assert y_off.data_ptr() % 32 == 16
    y, _, _ = namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, rope_base=wl.base, y=y_off,
                                  status=ro.status, **kw)
    torch.cuda.synchronize()
    assert torch.equal(y.view(torch.int16), y_ref.view(torch.int16))
    assert int(ro.status.item()) == 0
