"""GPU parity of the decode step (Sec. 3.1 last paragraph; Sec. 3.2 "Efficient execution").

Each new token routes (T = 1), appends k~ and v to its selected heads' caches at rank
seg_len, attends over seg_len + 1 rows, writes g * h and bumps seg_len.
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


def _variant(name: str) -> dict:
    return dict(interleaved="interleaved" in name, global_positions=name.startswith("global"))


def _prefix_state(namoh, B, T, Hr, Kr, d, g, base, headroom, seed, variant="rank"):
    """GPU prefill of a T-token prefix into caches with `headroom` free rows per segment."""
    scores = ni.router_scores(seed, B, T, Hr)
    R = B * T * Kr
    q, k, v = ni.qkv_rows(seed, R, d, g)
    ro = namoh.namoh_route(torch.from_numpy(scores).cuda(), Kr)
    seg = ro.seg_offsets.cpu().numpy().astype(np.int64)
    nseg = B * Hr
    seg_base = seg[:-1] + np.arange(nseg) * headroom
    n = seg[1:] - seg[:-1]
    cap = (n + headroom).astype(np.int32)
    rows = int(seg[-1] + nseg * headroom)
    kc = torch.zeros((rows, d), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros((rows, d), dtype=torch.bfloat16, device="cuda")
    seg_len = torch.zeros(nseg, dtype=torch.int32, device="cuda")
    namoh.namoh_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src, ro.gate, B=B, T=T,
                        H=Hr * g, K=Kr * g, group=g, rope_base=base, k_cache=kc, v_cache=vc,
                        seg_base=torch.from_numpy(seg_base).cuda(), seg_cap=torch.from_numpy(cap).cuda(),
                        seg_len=seg_len, status=ro.status, **_variant(variant))
    torch.cuda.synchronize()
    assert int(ro.status.item()) == 0
    return dict(kc=kc, vc=vc, seg_len=seg_len, seg_base=seg_base, cap=cap, n=n, rows=rows,
                seg_base_d=torch.from_numpy(seg_base).cuda(), cap_d=torch.from_numpy(cap).cuda(),
                host=dict(scores=scores, q=q, k=k, v=v, T=T, Kr=Kr, d=d, g=g, base=base, variant=variant))


def _oracle_caches(oracle_mod, st):
    """The oracle's own prefix state: its routing of the prefix, its fp64 rotated keys and the exact
    values, laid out at the same segment bases (nothing is taken from the GPU's caches)."""
    h = st["host"]
    d = h["d"]
    ref = oracle_mod.route(h["scores"], h["Kr"])
    vkw = _variant(h["variant"])
    pos = oracle_mod.global_positions(ref["row_src"], h["T"], h["Kr"]) if vkw["global_positions"] else None
    _, krot = oracle_mod.prefill(h["q"], h["k"], h["v"], ref["seg_offsets"], ref["row_src"], ref["gate"], d, h["g"],
                                 h["base"], return_krot=True, interleaved=vkw["interleaved"], pos=pos)
    seg = ref["seg_offsets"].astype(np.int64)
    vals = ni.bf16_to_f32(h["v"]).astype(np.float64)
    kc = np.zeros((st["rows"], d))
    vc = np.zeros((st["rows"], d))
    base = st["seg_base"].astype(np.int64).copy()
    for s_ in range(len(seg) - 1):
        lo, hi = int(seg[s_]), int(seg[s_ + 1])
        kc[base[s_]:base[s_] + hi - lo] = krot[lo:hi]
        vc[base[s_]:base[s_] + hi - lo] = vals[lo:hi]
    return kc, vc, base, (seg[1:] - seg[:-1]).astype(np.int32), st["cap"].astype(np.int32).copy()


@pytest.mark.parametrize("B,T,Hr,Kr,d,g,steps", [
    (3, 300, 8, 2, 128, 1, 5),
    (2, 257, 4, 4, 64, 1, 3),
    (2, 200, 4, 2, 128, 2, 4),
    (1, 130, 8, 1, 128, 8, 3),
    (64, 40, 32, 4, 128, 1, 2),
])
def test_decode_matches_oracle(namoh, oracle_mod, B, T, Hr, Kr, d, g, steps):
    _decode_check(namoh, oracle_mod, B, T, Hr, Kr, d, g, steps, "rank")


def _token_positions(B, T, t, steps):
    """Distinct per-sequence token indices, up to the largest the ABI accepts (2^24 - 1)."""
    tp = [T + t] + [131072 * b + 11 * b + t for b in range(1, B - 1)] + ([(1 << 24) - steps + t] if B > 1 else [])
    return np.array(tp, np.int64)


def _decode_check(namoh, oracle_mod, B, T, Hr, Kr, d, g, steps, variant):
    base = 10000.0
    vkw = _variant(variant)
    st = _prefix_state(namoh, B, T, Hr, Kr, d, g, base, steps, seed=21, variant=variant)
    okc, ovc, obase, olen, ocap = _oracle_caches(oracle_mod, st)
    sc, q, k, v = ni.decode_step_inputs(22, steps, B, Hr, Kr, d, g)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for t in range(steps):
        tp = _token_positions(B, T, t, steps) if vkw["global_positions"] else None
        ro = namoh.namoh_route(torch.from_numpy(sc[t][:, None, :]).cuda(), Kr, compact=False)
        y = namoh.namoh_decode(ro.topk_head.view(B, Kr), ro.gate.view(B, Kr), dev_bf16(q[t]), dev_bf16(k[t]),
                               dev_bf16(v[t]), H=Hr * g, K=Kr * g, group=g, rope_base=base, k_cache=st["kc"],
                               v_cache=st["vc"], seg_base=st["seg_base_d"], seg_len=st["seg_len"],
                               seg_cap=st["cap_d"], status=status, interleaved=vkw["interleaved"],
                               token_pos=None if tp is None else torch.from_numpy(tp).cuda())
        torch.cuda.synchronize()
        ref = oracle_mod.route(sc[t][:, None, :], Kr)
        np.testing.assert_array_equal(ro.topk_head.cpu().numpy(), ref["topk_head"])
        y_ref = oracle_mod.decode_step(ref["topk_head"][:, 0], ref["gate"][:, 0], q[t], k[t], v[t], Hr, d, g, base,
                                       okc, ovc, obase, olen, ocap, interleaved=vkw["interleaved"], token_pos=tp)
        gate = np.repeat(ref["gate"][:, 0], g, axis=1)
        assert_close_attention(bf16_to_f64(y), y_ref, gate, what=f"step {t}")
        np.testing.assert_array_equal(st["seg_len"].cpu().numpy(), olen)
    assert int(status.item()) == 0
    # M_KV = T K after the prefix and + K per step (App. B.5 Eq. app-routed-kv)
    assert int(st["seg_len"].sum().item()) == B * (T + steps) * Kr
    # the appended keys: the oracle's k~ rounded to bf16
    kc_got = bf16_to_f64(st["kc"])
    for s_ in range(len(olen)):
        lo, hi = int(obase[s_]), int(obase[s_] + olen[s_])
        assert np.all(np.abs(kc_got[lo:hi] - okc[lo:hi]) <= np.abs(okc[lo:hi]) * 2.0 ** -7 + 1e-6)


@pytest.mark.parametrize("variant", ["interleaved", "global", "global_interleaved"])
@pytest.mark.parametrize("B,T,Hr,Kr,d,g,steps", [
    (3, 300, 8, 2, 128, 1, 3),
    (2, 257, 4, 4, 64, 1, 2),
    (2, 200, 4, 2, 128, 2, 3),
])
def test_decode_rope_variants_match_oracle(namoh, oracle_mod, B, T, Hr, Kr, d, g, steps, variant):
    """Interleaved pairing, and global positions from token_pos (Sec. 3.2: t instead of rho)."""
    _decode_check(namoh, oracle_mod, B, T, Hr, Kr, d, g, steps, variant)


@pytest.mark.parametrize("variant", ["rank", "global_interleaved"])
def test_prefill_then_decode_equals_longer_prefill(namoh, oracle_mod, variant):
    """Prefill over T tokens plus decode steps reproduces prefill over T + steps tokens."""
    B, T, Hr, Kr, d, steps, base = 2, 200, 8, 2, 128, 3, 10000.0
    vkw = _variant(variant)
    Tt = T + steps
    s = ni.router_scores(31, B, Tt, Hr)
    R = B * Tt * Kr
    q, k, v = ni.qkv_rows(31, R, d)
    ref = oracle_mod.route(s, Kr)
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), Kr)
    y_full, _, _ = namoh.namoh_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), ro.seg_offsets, ro.row_src, ro.gate,
                                       B=B, T=Tt, H=Hr, K=Kr, rope_base=base, **vkw)
    # prefix rows: the packed rows of tokens < T keep their order
    tok = ref["row_src"] // Kr % Tt
    keep = np.nonzero(tok < T)[0]
    ro_p = namoh.namoh_route(torch.from_numpy(np.ascontiguousarray(s[:, :T])).cuda(), Kr)
    seg = ro_p.seg_offsets.cpu().numpy().astype(np.int64)
    nseg = B * Hr
    seg_base = seg[:-1] + np.arange(nseg) * steps
    cap = (seg[1:] - seg[:-1] + steps).astype(np.int32)
    rows = int(seg[-1] + nseg * steps)
    kc = torch.zeros((rows, d), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    seg_len = torch.zeros(nseg, dtype=torch.int32, device="cuda")
    sb, cp = torch.from_numpy(seg_base).cuda(), torch.from_numpy(cap).cuda()
    namoh.namoh_prefill(dev_bf16(q[keep]), dev_bf16(k[keep]), dev_bf16(v[keep]), ro_p.seg_offsets, ro_p.row_src,
                        ro_p.gate, B=B, T=T, H=Hr, K=Kr, rope_base=base, k_cache=kc, v_cache=vc, seg_base=sb,
                        seg_cap=cp, seg_len=seg_len, **vkw)
    yf = bf16_to_f64(y_full).reshape(B, Tt, Kr, d)
    for t in range(T, Tt):
        rows_t = ref["row"][:, t]
        yd = namoh.namoh_decode(ro.topk_head[:, t].contiguous(), ro.gate[:, t].contiguous(), dev_bf16(q[rows_t]),
                                dev_bf16(k[rows_t]), dev_bf16(v[rows_t]), H=Hr, K=Kr, rope_base=base, k_cache=kc,
                                v_cache=vc, seg_base=sb, seg_len=seg_len, seg_cap=cp,
                                interleaved=vkw["interleaved"],
                                token_pos=torch.full((B,), t, dtype=torch.int64, device="cuda")
                                if vkw["global_positions"] else None)
        torch.cuda.synchronize()
        assert_close_attention(bf16_to_f64(yd), yf[:, t], ref["gate"][:, t], what=f"token {t}")


def test_decode_full_segment_sets_capacity(namoh):
    B, T, Hr, Kr, d = 2, 100, 4, 2, 128
    st = _prefix_state(namoh, B, T, Hr, Kr, d, 1, 1e4, 0, seed=41)  # no headroom: every segment is full
    sc, q, k, v = ni.decode_step_inputs(42, 1, B, Hr, Kr, d)
    ro = namoh.namoh_route(torch.from_numpy(sc[0][:, None, :]).cuda(), Kr, compact=False)
    before = st["seg_len"].clone()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    y = namoh.namoh_decode(ro.topk_head.view(B, Kr), ro.gate.view(B, Kr), dev_bf16(q[0]), dev_bf16(k[0]),
                           dev_bf16(v[0]), H=Hr, K=Kr, k_cache=st["kc"], v_cache=st["vc"], seg_base=st["seg_base_d"],
                           seg_len=st["seg_len"], seg_cap=st["cap_d"], status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & namoh.NAMOH_DEV_CAPACITY
    assert torch.equal(st["seg_len"], before)
    assert float(y.float().abs().max().item()) == 0.0


def test_decode_full_size(namoh, oracle_mod):
    """64 sequences with 131072-token routed prefixes (H = 32, K = 4, d = 128): the 17 GB cache
    is seeded N(0, 1) bf16 on the device (already-rotated keys and values); two decode steps.
    Every sequence and slot of both steps is compared with the oracle, which continues from the
    seeded prefix rows and from the rows it appended itself (never from rows the GPU wrote)."""
    wl = ni.DECODE
    B, Hr, Kr, d = wl.B, wl.Hr, wl.Kr, wl.d
    s = ni.router_scores(wl.seed, B, wl.prefix, Hr)
    ro = namoh.namoh_route(torch.from_numpy(s).cuda(), Kr)
    del s
    seg = ro.seg_offsets.cpu().numpy().astype(np.int64)
    del ro
    steps = 2
    nseg = B * Hr
    n = seg[1:] - seg[:-1]
    seg_base = seg[:-1] + np.arange(nseg) * steps
    cap = (n + steps).astype(np.int32)
    rows = int(seg[-1] + nseg * steps)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(wl.seed)
    kc = torch.randn((rows, d), generator=gen, device="cuda", dtype=torch.bfloat16)
    vc = torch.randn((rows, d), generator=gen, device="cuda", dtype=torch.bfloat16)
    # the seeded prefix of every segment, as the oracle reads it: rows base .. base + n - 1 are
    # never rewritten by decode (it appends after them), so they can be copied when first needed
    seg_len = torch.from_numpy(n.astype(np.int32)).cuda()
    sb, cp = torch.from_numpy(seg_base).cuda(), torch.from_numpy(cap).cuda()
    sc, q, k, v = ni.decode_step_inputs(wl.seed, steps, B, Hr, Kr, d)
    appended = {}  # segment -> (k~ rows, v rows) the oracle appended, fp64
    o_len = n.astype(np.int32).copy()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for t in range(steps):
        rt = namoh.namoh_route(torch.from_numpy(sc[t][:, None, :]).cuda(), Kr, compact=False)
        y = namoh.namoh_decode(rt.topk_head.view(B, Kr), rt.gate.view(B, Kr), dev_bf16(q[t]), dev_bf16(k[t]),
                               dev_bf16(v[t]), H=Hr, K=Kr, rope_base=wl.base, k_cache=kc, v_cache=vc, seg_base=sb,
                               seg_len=seg_len, seg_cap=cp, status=status)
        torch.cuda.synchronize()
        ref = oracle_mod.route(sc[t][:, None, :], Kr)
        np.testing.assert_array_equal(rt.topk_head.view(B, Kr).cpu().numpy(), ref["topk_head"][:, 0])
        top, gate = ref["topk_head"][:, 0], ref["gate"][:, 0]
        yh = bf16_to_f64(y)
        for b in range(B):
            # this sequence's selected histories as a small cache: segment i = slot i
            lens, parts_k, parts_v = [], [], []
            for slot in range(Kr):
                sidx = b * Hr + int(top[b, slot])
                lo = int(seg_base[sidx])
                pk = bf16_to_f64(kc[lo:lo + int(n[sidx])])
                pv = bf16_to_f64(vc[lo:lo + int(n[sidx])])
                ak, av = appended.get(sidx, ([], []))
                parts_k.append(np.concatenate([pk] + [a[None] for a in ak] + [np.zeros((1, d))]))
                parts_v.append(np.concatenate([pv] + [a[None] for a in av] + [np.zeros((1, d))]))
                lens.append(int(n[sidx]) + len(ak))
                assert lens[-1] == o_len[sidx]
            okc, ovc = np.ascontiguousarray(np.concatenate(parts_k)), np.ascontiguousarray(np.concatenate(parts_v))
            caps = np.array([len(p_) for p_ in parts_k], np.int32)
            bases = np.concatenate([[0], np.cumsum(caps)[:-1]]).astype(np.int64)
            olen_b = np.array(lens, np.int32)
            y_ref = oracle_mod.decode_step(np.arange(Kr, dtype=np.int32)[None], gate[b:b + 1], q[t][b:b + 1],
                                           k[t][b:b + 1], v[t][b:b + 1], Kr, d, 1, wl.base, okc, ovc, bases, olen_b,
                                           caps)
            assert_close_attention(yh[b:b + 1], y_ref, gate[b:b + 1], what=f"step {t} seq {b}")
            for slot in range(Kr):
                sidx = b * Hr + int(top[b, slot])
                row = int(bases[slot] + lens[slot])
                ak, av = appended.setdefault(sidx, ([], []))
                ak.append(okc[row].copy())
                av.append(ovc[row].copy())
                o_len[sidx] += 1
                # the GPU's appended k~ is the oracle's rounded to bf16
                got_k = bf16_to_f64(kc[int(seg_base[sidx]) + row - int(bases[slot])])
                assert np.all(np.abs(got_k - okc[row]) <= np.abs(okc[row]) * 2.0 ** -7 + 1e-6), (t, b, slot)
        np.testing.assert_array_equal(seg_len.cpu().numpy(), o_len)
    assert int(status.item()) == 0
