"""GPU parity of the shared heads (the paper's shared-head variant, Sec. 4.4): always-active heads
over the full causal prefix or a sliding window of the last w tokens, global RoPE, no gate.
The attention kernel runs them as segments holding every token (rank = t) with its key tiles
starting at the window; decode attends over the last min(n + 1, w) cached rows.
"""
import numpy as np
import pytest
import torch

from _gpu_helpers import assert_close_attention, bf16_to_f64, dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def namoh():
    import paper_2609_38832_gb300 as pkg
    return pkg


def _qkv(seed, shape):
    rng = np.random.default_rng(seed)
    import namoh_inputs as ni
    return tuple(ni.bf16_bits(rng.standard_normal(shape).astype(np.float32)) for _ in range(3))


@pytest.mark.parametrize("B,Hs,T,d,window", [
    (2, 2, 300, 128, 0),      # full causal prefix
    (2, 2, 300, 128, 128),    # the paper's window, several query tiles
    (1, 4, 1000, 64, 128),
    (2, 1, 333, 128, 37),     # a window inside one key tile
    (1, 2, 257, 128, 1),      # each token attends to itself only
    (1, 2, 4096, 128, 128),   # a long sequence
    # more query tiles than SMs: CTAs run several consecutive tiles, the diagonal key tile of one
    # serving as the previous tile of the next, and runs cross segment boundaries
    (4, 4, 4096, 128, 128),   # the bench's shape
    (1, 8, 5000, 64, 100),    # d = 64, a window inside one key tile, a ragged last tile
    (2, 3, 7000, 128, 2),     # the smallest window that reads the previous key tile
    (3, 2, 100, 128, 50),     # sequences shorter than one query tile
])
def test_shared_prefill_matches_oracle(namoh, oracle_mod, B, Hs, T, d, window):
    q, k, v = _qkv(60, (B, Hs, T, d))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    y, _, _ = namoh.namoh_shared_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), window=window, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref = oracle_mod.shared_prefill(q, k, v, window, 1e4)
    got = bf16_to_f64(y).reshape(-1, d)
    assert_close_attention(got, ref.reshape(-1, d), np.ones(got.shape[0]))


@pytest.mark.parametrize("window", [0, 128])
def test_shared_decode_matches_oracle_and_longer_prefill(namoh, oracle_mod, window):
    """Prefill over T tokens into caches with headroom, then decode steps (every shared head,
    the same window): each step matches the oracle continuing from its own prefix state, and the
    GPU prefill over T + steps tokens."""
    B, Hs, T, d, steps = 2, 3, 300, 128, 3
    q, k, v = _qkv(61, (B, Hs, T + steps, d))
    nseg = B * Hs
    cap = T + steps
    seg_base = torch.arange(nseg, dtype=torch.int64, device="cuda") * cap
    seg_cap = torch.full((nseg,), cap, dtype=torch.int32, device="cuda")
    seg_len = torch.zeros(nseg, dtype=torch.int32, device="cuda")
    kc = torch.zeros((nseg * cap, d), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    namoh.namoh_shared_prefill(dev_bf16(np.ascontiguousarray(q[:, :, :T])), dev_bf16(np.ascontiguousarray(k[:, :, :T])),
                               dev_bf16(np.ascontiguousarray(v[:, :, :T])), window=window, k_cache=kc, v_cache=vc,
                               seg_base=seg_base, seg_cap=seg_cap, seg_len=seg_len, status=status)
    y_full, _, _ = namoh.namoh_shared_prefill(dev_bf16(q), dev_bf16(k), dev_bf16(v), window=window, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    np.testing.assert_array_equal(seg_len.cpu().numpy(), T)
    # the oracle's own prefix state: keys rotated at t = 0 .. T-1 in fp64, exact values
    okc, ovc = np.zeros((nseg * cap, d)), np.zeros((nseg * cap, d))
    import namoh_inputs as ni
    for b in range(B):
        for j in range(Hs):
            lo = (b * Hs + j) * cap
            okc[lo:lo + T] = oracle_mod.rope(np.ascontiguousarray(k[b, j, :T]), np.arange(T), 1e4)
            ovc[lo:lo + T] = ni.bf16_to_f32(v[b, j, :T]).astype(np.float64)
    obase = (np.arange(nseg) * cap).astype(np.int64)
    olen = np.full(nseg, T, np.int32)
    ocap = np.full(nseg, cap, np.int32)
    yf = bf16_to_f64(y_full)
    for st in range(steps):
        t = T + st
        qs, ks, vs = (np.ascontiguousarray(a[:, :, t]) for a in (q, k, v))
        y = namoh.namoh_shared_decode(dev_bf16(qs), dev_bf16(ks), dev_bf16(vs), k_cache=kc, v_cache=vc,
                                      seg_base=seg_base, seg_len=seg_len, seg_cap=seg_cap, window=window,
                                      status=status)
        torch.cuda.synchronize()
        ref = oracle_mod.shared_decode_step(qs, ks, vs, d, 1e4, okc, ovc, obase, olen, ocap, window)
        got = bf16_to_f64(y).reshape(B, Hs, d)
        assert_close_attention(got.reshape(-1, d), ref.reshape(-1, d), np.ones(B * Hs), what=f"step {st}")
        assert_close_attention(got.reshape(-1, d), yf[:, t].reshape(-1, d), np.ones(B * Hs), what=f"prefill {st}")
        np.testing.assert_array_equal(seg_len.cpu().numpy(), olen)
    assert int(status.item()) == 0
