"""Helpers shared by the GPU parity tests (device transfer, tolerances, sampling)."""
from __future__ import annotations

import numpy as np
import torch

# Attention outputs from bf16 inputs against the fp64 oracle: max abs <= 2e-2 and
# mean abs <= 2e-3, on both y = g * h and on h itself.
MAX_ABS = 2e-2
MEAN_ABS = 2e-3
# fp32 gates against fp64 softmax (relative).
GATE_RTOL = 1e-5


def dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def host_bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close_attention(got: np.ndarray, expect: np.ndarray, gate: np.ndarray | None = None, what: str = "y"):
    """got / expect [..., d]; gate broadcastable to [...] (to also check h = y / gate)."""
    err = np.abs(got - expect)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    assert err.max() <= MAX_ABS, f"{what}: max abs error {err.max():.3e} > {MAX_ABS}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean abs error {err.mean():.3e} > {MEAN_ABS}"
    if gate is not None:
        g = np.asarray(gate, np.float64)[..., None]
        eh = np.abs(got / g - expect / g)
        assert eh.max() <= MAX_ABS, f"{what}/gate: max abs error {eh.max():.3e} > {MAX_ABS}"
        assert eh.mean() <= MEAN_ABS, f"{what}/gate: mean abs error {eh.mean():.3e} > {MEAN_ABS}"


def sample_rows(seg_offsets: np.ndarray, count: int, seed: int = 0, tile: int = 128) -> np.ndarray:
    """Packed rows to check at full size: each segment's first and last row, rows on both
    sides of every 128-row tile boundary of the longest segment, and random rows."""
    rng = np.random.default_rng(seed)
    seg = np.asarray(seg_offsets, np.int64)
    picks = set()
    for s in range(len(seg) - 1):
        if seg[s + 1] > seg[s]:
            picks.add(int(seg[s]))
            picks.add(int(seg[s + 1] - 1))
    longest = int(np.argmax(seg[1:] - seg[:-1]))
    n = int(seg[longest + 1] - seg[longest])
    for b in range(tile, n, tile * max(1, n // tile // 16)):
        picks.add(int(seg[longest] + b - 1))
        picks.add(int(seg[longest] + b))
    R = int(seg[-1])
    picks.update(int(x) for x in rng.integers(0, R, size=count))
    return np.array(sorted(picks), np.int64)
