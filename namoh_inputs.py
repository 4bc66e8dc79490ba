"""Seeded synthetic inputs for the NAMOH routed-attention path.

Shared by the tests, the smoke check and the benchmark, and by both the CUDA
path and the fp64 oracle.  This module holds none of the method's arithmetic:
only random draws, the bf16 encoding of those draws and the fixed workload
shapes.

Recipe (the paper's training/eval data are not available, so these stand in):
  * router logits ``x_t W_r``: i.i.d. N(0, 1) fp32 from ``numpy.random.default_rng``
    (PCG64) seeded with ``[seed, 0]``;
  * the skewed workload adds a per-head bias ``log((h+1)^-1)`` (Zipf, s = 1), computed
    in fp64, rounded to fp32 and added in fp32;
  * Q / K / V: i.i.d. N(0, 1) fp32 from ``default_rng([seed, 1])`` drawn directly in
    packed-row order, rounded to bf16 with round-to-nearest-even.
"""
from __future__ import annotations

import dataclasses

import numpy as np


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest, ties to even."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> exact fp32 values."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def router_scores(seed: int, B: int, T: int, H: int, zipf_bias: bool = False) -> np.ndarray:
    """Router logits [B, T, H] fp32."""
    rng = np.random.default_rng([seed, 0])
    s = rng.standard_normal((B, T, H), dtype=np.float32)
    if zipf_bias:
        bias = np.array([-np.log(h + 1.0) for h in range(H)], dtype=np.float64).astype(np.float32)
        s = (s + bias[None, None, :]).astype(np.float32)
    return s


def qkv_rows(seed: int, R: int, d: int, g: int = 1):
    """Packed-row Q [R*g, d], K [R, d], V [R, d] as bf16 bit patterns (uint16)."""
    rng = np.random.default_rng([seed, 1])
    q = bf16_bits(rng.standard_normal((R * g, d), dtype=np.float32))
    k = bf16_bits(rng.standard_normal((R, d), dtype=np.float32))
    v = bf16_bits(rng.standard_normal((R, d), dtype=np.float32))
    return q, k, v


def decode_step_inputs(seed: int, steps: int, B: int, Hr: int, Kr: int, d: int, g: int = 1):
    """Per-step router logits [steps, B, Hr] and q [steps, B, Kr*g, d], k/v [steps, B, Kr, d] (bf16 bits)."""
    rng = np.random.default_rng([seed, 2])
    scores = rng.standard_normal((steps, B, Hr), dtype=np.float32)
    q = bf16_bits(rng.standard_normal((steps, B, Kr * g, d), dtype=np.float32))
    k = bf16_bits(rng.standard_normal((steps, B, Kr, d), dtype=np.float32))
    v = bf16_bits(rng.standard_normal((steps, B, Kr, d), dtype=np.float32))
    return scores, q, k, v


@dataclasses.dataclass(frozen=True)
class PrefillWorkload:
    """A prefill workload: B sequences of T tokens, H routed heads (query heads), K active,
    head width d, g query heads per KV group (1 = no grouping), RoPE base."""
    name: str
    B: int
    T: int
    H: int
    K: int
    d: int
    g: int = 1
    base: float = 10000.0
    zipf_bias: bool = False
    seed: int = 0

    @property
    def Hr(self) -> int:  # routed units (heads, or KV groups when g > 1)
        return self.H // self.g

    @property
    def Kr(self) -> int:  # routed units selected per token
        return self.K // self.g

    @property
    def rows(self) -> int:  # packed KV rows R = B*T*Kr
        return self.B * self.T * self.Kr

    def scores(self) -> np.ndarray:
        return router_scores(self.seed, self.B, self.T, self.Hr, self.zipf_bias)

    def qkv(self):
        return qkv_rows(self.seed, self.rows, self.d, self.g)


@dataclasses.dataclass(frozen=True)
class DecodeWorkload:
    """B sequences with a routed prefix of `prefix` tokens, then `steps` one-token steps."""
    name: str
    B: int
    prefix: int
    H: int
    K: int
    d: int
    steps: int
    g: int = 1
    base: float = 10000.0
    seed: int = 0

    @property
    def Hr(self) -> int:
        return self.H // self.g

    @property
    def Kr(self) -> int:
        return self.K // self.g


# The five workloads, by what they are.
PR1 = PrefillWorkload("pr1_b1_t512_h8_k2_d64", B=1, T=512, H=8, K=2, d=64)
BALANCED = PrefillWorkload("balanced_b4_t4096_h16_k4_d128", B=4, T=4096, H=16, K=4, d=128)
SKEWED = PrefillWorkload("skewed_b1_t32768_h32_k4_d128_zipf", B=1, T=32768, H=32, K=4, d=128,
                         base=500000.0, zipf_bias=True)
H_SWEEP = tuple(PrefillWorkload(f"hsweep_b1_t16384_h{h}_k4_d128", B=1, T=16384, H=h, K=4, d=128)
                for h in (8, 16, 32, 64))
# KV-group routing: 64 query heads in 8 groups of g = 8; 4 of the 8 groups are selected.
GQA = PrefillWorkload("gqa_b1_t16384_h64_g8_k32_d128", B=1, T=16384, H=64, K=32, d=128, g=8)
DECODE = DecodeWorkload("decode_b64_prefix131072_h32_k4_d128", B=64, prefix=131072, H=32, K=4, d=128,
                        steps=256)
