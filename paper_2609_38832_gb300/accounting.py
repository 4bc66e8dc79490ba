"""Host-side work and traffic accounting for the routed-attention path.

These are the counts the benchmark divides by time; none of them runs on the
GPU path and none depends on the oracle.

* App. B.5, Eq. (app-routed-interactions): the causal interaction count of one
  sequence is C_attn = sum_i n_i (n_i + 1) / 2.
* App. B.7, Eq. (app-group-prefill): under KV-group routing each local rank
  produces g queries, so C_attn = g * sum_j n_j (n_j + 1) / 2.
* App. B.5, Eq. (app-routed-kv): M_KV = sum_i n_i = T K (storage) and
  A_KV(T) = sum_{i in S_K(T)} n_i (activation of the next token).
* App. B.5, Eq. (app-load-cv): CV(n)^2 with the population variance.
* App. B.5, Eq. (app-interaction-bounds):
  T^2 K^2 / (2H) + T K / 2 <= C_attn <= K T (T + 1) / 2.

Each interaction costs one d-length dot product for Q K^T and one d-length
axpy for P V, i.e. 4 d flops (2 d multiply-adds counted as 2 flops each).
"""
from __future__ import annotations

import numpy as np


def interaction_count(n, g: int = 1) -> int:
    """C_attn = g * sum n (n + 1) / 2 over every (sequence, head) segment length in `n`."""
    n = np.asarray(n, dtype=np.int64).reshape(-1)
    return int(g) * int(np.sum(n * (n + 1) // 2))


def attention_flops(n, d: int, g: int = 1) -> int:
    """Algorithmic flops of routed causal attention: 4 d C_attn (exact causal pairs, no tile padding)."""
    return 4 * int(d) * interaction_count(n, g)


def kv_storage(n) -> int:
    """M_KV: stored key-value pairs after the prefix."""
    return int(np.sum(np.asarray(n, dtype=np.int64)))


def kv_activation(n_seq, heads) -> int:
    """A_KV(T): historical pairs the next token reads through its selected heads."""
    n_seq = np.asarray(n_seq, dtype=np.int64)
    return int(sum(int(n_seq[h]) for h in heads))


def cv2(n) -> float:
    """Squared coefficient of variation of the loads (population variance)."""
    n = np.asarray(n, dtype=np.float64)
    mean = n.mean()
    return float(((n - mean) ** 2).mean() / (mean * mean)) if mean > 0 else 0.0


def interaction_bounds(T: int, K: int, H: int) -> tuple[float, float]:
    """Lower / upper bound on C_attn for one sequence."""
    lower = T * T * K * K / (2.0 * H) + T * K / 2.0
    upper = K * T * (T + 1) / 2.0
    return lower, upper


def segment_lengths(seg_offsets) -> np.ndarray:
    """n per segment from the packed offsets."""
    s = np.asarray(seg_offsets, dtype=np.int64)
    return s[1:] - s[:-1]


def route_bytes(B: int, T: int, H: int, K: int, compaction: bool = True) -> int:
    """Algorithmic HBM bytes of routing: read the fp32 logits, write topk_head and gate,
    and with compaction also rank, row, row_src and the (B*H + 1) offsets."""
    tokens = B * T
    b = tokens * H * 4 + tokens * K * 8
    if compaction:
        b += tokens * K * 12 + (B * H + 1) * 4
    return b


def rope_pack_bytes(R: int, d: int, g: int = 1, copy_v: bool = True) -> int:
    """Algorithmic HBM bytes of RoPE/pack: read Q (R g rows) and K, write Q~ and K~ (bf16),
    plus reading and writing V when it is copied into a separate cache."""
    rows = R * g + R + (R if copy_v else 0)
    return 2 * rows * d * 2


def decode_bytes(lengths_after_append, d: int, g: int = 1) -> int:
    """Algorithmic HBM bytes of one decode step: every selected (sequence, head) history of
    n + 1 rows read once for K~ and once for V (bf16), plus q / k / v in and y out."""
    L = np.asarray(lengths_after_append, dtype=np.int64)
    pairs = L.size
    hist = int(np.sum(L)) * 2 * d * 2
    small = pairs * (g * d * 2 + 2 * d * 2 + g * d * 2 + 2 * d * 2)
    return hist + small
