"""Host-side accounting (App. B.7) against brute-force counts and the paper's closed forms."""
import numpy as np
import pytest

import namoh_inputs as ni
from paper_2609_38832_gb300 import accounting as acc


def _brute_pairs(mask):
    """Count (t, s, i) with m_{t,i} = m_{s,i} = 1 and s <= t (App. B: R = tril(M M^T))."""
    M = mask.astype(np.int64)
    R = np.tril(M @ M.T)
    return int(R.sum())


@pytest.mark.parametrize("T,H,K", [(64, 8, 2), (100, 16, 4), (33, 5, 5)])
def test_interaction_count_matches_brute_force(oracle_mod, T, H, K):
    s = ni.router_scores(9, 1, T, H)
    out = oracle_mod.route(s, K)
    mask = np.zeros((T, H), np.int64)
    np.put_along_axis(mask, out["topk_head"][0].astype(np.int64), 1, axis=-1)
    c = acc.interaction_count(out["n"])
    assert c == _brute_pairs(mask)
    # Eq. (namoh-attention-work): T^2 K^2/(2H) [1 + CV^2] + T K / 2
    closed = T * T * K * K / (2 * H) * (1 + acc.cv2(out["n"][0])) + T * K / 2
    assert abs(c - closed) < 1e-6 * c
    lo, hi = acc.interaction_bounds(T, K, H)
    assert lo - 1e-9 <= c <= hi + 1e-9
    assert acc.kv_storage(out["n"]) == T * K


def test_upper_bound_attained_when_all_tokens_share_heads():
    T, H, K = 50, 8, 3
    n = np.zeros(H, np.int64)
    n[:K] = T
    assert acc.interaction_count(n) == acc.interaction_bounds(T, K, H)[1]


def test_group_interaction_factor():
    # Eq. (app-group-prefill): each local rank produces g queries
    n = np.array([10, 0, 7, 3])
    assert acc.interaction_count(n, g=4) == 4 * acc.interaction_count(n)
    assert acc.attention_flops(n, 128, 4) == 4 * 128 * acc.interaction_count(n, 4)


def test_kv_activation():
    n = np.array([5, 9, 2, 7])
    assert acc.kv_activation(n, [1, 3]) == 16
