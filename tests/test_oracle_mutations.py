"""The oracle's pins must fail when a plausible mistake is planted in the oracle.

Each case copies the oracle's C source to a temporary directory, applies one textual
mutation (a dropped term, a wrong sign, an off-by-one index, a wrong tie rule ...),
and runs the pin tests against that copy in a subprocess.  The mutated copy never
touches the real oracle build.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "namoh_oracle.c")

MUTATIONS = {
    "rope_sign": ("out[i1] = x1 * c + x0 * s;", "out[i1] = x1 * c - x0 * s;"),
    "interleave_pairs_swapped": ("int i0 = interleaved ? 2 * j : j, i1 = interleaved ? 2 * j + 1 : j + half;",
                                 "int i0 = interleaved ? 2 * j + 1 : j, i1 = interleaved ? 2 * j : j + half;"),
    "global_key_uses_rank": ("c->pos ? (double)c->pos[row] : (double)(row - off)",
                             "c->pos ? (double)(row - off) : (double)(row - off)"),
    "varlen_segments_of_sequence_0": ("int r = seg_offsets[(long)b * H + topk_head[idx]] + rank[idx];",
                                      "int r = seg_offsets[topk_head[idx]] + rank[idx];"),
    "proj_query_heads_swapped": ("c->q[(r * c->g + n / c->d) * c->d + n % c->d] = acc;",
                                 "c->q[(r * c->g + (c->g - 1 - n / c->d)) * c->d + n % c->d] = acc;"),
    "proj_wrong_group": ("const int hr = lo % c->Hr;", "const int hr = (lo + 1) % c->Hr;"),
    "proj_out_drops_first_slot": ("for (int k = 0; k < c->Kr; ++k) {", "for (int k = 1; k < c->Kr; ++k) {"),
    "shared_window_one_too_wide": ("(c->window > 0 && t + 1 > c->window) ? t + 1 - c->window : 0;",
                                   "(c->window > 0 && t + 1 > c->window) ? t - c->window : 0;"),
    "decode_window_one_too_wide": ("(window > 0 && rho + 1 > window) ? rho + 1 - window : 0;",
                                   "(window > 0 && rho + 1 > window) ? rho - window : 0;"),
    "decode_ignores_token_pos": ("const double p = token_pos ? (double)token_pos[b] : (double)rho;",
                                 "const double p = token_pos ? (double)rho : (double)rho;"),
    "no_scale": ("double scale = 1.0 / sqrt((double)d);", "double scale = 1.0;"),
    "causal_drops_self": ("attend(qr, c->krot + off * d, vals, r + 1, d, w, h);",
                          "attend(qr, c->krot + off * d, vals, r > 0 ? r : 1, d, w, h);"),
    "ties_to_upper_index": ("return a < b;", "return a > b;"),
    "theta_exponent": ("double theta = pow(base, -2.0 * (double)j / (double)d);",
                       "double theta = pow(base, -1.0 * (double)j / (double)d);"),
    "gates_renormalised": ("for (int i = 0; i < H; ++i) z += exp((double)s[i] - mx);",
                           "for (int i = 0; i < K; ++i) z += exp((double)s[order[i]] - mx);"),
    "query_rank_shift": ("rope_rotate(qin, d, c->pos ? (double)c->pos[row] : (double)r, c->base",
                         "rope_rotate(qin, d, c->pos ? (double)c->pos[row] : (double)(r + 1), c->base"),
    "decode_rank_shift": ("const double p = token_pos ? (double)token_pos[b] : (double)rho;",
                          "const double p = token_pos ? (double)token_pos[b] : (double)(rho + 1);"),
    "biased_gate_includes_bias": ("gate[t * K + k] = a[order[k]];", "gate[t * K + k] = kt[order[k]];"),
    "biased_key_drops_bias": ("kt[i] = a[i] + (double)bias[i];", "kt[i] = a[i];"),
    "biased_ties_to_upper_index": ("while (j > 0 && kt[i] > kt[order[j - 1]]) {",
                                   "while (j > 0 && kt[i] >= kt[order[j - 1]]) {"),
    "sa_budget_floor": ("return (nb * a_num + a_den - 1) / a_den;", "return (nb * a_num) / a_den;"),
    "sa_keeps_lowest_scores": ("if (!take[b] && (best < 0 || score[b] > score[best])) best = b;",
                               "if (!take[b] && (best < 0 || score[b] < score[best])) best = b;"),
    "sa_current_block_shift": ("long cur = r / Bk;                        /* current block: N_B(r) - 1 */",
                               "long cur = (r + 1) / Bk;                  /* current block: N_B(r) - 1 */"),
    "sa_drops_current_block": ("long e1 = b < cur ? (b + 1) * Bk : r + 1;", "long e1 = b < cur ? (b + 1) * Bk : r;"),
    "sa_pools_shifted_rows": ("for (long t = b * Bk; t < (b + 1) * Bk; ++t) acc += c->krot[(off + t) * d + cc];",
                              "for (long t = b * Bk; t < (b + 1) * Bk; ++t) acc += c->krot[(off + t + 1) * d + cc];"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(tmp_path, name):
    before, after = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(before) == 1, f"mutation anchor for {name} not found exactly once"
    shutil.copytree(os.path.join(ROOT, "oracle"), tmp_path / "oracle",
                    ignore=shutil.ignore_patterns("*.so", "*.tmp*", "__pycache__"))
    (tmp_path / "oracle" / "namoh_oracle.c").write_text(src.replace(before, after))
    shutil.copy(os.path.join(ROOT, "namoh_inputs.py"), tmp_path)
    shutil.copytree(os.path.join(ROOT, "paper_2609_38832_gb300"), tmp_path / "paper_2609_38832_gb300",
                    ignore=shutil.ignore_patterns("*.so", "__pycache__", "csrc", "_build"))
    os.makedirs(tmp_path / "tests")
    for f in ("conftest.py", "test_oracle_route.py", "test_oracle_attention.py", "test_oracle_layer.py",
              "test_oracle_shared.py", "test_oracle_sa.py", "test_accounting.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), tmp_path / "tests")
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), tmp_path / "tests" / "golden")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", "-m", "not gpu",
                        "tests"], cwd=tmp_path, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"mutation {name} survived the pins:\n{r.stdout[-2000:]}"
