"""Planted mistakes in the oracle must be caught by its pins.

Each case copies ``oracle/hedgefb_oracle.c``, replaces one exact snippet by a
plausible mistake (a dropped term, a flipped sign, a shifted or transposed
index, a wrong tie rule), builds the copy and runs the pins against it.  The
case passes when at least one pin fails.  CPU only.
"""
import os

import pytest

import oracle
from oracle_pins import ALL_CHECKS

MUTANTS = {
    "overlap_max_not_min": ("a += (P[v] < Q[v]) ? P[v] : Q[v];", "a += (P[v] < Q[v]) ? Q[v] : P[v];"),
    "tv_no_half": ("return 0.5 * t;", "return t;"),
    "softmax_max_without_T": ("double s = orc_decode(row, dtype, v) / T;\n    if (s > m)",
                              "double s = orc_decode(row, dtype, v);\n    if (s > m)"),
    "softmax_sum_without_T": ("sum += exp(orc_decode(row, dtype, v) / T - m);",
                              "sum += exp(orc_decode(row, dtype, v) - m);"),
    "softmax_prob_without_T": ("P[v] = exp(orc_decode(row, dtype, v) / T - lse);",
                               "P[v] = exp(orc_decode(row, dtype, v) - lse);"),
    "lse_drops_max": ("double lse = m + log(sum);", "double lse = log(sum);"),
    "elen_prefix_starts_at_zero": ("double e = 1.0, prod = 1.0;", "double e = 0.0, prod = 1.0;"),
    "elen_thm3_weight_k_minus_1": ("e += (double)k * (1.0 - gk) * prod;",
                                   "e += (double)(k - 1) * (1.0 - gk) * prod;"),
    "elen_thm3_no_gamma_K_plus_1_zero": ("double gk = (k <= K) ? gamma[k - 1] : 0.0;",
                                         "double gk = (k <= K) ? gamma[k - 1] : 1.0;"),
    "loss_length_over_K": ("return 1.0 - e_len / (double)(K + 1);", "return 1.0 - e_len / (double)K;"),
    "loss_accept_sums_gamma": ("s += 1.0 - gamma[k];", "s += gamma[k];"),
    "hedge_sign": ("w[i] = exp(-eta * (L[i] - L[best]));", "w[i] = exp(eta * (L[i] - L[best]));"),
    "hedge_argmax_of_loss": ("if (L[i] < L[best]) best = i;", "if (L[i] > L[best]) best = i;"),
    "nh_regret_sign": ("inc += p[j] * (loss[j] - loss[i]);", "inc += p[j] * (loss[i] - loss[j]);"),
    "nh_learner_loss_unweighted": ("inc += p[j] * (loss[j] - loss[i]);",
                                   "inc += (loss[j] - loss[i]) / (double)N;"),
    "nh_weight_drops_r_over_c": ("p[i] = (r / c) * exp(r * r / (2.0 * c));", "p[i] = exp(r * r / (2.0 * c));"),
    "nh_equation_c_not_2c": ("s += exp(r * r / (2.0 * c));", "s += exp(r * r / c);"),
    "nh_uniform_branch_picks_argmax": ("p[i] = 1.0 / (double)N;\n    *sel = 0;",
                                       "p[i] = 1.0 / (double)N;\n    *sel = best;"),
    "argmax_last_on_ties": ("if (z > bz) { bz = z; best = v; }", "if (z >= bz) { bz = z; best = v; }"),
    "bf16_shift_15": ("((uint32_t)h) << 16;", "((uint32_t)h) << 15;"),
    "fp16_bias": ("expo - 25);", "expo - 24);"),
    "nonfinite_misses_inf": ("if (isnan(z) || z == INFINITY) return 0;", "if (isnan(z)) return 0;"),
    "drafter_index_transposed": ("int64_t drow = ((int64_t)i * B + b) * P + k;",
                                 "int64_t drow = ((int64_t)b * N + i) * P + k;"),
    "target_index_transposed": ("((int64_t)b * P + k);", "((int64_t)k * B + b);"),
    "elen_uses_all_P_positions": ("* P, P - 1);", "* P, P);"),
    "greedy_inverted": ("a = (jt < 0 || jd < 0) ? NAN : (jt == jd ? 1.0 : 0.0);",
                        "a = (jt < 0 || jd < 0) ? NAN : (jt != jd ? 1.0 : 0.0);"),
    "played_loss_wrong_drafter": ("played[b] += f[selected[b]];", "played[b] += f[0];"),
    "topl_ties_toward_higher_index": ("if (best < 0 || z > bz) { best = v; bz = z; }",
                                      "if (best < 0 || z >= bz) { best = v; bz = z; }"),
    "topl_smallest_first": ("if (best < 0 || z > bz) { best = v; bz = z; }",
                            "if (best < 0 || z < bz) { best = v; bz = z; }"),
    "topl_drops_last_candidate": ("for (int r = 0; r < L; ++r) a += Pt[idx[r]];",
                                  "for (int r = 0; r + 1 < L; ++r) a += Pt[idx[r]];"),
    "topl_greedy_first_child_only": ("for (int r = 0; r < L; ++r)\n        if (idx[r] == jt) a = 1.0;",
                                     "for (int r = 0; r < 1; ++r)\n        if (idx[r] == jt) a = 1.0;"),
    "topl_repeats_tokens": ("if (idx[q] == v) { taken = 1; break; }", "if (idx[q] == v) { break; }"),
    "topl_target_index_transposed": ("int64_t row_t = (int64_t)b * P + k;",
                                     "int64_t row_t = (int64_t)k * B + b;"),
    "topl_drafter_index_transposed": ("const int64_t row_d = ((int64_t)i * B + b) * P + k;",
                                      "const int64_t row_d = ((int64_t)b * N + i) * P + k;"),
    "topl_elen_all_positions": ("e_len[i * B + b] = orc_elen_prefix(gam, P - 1);",
                                "e_len[i * B + b] = orc_elen_prefix(gam, P);"),
    "pruned_ignores_keep": ("int kept = keep < n ? keep : n;", "int kept = n;"),
    "pruned_keeps_one_more": ("int kept = keep < n ? keep : n;",
                              "int kept = keep + 1 < n ? keep + 1 : n;"),
    "pruned_keep_unchecked": ("if (L < 1 || keep < 0 || keep > L)", "if (L < 1)"),
    "pruned_greedy_whole_set": ("for (int r = 0; r < kept; ++r)\n        if (idx[r] == jt) a = 1.0;",
                                "for (int r = 0; r < n; ++r)\n        if (idx[r] == jt) a = 1.0;"),
    "pruned_drafter_index_transposed": (
        "const int64_t row_drf = ((int64_t)i * B + b) * P + k;",
        "const int64_t row_drf = ((int64_t)b * N + i) * P + k;"),
    "pruned_elen_all_positions": ("e_len[(size_t)i * B + b] = orc_elen_prefix(gam, P - 1);",
                                  "e_len[(size_t)i * B + b] = orc_elen_prefix(gam, P);"),
    "hedge_state_not_cumulative": ("for (int i = 0; i < N; ++i) col[i] += f[i];",
                                   "for (int i = 0; i < N; ++i) col[i] = f[i];"),
    "sample_at_or_above": ("if (run > thr) return i;", "if (run >= thr) return i;"),
    "sample_threshold_unscaled": ("const float thr = u * total;", "const float thr = u;"),
    "chunk_loss_reads_past_horizon": ("return orc_loss_length(orc_elen_prefix(gamma, k), k);",
                                      "return orc_loss_length(orc_elen_prefix(gamma, k + 1), k);"),
    "chunk_played_wrong_drafter": ("played[b] = played[b] + lv[selected[b]];",
                                   "played[b] = played[b] + lv[0];"),
    "token_window_shifted": ("return orc_loss_length(orc_elen_prefix(g + s, K), K);",
                             "return orc_loss_length(orc_elen_prefix(g + s + 1, K), K);"),
    "token_revealed_one_early": ("int64_t late = (loss_kind == ORC_LOSS_LENGTH) ? n - K : n;",
                                 "int64_t late = (loss_kind == ORC_LOSS_LENGTH) ? n - K + 1 : n;"),
    "token_hybrid_ignored": ("const int kind = done < accept_first ? ORC_LOSS_ACCEPT : loss_kind;",
                             "const int kind = loss_kind;"),
    "token_played_by_drafter_0": ("who[n] = choice;", "who[n] = 0;"),
    "qfid_hedge_not_cumulative": ("for (int i = 0; i < N; ++i) st[i] = st[i] + lv[i];",
                                  "for (int i = 0; i < N; ++i) st[i] = lv[i];"),
    "apply_batch_reversed": ("for (int i = 0; i < N; ++i) one[i] = lv[((size_t)c * N + i) * B + b];",
                             "for (int i = 0; i < N; ++i) one[i] = lv[((size_t)(count - 1 - c) * N + i) * B + b];"),
    "schedule_skip_strict": ("evaluate = s[1] >= skip_tokens;", "evaluate = s[1] > skip_tokens;"),
    "schedule_batch_off_by_one": ("apply = ((r - warmup + 1) % batch_rounds) == 0;",
                                  "apply = ((r - warmup) % batch_rounds) == 0;"),
    "schedule_hybrid_never": ("act[1] = (evaluate && s[2] < hybrid_vectors) ? ORC_LOSS_ACCEPT : ORC_LOSS_LENGTH;",
                              "act[1] = ORC_LOSS_LENGTH;"),
    "schedule_skip_keeps_count": ("    if (evaluate) s[1] = 0;\n", "\n"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    with open(oracle._SRC) as f:
        src = f.read()
    assert src.count(old) == 1, f"snippet for {name} must occur exactly once"
    mpath = os.path.join(tmp_path, "mutant.c")
    with open(mpath, "w") as f:
        f.write(src.replace(old, new))
    lib = oracle.build(mpath, os.path.join(tmp_path, f"libmutant_{name}.so"))
    o = oracle.Oracle(lib)
    for check in ALL_CHECKS:
        try:
            check(o)
        except AssertionError:
            return
    pytest.fail(f"no pin caught the planted mistake {name}")
