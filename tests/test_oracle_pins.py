"""The CPU oracle against its pins (no GPU), and planted mistakes in copies of
the oracle source, each of which some pin must catch."""
import os

import pytest

import oracle_pins as P


@pytest.mark.parametrize("check", P.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(oracle_mod, check):
    check()


def test_learnable_records_accuracy(oracle_mod):
    acc_train, acc_test = P.check_learnable()
    assert acc_train >= P.LEARN_MIN_TRAIN_ACC
    assert acc_test >= 0.7, acc_test


# Plausible mistakes: (name, exact text in bmlp_oracle.c, replacement).
MUTANTS = [
    ("sign_zero_negative", "static int32_t sign_of(int32_t v) { return v >= 0 ? +1 : -1; }",
     "static int32_t sign_of(int32_t v) { return v > 0 ? +1 : -1; }"),
    ("argmax_ties_high", "      if (v[j] > v[jmax]) jmax = j;\n    int32_t second",
     "      if (v[j] >= v[jmax]) jmax = j;\n    int32_t second"),
    ("tau_distinct_values", "if (j != jmax && v[j] > second)", "if (v[j] != v[jmax] && v[j] > second)"),
    ("margin_not_strict", "(int64_t)t * r_den < (int64_t)r_num * K", "(int64_t)t * r_den <= (int64_t)r_num * K"),
    ("select_most_negative", "delta[k] > delta[best]", "delta[k] < delta[best]"),
    ("select_allows_zero", "if (delta[k] < 0 &&", "if (delta[k] <= 0 &&"),
    ("cp_sign_flipped", "*h = clip(*h + 2 * a_prev[(int64_t)mu * K_prev + i] * rho, h_max);",
     "*h = clip(*h - 2 * a_prev[(int64_t)mu * K_prev + i] * rho, h_max);"),
    ("cp_no_clip", "*h = clip(*h + 2 * a_prev[(int64_t)mu * K_prev + i] * rho, h_max);",
     "*h = *h + 2 * a_prev[(int64_t)mu * K_prev + i] * rho;"),
    ("cp_descending_mu", "  for (int32_t mu = 0; mu < b; mu++)\n    for (int32_t g = 0; g < G; g++) {\n      int32_t k = sel",
     "  for (int32_t mu = b - 1; mu >= 0; mu--)\n    for (int32_t g = 0; g < G; g++) {\n      int32_t k = sel"),
    ("reinforce_toward_zero", "*h = clip(*h + 2 * (*h > 0 ? 1 : -1), h_max);",
     "*h = clip(*h - 2 * (*h > 0 ? 1 : -1), h_max);"),
    ("threshold_floor", "return (uint64_t)ceil(x * 4294967296.0);", "return (uint64_t)floor(x * 4294967296.0);"),
    ("r_first_exponent", "first[j] = thr((1.0 - pw[j + 1]) / p_any);", "first[j] = thr((1.0 - pw[j]) / p_any);"),
    ("r_gap_exponent", "gap[g] = thr(1.0 - pw[g + 1]);", "gap[g] = thr(1.0 - pw[g]);"),
    ("r_block_gate_ignored", "if (!((uint64_t)w[b % 4] < any[x])) continue;", "(void)any;"),
    ("r_one_event_per_block", "      if (g > n - 2 - p) break;", "      break;"),
    ("r_tail_uses_full_tables", "const int32_t x = (n == 64) ? 0 : 1;", "const int32_t x = 0;"),
    ("r_event_stream_tag", "((4u + (uint32_t)(e->used / 4)) << 16)", "((5u + (uint32_t)(e->used / 4)) << 16)"),
    ("r_first_scan_short", "while (p < n - 1 && !((uint64_t)V < first[x][p])) p++;",
     "while (p < n - 2 && !((uint64_t)V < first[x][p])) p++;"),
    ("r_gap_end_exclusive", "while (g <= n - 2 - p && !((uint64_t)V < gap[x][g])) g++;",
     "while (g < n - 2 - p && !((uint64_t)V < gap[x][g])) g++;"),
    ("philox_7_rounds", "for (int round = 0; round < 10; round++)", "for (int round = 0; round < 7; round++)"),
    ("update_without_marks", "if (!any) continue; /* O6 */", "(void)any;"),
    ("gamma_ties_small", "(dist == best_dist && g > best)", "(dist == best_dist && g < best)"),
    ("pr_without_sqrt", "m->p_r = m->p_r * sqrt(E);", "m->p_r = m->p_r * E;"),
    ("binarize_upper_median", "const float med = s[(K + 1) / 2 - 1];", "const float med = s[K / 2];"),
    ("binarize_not_strict", "a[mu * K + i] = (int8_t)(row[i] > med ? 1 : -1);",
     "a[mu * K + i] = (int8_t)(row[i] >= med ? 1 : -1);"),
    ("early_exit_layers_reversed", "pred[(int64_t)(l - 1) * n + start + mu] = jmax;",
     "pred[(int64_t)(L - l) * n + start + mu] = jmax;"),
    ("layer_errors_count_marks", "m->layer_err[l] += ell[mu]; /* O17 */", "m->layer_err[l] += mark[l][mu];"),
    ("group_ties_by_position", "(delta[k] == delta[best] && k < best)", "(0)"),
    ("group_key_word", "v[k].u = w[k % 4];", "v[k].u = w[0];"),
    ("group_mode2_fixed", "const uint32_t tt = (mode == 2) ? t : 0u;", "const uint32_t tt = 0u;"),
    ("forward_drops_sign", "zr[k] += ai * (hrow[k] > 0 ? 1 : -1);", "zr[k] += ai * hrow[k];"),
    ("expand_sign_zero_negative", "a[mu * K + k] = (int8_t)(z >= 0 ? 1 : -1);",
     "a[mu * K + k] = (int8_t)(z > 0 ? 1 : -1);"),
    ("expand_weights_transposed", "(int64_t)e[(int64_t)k * D + i];", "(int64_t)e[(int64_t)i * K + k];"),
    ("expand_input_signed", "z += (int64_t)x[mu * D + i]", "z += (int64_t)(int8_t)x[mu * D + i]"),
    ("expand_stream_tag", "(uint32_t)k, 33u << 16, 0u, w);", "(uint32_t)k, 32u << 16, 0u, w);"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(oracle_mod, tmp_path, name, old, new):
    src = oracle_mod.source()
    assert src.count(old) == 1, "mutation anchor not found exactly once: " + name
    path = oracle_mod.compile_variant(src.replace(old, new), os.path.join(tmp_path, name + ".so"))
    caught = []
    with oracle_mod.use_library(path):
        for check in P.ALL_CHECKS:
            try:
                check()
            except AssertionError:
                caught.append(check.__name__)
                break
    assert caught, "no pin caught the planted mistake " + name
