"""Each planted mistake in a copy of the oracle must be caught by the pins.

The mutants are textual edits of oracle/moce_oracle.c compiled to a temporary
library; the real oracle is never modified.
"""
import os
import subprocess

import pytest

import oracle
import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "moce_oracle.c")

MUTANTS = {
    "softmax_sign": ("ae[i] = exp(((double)L[i] - m) / t);", "ae[i] = exp((m - (double)L[i]) / t);"),
    "gate_input_reversed": ("u[i] = z[(size_t)n * C + packed_idx[(size_t)e * k + i]];",
                            "u[i] = z[(size_t)n * C + packed_idx[(size_t)e * k + (k - 1 - i)]];"),
    "gate_W1_transposed": ("s += (double)W1[(size_t)j * k + i] * u[i];",
                           "s += (double)W1[(size_t)i * k + j] * u[i];"),
    "gate_b1_dropped": ("double s = (double)b1[j];\n                for (int i = 0;",
                        "double s = 0.0;\n                for (int i = 0;"),
    "gate_relu_dropped": ("h[j] = s > 0.0 ? s : 0.0;", "h[j] = s;"),
    "gate_b2_dropped": ("double g = (double)b2;\n            for (int j = 0; j < k; ++j)\n                g += (double)w2[j] * h[j];",
                        "double g = 0.0;\n            for (int j = 0; j < k; ++j)\n                g += (double)w2[j] * h[j];"),
    "sigmoid_sign": ("double sig = 1.0 / (1.0 + exp(-g));\n            if (g_out)",
                     "double sig = 1.0 / (1.0 + exp(g));\n            if (g_out)"),
    "tau_reversed": ("tau[(size_t)n * R + e] = tau_min + (tau_max - tau_min) * sig;",
                     "tau[(size_t)n * R + e] = tau_max - (tau_max - tau_min) * sig;"),
    "pool_not_divided": ("z[(size_t)n * C + c] = s / (double)HW;", "z[(size_t)n * C + c] = s;"),
    "mix_index_shift": ("s += ae[i] * (double)x[x_at(layout, n, p, packed_idx[(size_t)e * k + i], HW, C)];",
                        "s += ae[i] * (double)x[x_at(layout, n, p, packed_idx[(size_t)e * k + (i + 1) % k], HW, C)];"),
    "mix_last_term_dropped": ("for (int i = 0; i < k; ++i)\n                    s += ae[i]",
                              "for (int i = 0; i < k - 1; ++i)\n                    s += ae[i]"),
    "residual_not_divided": ("r /= (double)n_resid;", "r *= 1.0;"),
    "residual_complement_flipped": ("if (!covered[c])\n                resid[m++] = c;",
                                    "if (covered[c])\n                resid[m++] = c;"),
    "pack_ascending": ("if (a->logit > b->logit)\n        return -1;", "if (a->logit < b->logit)\n        return -1;"),
    "pack_ties_descending_index": ("return (a->idx > b->idx) - (a->idx < b->idx);",
                                   "return (a->idx < b->idx) - (a->idx > b->idx);"),
    "pack_no_duplicate_check": ("seen_in_row[c] == e", "0"),
    "coverage_softmax_over_experts": ("        for (int c = 0; c < C; ++c)\n            sum += exp((double)Le[c] - m);",
                                      "        for (int c = 0; c < C; ++c)\n            sum += exp((double)Le[c] - m) * (double)R / (double)C;"),
    "coverage_u_not_averaged": ("u[c] = s / (double)R;", "u[c] = s;"),
    "coverage_no_eps": ("const double D = ubar * ubar + eps;", "const double D = ubar * ubar;"),
    # (a term that is the same for every channel cancels in dL/dL through the
    # softmax Jacobian, so dropping one is not a mistake; flipping the
    # per-channel deviation is)
    "coverage_grad_deviation_sign": ("g[c] = 2.0 * (u[c] - ubar) / D", "g[c] = 2.0 * (ubar - u[c]) / D"),
    "backward_softmax_mean_dropped": ("const double ds = a[i] * (da[i] - ada);",
                                      "const double ds = a[i] * da[i];"),
    "backward_dtau_sign": ("dtau -= ds * (double)L[i] / (tau * tau);",
                           "dtau += ds * (double)L[i] / (tau * tau);"),
    "backward_pool_not_divided": ("dx[x_at(layout, n, p, c, HW, C)] = dz[c] / (double)HW;",
                                  "dx[x_at(layout, n, p, c, HW, C)] = dz[c];"),
    "backward_relu_mask_dropped": ("dh[j] = hpre[j] > 0.0 ? dg * (double)w2[j] : 0.0;",
                                   "dh[j] = dg * (double)w2[j];"),
    "backward_du_uses_W1_rows": ("du += (double)W1[(size_t)j * k + i] * dh[j];",
                                 "du += (double)W1[(size_t)i * k + j] * dh[j];"),
    "backward_residual_not_divided": ("const double d = (double)dy[x_at(layout, n, p, R, HW, E)] / (double)n_resid;",
                                      "const double d = (double)dy[x_at(layout, n, p, R, HW, E)];"),
    "dynamic_relu_dropped": ("h[j] = (s > 0.0) ? s : 0.0; /* ReLU", "h[j] = s; /* ReLU"),
    "dynamic_bias_dropped": ("double s = (double)bh[j];", "double s = 0.0;"),
    "dynamic_V_transposed": ("(double)V[(size_t)c * d + j];", "(double)V[(size_t)j * C + c];"),
    "dynamic_Wh_transposed": ("s += (double)Wh[(size_t)j * C + c] * zn[c];",
                              "s += (double)Wh[(size_t)c * d + j] * zn[c];"),
    "dynamic_Q_uses_channel": ("off += (double)Q[(size_t)e * d + j] * h[j]",
                               "off += (double)Q[(size_t)(c % R) * d + j] * h[j]"),
    "dynamic_offset_sign": ("Ldyn[((size_t)n * R + e) * C + c] = (double)L[(size_t)e * C + c] + off;",
                            "Ldyn[((size_t)n * R + e) * C + c] = (double)L[(size_t)e * C + c] - off;"),
    "topk_reads_first_row": ("float v = L[(size_t)e * C + c];", "float v = L[c];"),
    "topk_off_by_one": ("idx_out[(size_t)e * k + i] = row[i].idx;",
                        "idx_out[(size_t)e * k + i] = row[i + 1].idx;"),
    "coverage_grad_softmax_jacobian_dot_dropped": ("p[(size_t)e * C + c] * (g[c] - dot) / (double)R;",
                                                   "p[(size_t)e * C + c] * g[c] / (double)R;"),
}

PIN_CHECKS = [
    pins.test_worked_tiny_layer,
    lambda: pins.test_pack_equals_bruteforce_sort(0),
    pins.test_pack_permutation_invariant,
    pins.test_pack_ties_and_signed_zero,
    pins.test_topk_equals_stable_argsort,
    lambda: pins.test_pack_rejects("dup"),
    lambda: pins.test_cyclic_supports_residual_closed_form(64, 15, 4),
    lambda: pins.test_pool_closed_forms("nhwc"),
    pins.test_gate_zero_hidden_gives_sigmoid_of_bias,
    pins.test_gate_reads_inputs_in_descending_logit_order_and_w1_rows_are_hidden_units,
    pins.test_gate_relu_clamps,
    pins.test_weights_convex_and_order_invariant,
    pins.test_weights_unit_temperature_is_plain_softmax,
    pins.test_weights_temperature_limits,
    pins.test_mix_bounds_and_residual_mean,
    pins.test_empty_residual_is_exactly_zero,
    lambda: pins.test_forward_equals_bruteforce("nhwc", 0),
    pins.test_fixed_temperature_is_a_linear_map,
    pins.test_coverage_uniform_rows_are_zero,
    lambda: pins.test_coverage_one_expert_two_channels_closed_form(2.5, -1.0),
    pins.test_coverage_row_shift_and_channel_permutation,
    pins.test_coverage_equals_numpy_definition_and_finite_differences,
    lambda: pins.test_backward_equals_central_differences("nhwc"),
    pins.test_backward_constant_temperature_is_the_transposed_linear_map,
    lambda: pins.test_dynamic_offset_vanishes("h"),
    pins.test_dynamic_single_coupling_lands_on_one_expert_and_channel,
    lambda: pins.test_dynamic_router_reads_the_pooled_descriptor("nhwc"),
    pins.test_dynamic_offset_has_rank_at_most_d_and_is_bilinear,
    pins.test_dynamic_supports_follow_each_example,
]


def _build_mutant(tmp_path, name, old, new):
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation site for {name} not unique"
    src = tmp_path / f"{name}.c"
    src.write_text(text.replace(old, new))
    so = tmp_path / f"lib{name}.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so), str(src), "-lm"],
                   check=True)
    return str(so)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(tmp_path, name):
    old, new = MUTANTS[name]
    so = _build_mutant(tmp_path, name, old, new)
    failures = 0
    with oracle._use_library(so):
        for check in PIN_CHECKS:
            try:
                check()
            except (Exception, pytest.fail.Exception):  # a failed assertion or an oracle error
                failures += 1
    assert failures > 0, f"no pin catches mutant {name}"
