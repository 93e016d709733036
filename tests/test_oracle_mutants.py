"""Planted mistakes in a copy of the oracle must each trip at least one pin.

Each mutant is a one-place textual change to oracle.c (a dropped term, a wrong
sign, a wrong or transposed index, a wrong operand), compiled on the CPU into
a temporary library; the real oracle is never touched.
"""
import os

import pytest

import oracle
from tests.oracle_pins import ALL_PINS

MUTANTS = {
    "drop_skip_term": ("y[t] = acc + p->Dskip[c] * u[t];", "y[t] = acc;"),
    "wrong_sign_in_abar": ("double abar = exp(delta * A[n]);", "double abar = exp(-delta * A[n]);"),
    "C_replaced_by_B": ("acc += Ck[n * L + t] * h[n];", "acc += Bk[n * L + t] * h[n];"),
    "input_without_u": ("h[n] = abar * h[n] + bbar * u[t];", "h[n] = abar * h[n] + bbar;"),
    "bias_dropped": ("double v = dl[t] + p->bias[c];", "double v = dl[t];"),
    "bias_wrong_channel": ("double v = dl[t] + p->bias[c];", "double v = dl[t] + p->bias[d];"),
    "softplus_wrong_branch": ("log1p(exp(-fabs(x)))", "log1p(exp(-x))"),
    "nonzero_initial_state": ("for (long n = 0; n < N; ++n) h[n] = 0.0;\n    for (long t = 0; t < L; ++t) {\n        double v",
                              "for (long n = 0; n < N; ++n) h[n] = 1.0;\n    for (long t = 0; t < L; ++t) {\n        double v"),
    "zoh_missing_delta": ("return expm1(delta * a) / a * b;", "return expm1(delta * a) / (delta * a) * b;"),
    "column_major_as_row_major": ("case 1: return w * H + h;", "case 1: return h * W + w;"),
    "reverse_off_by_one": ("case 2: return L - 1 - (h * W + w);", "case 2: return (L - (h * W + w)) % L;"),
    "merge_wrong_direction": ("(s0[seq_pos(0, h, w, H, W)] + s2[seq_pos(2, h, w, H, W)])",
                              "(s0[seq_pos(0, h, w, H, W)] + s2[seq_pos(3, h, w, H, W)])"),
    "mean_sum_not_mean": ("abar[n] /= (double)D; bubar[n] /= (double)D;", "bubar[n] /= (double)D;"),
    "mean_wrong_channel_A": ("abar[n] += exp(delta * p->A[c * N + n]);",
                             "abar[n] += exp(delta * p->A[(k * D) * N + n]);"),
    "mean_skip_wrong_channel": (": p->Dskip[c] * u[d * L + t];", ": p->Dskip[k * D] * u[d * L + t];"),
    "mean_output_before_update": ("h[n] = abar[n] * h[n] + bubar[n];\n            ybar += Ck[n * L + t] * h[n];",
                                  "ybar += Ck[n * L + t] * h[n];\n            h[n] = abar[n] * h[n] + bubar[n];"),
    "mean_bu_without_u": ("p->b_mode) * u[d * L + t];", "p->b_mode);"),
    "disc_abar_sign": ("dA[(row * N + n) * L + l] = exp(dlt * a);", "dA[(row * N + n) * L + l] = exp(-dlt * a);"),
    "disc_bu_wrong_b_row": ("dBu[(row * N + n) * L + l] =\n                            discretise_b(dlt, a, Bs[((b * K + k) * N + n) * L + l]",
                            "dBu[(row * N + n) * L + l] =\n                            discretise_b(dlt, a, Bs[((b * K + k) * N + 0) * L + l]"),
    "disc_mean_sum_not_mean": ("dAm[((b * K + k) * N + n) * L + l] = sa / (double)D;",
                               "dAm[((b * K + k) * N + n) * L + l] = sa;"),
    "disc_mean_bias_wrong_channel": ("double v = delta[row * L + l] + bias[c];\n                        double dlt = softplus_on ? softplus(v) : v;\n                        double a = A[c * N + n];\n                        sa",
                                     "double v = delta[row * L + l] + bias[k];\n                        double dlt = softplus_on ? softplus(v) : v;\n                        double a = A[c * N + n];\n                        sa"),
    "grouped_divides_by_D": ("h[n] = abar[n] / (double)Dg * h[n] + bubar[n] / (double)Dg;",
                             "h[n] = abar[n] / (double)D * h[n] + bubar[n] / (double)Dg;"),
    "grouped_first_group_only": ("long d0 = g * Dg;", "long d0 = 0;"),
    "selection_transposed_B": ("sb += WB[(k * N + n) * D + d] * uk[d * L + l];",
                               "sb += WB[(k * D + d) * N + n] * uk[d * L + l];"),
    "selection_C_from_B": ("sc += WC[(k * N + n) * D + d] * uk[d * L + l];",
                           "sc += WB[(k * N + n) * D + d] * uk[d * L + l];"),
    "selection_up_transposed": ("sd += Wup[(k * D + d) * R + r] * z[r];", "sd += Wup[(k * R + r) * D + d] * z[r];"),
    "selection_first_direction_weights": ("sz += Wz[(k * R + r) * D + d] * uk[d * L + l];",
                                          "sz += Wz[r * D + d] * uk[d * L + l];"),
    "bwd_carry_uses_previous_abar": ("lam[n] *= abar[t * N + n];", "lam[n] *= abar[(t > 0 ? t - 1 : 0) * N + n];"),
    "bwd_gu_without_mean_factor": ("gu[i] = Dskip[c] * gy[i] + gs[t] * delta / (double)M;",
                                   "gu[i] = Dskip[c] * gy[i] + gs[t] * delta;"),
    "bwd_without_softplus_derivative": ("double gv = softplus_on ? gd / (1.0 + exp(-v)) : gd;", "double gv = gd;"),
    "bwd_gabar_with_current_state": ("gab[t * N + n] = lam[n] * h[t * N + n];",
                                     "gab[t * N + n] = lam[n] * h[(t + 1) * N + n];"),
    "scan_only_drops_decay": ("h[n] = dA[(row * N + n) * L + l] * h[n] + dBu[(row * N + n) * L + l];",
                              "h[n] = h[n] + dBu[(row * N + n) * L + l];"),
    "scan_only_output_before_update": ("h[n] = dA[(row * N + n) * L + l] * h[n] + dBu[(row * N + n) * L + l];\n                        acc += Cs[((b * K + k) * N + n) * L + l] * h[n];",
                                       "acc += Cs[((b * K + k) * N + n) * L + l] * h[n];\n                        h[n] = dA[(row * N + n) * L + l] * h[n] + dBu[(row * N + n) * L + l];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(oracle.SOURCE).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    mpath = os.path.join(tmp_path, f"oracle_{name}.c")
    with open(mpath, "w") as f:
        f.write(src.replace(old, new))
    lib = oracle.compile_c(mpath, os.path.join(tmp_path, f"liboracle_{name}.so"))
    mutant = oracle.Oracle(lib)
    caught = []
    for pin in ALL_PINS:
        try:
            pin(mutant)
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches mutant {name}"
