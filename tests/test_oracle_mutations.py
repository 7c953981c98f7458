"""Each planted mistake in a copy of the C oracle must make at least one pin fail.

The mistakes are planted in a copy of the oracle's source text, compiled on the CPU into
a separate library; the oracle itself is never modified.
"""
import os

import numpy as np
import pytest

import oracle
import oracle_pins

# (name, exact text in flex_oracle.c, replacement, occurrence to replace (0 = first))
MUTATIONS = [
    ("swap_sin_cos_stationary",
     "phi[i] = c * cos(a);\n            phi[M + i] = c * sin(a);",
     "phi[i] = c * sin(a);\n            phi[M + i] = c * cos(a);", 0),
    ("omega_prime_without_half",
     "u += 0.5 * (w1[t] + w2[t]) * x[t];\n                w += 0.5 * (w1[t] - w2[t]) * x[t];\n            }\n            phi[i]",
     "u += (w1[t] + w2[t]) * x[t];\n                w += (w1[t] - w2[t]) * x[t];\n            }\n            phi[i]", 0),
    ("sum_instead_of_average_scale",
     "phi[i] = c * cos(u) * cos(w);", "phi[i] = 2.0 * c * cos(u) * cos(w);", 0),
    ("sin_block_uses_sin_w",
     "phi[M + i] = c * sin(u) * cos(w);", "phi[M + i] = c * sin(u) * sin(w);", 0),
    ("forget_normaliser_z", "dn += pq[f] * z[f];", "dn += pq[f];", 0),
    ("causal_mask_exclusive",
     "for (int i = 0; i < N; ++i) {\n        if (J->causal) {\n            feature(d, M, J->k + (size_t)i * d",
     "for (int i = 0; i < N; ++i) {\n        if (J->causal && i > 0) {\n            feature(d, M, J->k + (size_t)(i - 1) * d", 0),
    ("drop_half_in_dW1", "dW1[h * per + t] = 0.5 * (a + bb);", "dW1[h * per + t] = (a + bb);", 0),
    ("wrong_sign_du", "double du = c * cos(w) * (-sin(u) * dc + cos(u) * ds);",
     "double du = c * cos(w) * (sin(u) * dc + cos(u) * ds);", 0),
    ("wrong_sign_da_stationary", "double da = c * (-sin(a) * dc + cos(a) * ds);",
     "double da = c * (sin(a) * dc + cos(a) * ds);", 0),
    ("drop_normaliser_grad_in_dq", "double s = cc[i] * z[f];", "double s = 0.0;", 0),
    ("drop_normaliser_grad_in_dk", "dphi[f] = r[f] + dot(d, R + (size_t)f * d, vj);",
     "dphi[f] = dot(d, R + (size_t)f * d, vj);", 0),
    ("denominator_sign_in_c", "cc[i] = -s / den[i];", "cc[i] = s / den[i];", 0),
    ("reverse_scan_exclusive",
     "for (int j = N - 1; j >= 0; --j) {\n        if (J->causal)",
     "for (int j = N - 1; j >= 0; --j) {\n        if (J->causal && 0)", 0),
    ("decode_drops_new_value", "Su[(size_t)f * d + e] += pk[f] * v[u * d + e];",
     "Su[(size_t)f * d + e] += 0.0 * v[u * d + e];", 0),
    ("decode_forgets_z_update", "zu[f] += pk[f];", "zu[f] += 0.0;", 0),
    ("prefactor_sign_of_exponent", "return exp(dot(d, k, k) * itau);",
     "return exp(-dot(d, k, k) * itau);", 0),
    ("prefactor_dk_without_2", "dw * wk[j] * 2.0 * J->itau * kj[e];",
     "dw * wk[j] * J->itau * kj[e];", 0),
    ("prefactor_dtau_sign", "*J->dtau += -dw * wk[j]", "*J->dtau += dw * wk[j]", 0),
    ("prefactor_dphi_unweighted", "for (int f = 0; f < D; ++f) dphi[f] *= wk[j];",
     "for (int f = 0; f < D; ++f) dphi[f] *= 1.0;", 0),
    ("prefactor_decode_unweighted", "for (int f = 0; f < F; ++f) pk[f] *= wk;",
     "for (int f = 0; f < F; ++f) pk[f] *= 1.0;", 0),
    ("prefactor_noncausal_unweighted", "for (int f = 0; f < D; ++f) pk[f] *= wj;",
     "for (int f = 0; f < D; ++f) pk[f] *= 1.0;", 0),
    ("awd_teacher_without_sqrt_d", "/ sqrt((double)d);", "/ 1.0;", 0),
    ("awd_unnormalised_kernel", "const double r = at[j] / Dn;", "const double r = at[j];", 0),
    ("awd_causal_mask_exclusive", "const int J = causal ? i + 1 : N;",
     "const int J = causal ? (i > 0 ? i : 1) : N;", 0),
    ("awd_unweighted_keys", "for (int f = 0; f < D; ++f) PK[(size_t)i * D + f] *= wk;\n    }\n    double loss",
     "for (int f = 0; f < D; ++f) PK[(size_t)i * D + f] *= 1.0;\n    }\n    double loss", 0),
    ("awd_clamp_value", "(r > 0.0 ? log(r) : log(AWD_EPS))", "(r > 0.0 ? log(r) : log(1e-3))", 0),
    ("awdgrad_drop_row_sum_term", "const double g = -(dl / N) * (first - ci / Dn);",
     "const double g = -(dl / N) * (first);", 0),
    ("awdgrad_no_clamp_mask", "const double first = at[j] / Dn > 0.0 ? P[j] / at[j] : 0.0;",
     "const double first = P[j] / at[j];", 0),
    ("awdgrad_c_over_all_entries", "if (at[j] / Dn > 0.0) ci += P[j];", "ci += P[j];", 0),
    ("awdgrad_dtau_sign", "if (dtau) *dtau += -s * dot(d, kj, kj) * itau;",
     "if (dtau) *dtau += s * dot(d, kj, kj) * itau;", 0),
    ("awdgrad_key_chain_unweighted", "for (int f = 0; f < D; ++f) dPK[(size_t)i * D + f] *= wk[i];",
     "for (int f = 0; f < D; ++f) dPK[(size_t)i * D + f] *= 1.0;", 0),
    ("awdgrad_dtau_weight_twice", "double s = dot(D, PK + (size_t)i * D, dPK + (size_t)i * D);",
     "double s = dot(D, PK + (size_t)i * D, dPK + (size_t)i * D) * wk[i];", 0),
    ("awdgrad_causal_mask_exclusive",
     "const int J = causal ? i + 1 : N;\n        double smax = -INFINITY, Dn = 0.0, Z = 0.0, ci",
     "const int J = causal ? (i > 0 ? i : 1) : N;\n        double smax = -INFINITY, Dn = 0.0, Z = 0.0, ci", 0),
    ("awdgrad_ignores_dloss", "const double g = -(dl / N)", "const double g = -(1.0 / N)", 0),
    ("awdgrad_w2_sign", "dW2[h * per + t] = 0.5 * (dA[t] - dB[t]);",
     "dW2[h * per + t] = 0.5 * (dB[t] - dA[t]);", 0),
    ("awdgrad_drop_query_side",
     "feature_backward(d, M, q + (size_t)i * d, W1, W2, dPQ + (size_t)i * D, dx, dA, dB);",
     "(void)dPQ;", 0),
]


def _apply(src, old, new, occurrence):
    assert src.count(old) >= 1, "mutation target not found in the oracle source"
    pos = -1
    for _ in range(occurrence + 1):
        pos = src.index(old, pos + 1)
    return src[:pos] + new + src[pos + len(old):]


@pytest.mark.parametrize("name,old,new,occ", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, name, old, new, occ):
    with open(oracle.SOURCE) as f:
        src = f.read()
    path = oracle.compile_library(_apply(src, old, new, occ),
                                  os.path.join(str(tmp_path), f"mut_{name}.so"))
    mutant = oracle.Oracle(path)
    failed = []
    with np.errstate(all="ignore"):
        for pin in oracle_pins.ALL_PINS:
            try:
                pin(mutant)
            except (AssertionError, FloatingPointError, ValueError):
                failed.append(pin.__name__)
    assert failed, f"no pin caught the planted mistake {name}"
