"""Plant plausible mistakes in a copy of the oracle and check that the pins catch each one.

Each mutant is a one-line textual change to oracle/attn_oracle.c, compiled into a
temporary library on the CPU.  Every mutation keeps all memory accesses in bounds.
A mutant that passes every pin would mean the pins cannot tell that mistake apart
from the right answer.
"""
import os
import subprocess

import pytest

import oracle as oracle_pkg
import oracle_pins

SRC = os.path.join(os.path.dirname(oracle_pkg.__file__), "attn_oracle.c")

MUTANTS = {
    "no_max_shift": ("e[k] = exp(s[k] - m);", "e[k] = exp(s[k]);"),
    "min_instead_of_max": ("if (s[k] > m) m = s[k];", "if (s[k] < m) m = s[k];"),
    "exp_sign_flipped": ("e[k] = exp(s[k] - m);", "e[k] = exp(m - s[k]);"),
    "scale_dropped": ("s[k] = dot * p->scale;", "s[k] = dot;"),
    "key_features_reversed": ("dot += (double)q[j] * (double)kr[j];",
                              "dot += (double)q[j] * (double)kr[p->dk - 1 - j];"),
    "no_normalisation": ("w[k] = e[k] / Z;", "w[k] = e[k];"),
    "sum_skips_first": ("for (int64_t k = 0; k < p->Nk; ++k)\n        Z += e[k];",
                        "for (int64_t k = 1; k < p->Nk; ++k)\n        Z += e[k];"),
    "v_transposed": ("acc += w[k] * (double)Vh[k * p->dv + c];",
                     "acc += w[k] * (double)Vh[c * p->Nk + k];"),
    "all_heads_share_k": ("const float *Kh = p->K + bh * p->Nk * p->dk;",
                          "const float *Kh = p->K;"),
    "wrong_query_row": ("const float *q = p->Q + (bh * p->Nq + i) * p->dk;",
                        "const float *q = p->Q + (bh * p->Nq) * p->dk;"),
    "lse_without_max": ("if (lse_out) *lse_out = m + log(Z);", "if (lse_out) *lse_out = log(Z);"),
    "lse_log2": ("if (lse_out) *lse_out = m + log(Z);", "if (lse_out) *lse_out = m + log2(Z);"),
    "bwd_drops_rank_one_term": ("dS[k] = w[k] * (dP[k] - wdp);", "dS[k] = w[k] * dP[k];"),
    "bwd_sign_flipped": ("dS[k] = w[k] * (dP[k] - wdp);", "dS[k] = w[k] * (wdp - dP[k]);"),
    "bwd_dk_without_scale": ("dKh[k * dk + j] += scale * dS[k] * (double)q[j];",
                             "dKh[k * dk + j] += dS[k] * (double)q[j];"),
    "bwd_dv_from_ds": ("dVh[k * dv + c] += w[k] * (double)g[c];",
                       "dVh[k * dv + c] += dS[k] * (double)g[c];"),
    "bwd_dp_v_transposed": ("acc += (double)g[c] * (double)Vh[k * dv + c];",
                            "acc += (double)g[c] * (double)Vh[c * Nk + k];"),
    "proj_columns_shifted": ("acc += (double)x[c] * (double)W[c * ncol + col];",
                             "acc += (double)x[c] * (double)W[c * ncol + (col + H * dk) % ncol];"),
    "proj_head_feature_swapped": ("const int64_t h = col / dk, j = col % dk;",
                                  "const int64_t j = col / dk % dk, h = col % dk % H;"),
    "proj_w_transposed": ("acc += (double)x[c] * (double)W[c * ncol + col];",
                          "acc += (double)x[c] * (double)W[(col % d) * ncol + c];"),
    "bwd_dq_uses_q": ("acc += dS[k] * (double)Kh[k * dk + j];",
                      "acc += dS[k] * (double)Kh[j];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name, tmp_path):
    old, new = MUTANTS[name]
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation site for {name} not found exactly once"
    src = tmp_path / f"mutant_{name}.c"
    src.write_text(text.replace(old, new))
    lib = tmp_path / f"libmutant_{name}.so"
    r = subprocess.run(["gcc", *oracle_pkg.CFLAGS, str(src), "-o", str(lib), "-lm"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    mutant = oracle_pkg.Oracle(str(lib))
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(mutant)
        except (AssertionError, RuntimeError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"no pin detects mutant {name}"
