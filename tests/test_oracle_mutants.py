"""Plausible mistakes planted in a copy of the oracle must each fail a pin.

Each mutant is a text substitution on oracle/fem_oracle.c compiled on the CPU
into a temporary library; the pin checks of ``tests/oracle_pins.py`` are run
against it and at least one must fail.  This shows the pins constrain every
part of the oracle: the score, its scale and operands, the mask, both
log-sum-exps, the beta scaling, the beta = 0 limit and the channel and head
indexing.  No mutant reads outside its buffers.
"""
import os

import pytest

import oracle
from tests import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "fem_oracle.c")

MUTANTS = {
    "drop_score_scale": ("s[i] = dot * scale;", "s[i] = dot;"),
    "causal_mask_ignored": ("const int64_t n = causal ? t + 1 : T;", "const int64_t n = causal ? T : T;"),
    "sign_of_difference": ("out_t[j] = (G - lse) / b;", "out_t[j] = (lse - G) / b;"),
    "drop_lse_term": ("out_t[j] = (G - lse) / b;", "out_t[j] = G / b;"),
    "drop_beta_divide": ("out_t[j] = (G - lse) / b;", "out_t[j] = (G - lse);"),
    "swap_q_and_k": ("fem_oracle_row(q + row * d, k + bh * T * d,", "fem_oracle_row(k + row * d, q + bh * T * d,"),
    "wrong_head_beta": ("beta + h * d, n, d,", "beta + 0 * d, n, d,"),
    "wrong_value_channel": ("g += exp(s[i] + b * vbase[i * d + j] - a_max);",
                            "g += exp(s[i] + b * vbase[i * d + (d - 1 - j)] - a_max);"),
    "drop_beta_in_tilt": ("g += exp(s[i] + b * vbase[i * d + j] - a_max);",
                          "g += exp(s[i] + vbase[i * d + j] - a_max);"),
    "drop_max_add_back": ("const double G = a_max + log(g);", "const double G = log(g);"),
    "lse_without_max": ("const double lse = m + log(z);", "const double lse = log(z);"),
    "mean_unnormalised": ("mu += exp(s[i] - lse) * vbase[i * d + j];", "mu += exp(s[i] - m) * vbase[i * d + j];"),
    "score_self_dot": ("dot += q_t[c] * k_i[c];", "dot += q_t[c] * q_t[c];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique in fem_oracle.c"
    mutant_src = tmp_path / "mutant.c"
    mutant_src.write_text(src.replace(old, new))
    lib_path = oracle.build(force=True, src=str(mutant_src), out=str(tmp_path / "libmutant.so"))
    lib = oracle.load(lib_path)
    failures = []
    for check in oracle_pins.ALL_CHECKS:
        try:
            check(lib)
        except (AssertionError, ValueError, FloatingPointError) as e:
            failures.append(check.__name__)
    assert failures, f"mutant {name} passed every pin"
