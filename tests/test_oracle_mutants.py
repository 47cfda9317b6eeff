"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake in a temporary copy of oracle/nest_oracle.c
(on the CPU), builds it, and runs the pin suite against it through
NEST_ORACLE_LIB; the suite must fail.  The committed oracle is untouched.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "nest_oracle.c")

MUTANTS = {
    "dropped_square": ("acc += diff * diff;", "acc += diff;"),
    "wrong_sign": ("                            - oracle_elem(K, dtype",
                   "                            + oracle_elem(K, dtype"),
    "transposed_output": ("D[(int64_t)b * n + i] = acc;", "D[i * (int64_t)B + b] = acc;"),
    "reversed_tie_break": ("if (x->idx < y->idx) return -1;", "if (x->idx < y->idx) return 1;"),
    "dropped_mu_in_numerator": ("p_knn[values[idx[i]]] += exp(mu * (s[i] - s_max)) / Z;",
                                "p_knn[values[idx[i]]] += exp((s[i] - s_max)) / Z;"),
    "no_max_subtraction": ("Z += exp(mu * (s[i] - s_max));", "Z += exp(mu * s[i]);"),
    "swapped_lambda": ("(1.0 - lambda) * p_knn[w]", "lambda * p_knn[w]"),
    "rrc_without_abs": ("double a = fabs(s[i]);", "double a = s[i];"),
    "argmax_ties_to_larger_id": ("if (p_m[w] > p_m[best]) best = w;",
                                 "if (p_m[w] >= p_m[best]) best = w;"),
    "span_start_farthest": ("if (key < 0 || s[i] > key_s", "if (key < 0 || s[i] < key_s"),
    "span_rule_strict": ("*use_span = (lambda <= delta && key >= 0)",
                         "*use_span = (lambda < delta && key >= 0)"),
    "verify_without_gamma": ("ratio[b] = mx > 0.0 ? p / (gamma * mx) : 0.0;",
                             "ratio[b] = mx > 0.0 ? p / mx : 0.0;"),
    "verify_accepts_half": ("accept[b] = a > 0.5 ? 1 : 0;", "accept[b] = a >= 0.5 ? 1 : 0;"),
    "rrc_sigmoid_sign": ("return 1.0 / (1.0 + exp(-(ratio - alpha) / tau));",
                         "return 1.0 / (1.0 + exp((ratio - alpha) / tau));"),
    "rrc_ratio_inverted": ("double ratio = (hi == 0.0) ? 1.0 : lo / hi;",
                           "double ratio = (lo == 0.0) ? 1.0 : hi / lo;"),
    "rrc_counts_padding": ("        if (idx[i] < 0) continue;\n        double a = fabs(s[i]);",
                           "        double a = fabs(s[i]);"),
    "verify_counts_past_a_rejection": (
        "while (span_off[j] + n < span_off[j + 1] && accept[span_off[j] + n]) ++n;",
        "for (int32_t t = span_off[j]; t < span_off[j + 1]; ++t) n += accept[t];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    mutant_c = tmp_path / "mutant.c"
    mutant_c.write_text(src.replace(old, new))
    lib = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                    "-std=c11", str(mutant_c), "-o", str(lib), "-lm"], check=True)
    env = dict(os.environ, NEST_ORACLE_LIB=str(lib))
    res = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                          os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                         env=env, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert res.returncode != 0, f"pins did not catch mutant {name}:\n{res.stdout[-2000:]}"
