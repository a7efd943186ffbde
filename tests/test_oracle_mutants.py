"""Planted mistakes in the oracle must each break at least one pin (CPU only).

Every mutant is a copy of ``oracle/rikfad_oracle.c`` with one plausible
slip -- a dropped term, a wrong sign, a transposed index, a sub-step out of
place -- compiled into a temporary library and run through the fast pins.  A
mutant that passes every pin would mean the pins cannot see that mistake.
"""
import os
import subprocess

import pytest

import oracle
import pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "rikfad_oracle.c")

# (name, text to replace, replacement, which occurrence (0-based) or None for all)
MUTANTS = [
    ("kick_sign", "P[k] = P[k] - h * G[k];", "P[k] = P[k] + h * G[k];", 0),
    ("drift_uses_P_n", "X[k] = X[k] + h * P[k];", "X[k] = X[k] + h * (P[k] + h * G[k]);", 0),
    ("first_damp_full_step", "exp(-0.5 * h * friction_entry", "exp(-1.0 * h * friction_entry", 0),
    ("second_damp_dropped",
     "P[i * n + j] = P[i * n + j] * exp(-0.5 * h * friction_entry(R[i], C[j], denom));",
     "P[i * n + j] = P[i * n + j];", 1),
    ("friction_transposed", "friction_entry(R[i], C[j], denom)",
     "friction_entry(R[j % m], C[i % n], denom)", None),
    ("eps_on_column_total", "double denom = row_factor_total(m, R) + eps_stab;",
     "double denom = row_factor_total(n, C) + eps_stab;", 0),
    ("gain_without_mu", "-expm1(-alpha * h) / (mu * alpha)", "-expm1(-alpha * h) / alpha", 0),
    ("gain_first_order", "-expm1(-alpha * h) / (mu * alpha)", "h / mu", 0),
    ("decay_half", "const double decay = exp(-alpha * h);",
     "const double decay = exp(-0.5 * alpha * h);", 0),
    ("row_factor_from_column_sums", "R[i] = decay * R[i] + gain * rowsq[i];",
     "R[i] = decay * R[i] + gain * colsq[i % n];", 0),
    ("factors_fed_by_kicked_momentum", "const double q = P[i * n + j] * P[i * n + j];",
     "const double q = P[i * n + j] * P[i * n + j] * exp(h * friction_entry(R[i], C[j], "
     "row_factor_total(m, R) + eps_stab));", 0),
    ("damping_half", "const double damp = exp(-gamma * h);",
     "const double damp = exp(-0.5 * gamma * h);", 0),
    ("zero_denominator_unguarded", "if (denom == 0.0)\n        return 0.0;",
     "if (0)\n        return 0.0;", 0),
    ("vector_kick_sign", "p[k] = p[k] - h * g[k];", "p[k] = p[k] + h * g[k];", 0),
    ("vector_friction_fed_undamped", "xi[k] = decay * xi[k] + gain * p[k] * p[k];",
     "xi[k] = decay * xi[k] + gain * p[k] * p[k] * exp(h * xi[k]);", 0),
    ("vector_no_damping", "const double damp = exp(-gamma * h);", "const double damp = 1.0;", 1),
    ("vector_friction_not_updated",
     "for (int64_t k = 0; k < L; ++k)\n        xi[k] = decay * xi[k] + gain * p[k] * p[k];",
     "double xtmp = 0.0; (void)xtmp;", 0),
]


def _mutate(text, old, new, which):
    if which is None:
        assert old in text, old
        return text.replace(old, new)
    idx = -1
    for _ in range(which + 1):
        idx = text.index(old, idx + 1)
    return text[:idx] + new + text[idx + len(old):]


@pytest.mark.parametrize("name,old,new,which", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(name, old, new, which, tmp_path):
    src = _mutate(open(SRC).read(), old, new, which)
    c = tmp_path / "mutant.c"
    c.write_text(src)
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-o",
                    str(so), str(c), "-lm"], check=True)
    saved = oracle._lib
    oracle._lib = oracle.load(str(so))
    failed = []
    try:
        for pin in pins.FAST_PINS:
            try:
                pin()
            except (AssertionError, ValueError, FloatingPointError):
                failed.append(pin.__name__)
    finally:
        oracle._lib = saved
    assert failed, "mutant %s passed every pin" % name
