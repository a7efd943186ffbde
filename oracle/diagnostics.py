"""Oracle of the friction diagnostic (the paper's Section 4.4, "How close is
xi~ to the best rank-1 friction?"): full iKFAD run with R-iKFAD's factors
carried alongside as shadows, and the error of the rank-1 friction against
the Eckart-Young floor.

TEST INFRASTRUCTURE, like the rest of ``oracle/``: numpy, float64, written
from the paper's sub-steps (Appendix A table) with the element-wise friction
of Eqs. ikfad_1 to ikfad_3; shares no code with the CUDA path.  Pinned in
tests/test_oracle_diagnostics.py.
"""
import numpy as np


def shadow_step(X, P, XI, R, C, G, h, hp):
    """One BACD step of full iKFAD on an m x n matrix (element-wise friction
    XI), with R-iKFAD's factors R, C updated from the same half-damped
    momentum P^(1) by the factor filter of the Appendix A table, without
    entering the update.  Returns new (X, P, XI, R, C)."""
    X, P, XI = (np.array(a, np.float64) for a in (X, P, XI))
    R, C = np.array(R, np.float64), np.array(C, np.float64)
    G = np.asarray(G, np.float64)
    decay = np.exp(-hp.alpha * h)
    gain = (1.0 - np.exp(-hp.alpha * h)) / (hp.mu * hp.alpha)
    PB = P - h * G                                   # B
    X = X + h * PB                                   # A
    P1 = PB * np.exp(-(h / 2) * XI)                  # C, first half-damp with xi_n
    Q = P1 ** 2
    XI = decay * XI + gain * Q                       # C, element-wise friction filter
    R = decay * R + gain * Q.sum(axis=1)             # shadow factors: [P^(1)]^2 1_n
    C = decay * C + gain * Q.sum(axis=0)             # and ([P^(1)]^2)^T 1_m
    P2 = P1 * np.exp(-(h / 2) * XI)                  # C, second half-damp with xi_{n+1}
    P = P2 * np.exp(-hp.gamma * h)                   # D
    return X, P, XI, R, C


def friction_metrics(XI, R, C, eps_stab):
    """(rel_err, eckart_young_floor, stable_rank, sigma1, frob) of the friction
    XI against the rank-1 friction built from R, C (Eq. xi_def), by dense
    linear algebra: sigma1 is the largest singular value (numpy SVD)."""
    XI = np.asarray(XI, np.float64)
    frob2 = float(np.sum(XI * XI))
    if frob2 == 0.0:
        return 0.0, 0.0, 0.0, 0.0, 0.0
    den = float(np.sum(R)) + eps_stab
    XT = np.zeros_like(XI) if den == 0.0 else np.outer(R, C) / den
    rel_err = np.sqrt(float(np.sum((XI - XT) ** 2)) / frob2)
    sigma1 = float(np.linalg.svd(XI, compute_uv=False)[0])
    floor = np.sqrt(max(0.0, 1.0 - sigma1 ** 2 / frob2))
    return rel_err, floor, frob2 / sigma1 ** 2, sigma1, np.sqrt(frob2)
