"""Second, independent oracle variant: the R-iKFAD matrix step with the m x n
rank-1 friction tensor materialised (small matrices only).

TEST INFRASTRUCTURE, like the rest of ``oracle/``.  It is written with numpy
whole-array operations and shares nothing with ``rikfad_oracle.c``, so that
an indexing mistake in the C loops (a transposed factor, a row sum taken over
columns) shows up as a disagreement between the two.

Follows Appendix A, Table "Analytical sub-step update rules", with Eq. xi_def
for the friction and the zero-denominator convention of Theorem 3.
"""
import numpy as np


def friction_tensor(R, C, eps_stab):
    """xi~ = R C^T / (1_m^T R + eps_stab) as an explicit m x n array (Eq. xi_def)."""
    denom = float(np.sum(R)) + eps_stab
    if denom == 0.0:
        return np.zeros((R.size, C.size))
    return np.outer(R, C) / denom


def step_matrix_explicit(X, P, R, C, G, h, alpha, mu, gamma, eps_stab, return_p1=False):
    """Return (X, P, R, C) after one BACD step (and P^(1), the half-damped
    momentum of sub-step C, if ``return_p1``); inputs are not modified."""
    X = np.array(X, np.float64)
    P = np.array(P, np.float64)
    R = np.array(R, np.float64)
    C = np.array(C, np.float64)
    G = np.asarray(G, np.float64)
    PB = P - h * G                                        # B
    X = X + h * PB                                        # A
    P1 = PB * np.exp(-(h / 2) * friction_tensor(R, C, eps_stab))   # C, first half
    decay = np.exp(-alpha * h)
    gain = (1.0 - np.exp(-alpha * h)) / (mu * alpha)
    Q = P1 ** 2
    R = decay * R + gain * Q.sum(axis=1)                  # [P1]^2 1_n
    C = decay * C + gain * Q.sum(axis=0)                  # ([P1]^2)^T 1_m
    P2 = P1 * np.exp(-(h / 2) * friction_tensor(R, C, eps_stab))   # C, second half
    P = P2 * np.exp(-gamma * h)                           # D
    if return_p1:
        return X, P, R, C, P1
    return X, P, R, C
