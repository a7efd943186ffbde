"""Oracle runs executed in worker processes (spawned, so they never inherit a
CUDA context) while the GPU side of a test runs."""
import numpy as np

import oracle
from oracle import HParams
from paper_2609_30342_gb300 import workloads


def quadratic_run(m, n, seed, steps, h, alpha, mu, gamma, eps, snapshots):
    """Config-2 style run: f = 1/2 sum A (.) (X - X*)^2, X(0) = P(0) = 0.
    Returns the energy after every step (index 0 = initial) and (X, P, R, C)
    at the requested step counts."""
    prob = workloads.QuadraticProblem(m, n, seed)
    A = prob.A.astype(np.float64)
    Xs = prob.Xstar.astype(np.float64)
    X, P = prob.X0.astype(np.float64), prob.P0.astype(np.float64)
    R, C = np.zeros(m), np.zeros(n)
    hp = HParams(alpha, mu, gamma, eps)
    energy = [oracle.diag_quadratic_energy(A, Xs, X, P)]
    snaps = {}
    for k in range(1, steps + 1):
        oracle.step_matrix(X, P, R, C, A * (X - Xs), h, hp)
        energy.append(oracle.diag_quadratic_energy(A, Xs, X, P))
        if k in snapshots:
            snaps[k] = (X.copy(), P.copy(), R.copy(), C.copy())
    return np.array(energy), snaps
