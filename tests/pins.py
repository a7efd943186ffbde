"""Pins of the oracle: checks against facts that do not come from the oracle.

Each ``pin_*`` function raises ``AssertionError`` when the oracle disagrees
with the mathematics or with numbers the paper prints.  ``FAST_PINS`` are
cheap enough to be re-run against deliberately broken copies of the oracle
(tests/test_oracle_mutants.py), which shows that a plausible mistake anywhere
in it is caught.
"""
import numpy as np
from scipy.integrate import solve_ivp

import oracle
from oracle import HParams
from oracle.explicit import step_matrix_explicit


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


def _random_state(rng, m, n, factors=True):
    X = rng.standard_normal((m, n))
    P = rng.standard_normal((m, n))
    G = rng.standard_normal((m, n))
    if factors:
        R = rng.uniform(0.05, 1.5, m)
        C = rng.uniform(0.05, 2.5, n)
    else:
        R, C = np.zeros(m), np.zeros(n)
    return X, P, R, C, G


def pin_explicit_agreement():
    """C loops == numpy with the m x n friction tensor materialised."""
    rng = np.random.default_rng(11)
    cases = [(1, 1), (2, 2), (4, 3), (7, 5), (3, 8), (1, 7), (6, 1)]
    settings = [(0.0, 0.0, True), (0.0, 0.0, False), (1e-8, 0.4, True), (0.3, 0.0, True),
                (0.3, 0.7, False)]
    for m, n in cases:
        for eps, gamma, factors in settings:
            X, P, R, C, G = _random_state(rng, m, n, factors)
            h, alpha, mu = 0.13, 0.6, 0.8
            ref = step_matrix_explicit(X, P, R, C, G, h, alpha, mu, gamma, eps)
            got = [a.copy() for a in (X, P, R, C)]
            oracle.step_matrix(got[0], got[1], got[2], got[3], G, h, HParams(alpha, mu, gamma, eps))
            for g, r in zip(got, ref):
                assert _rel(g, r) < 1e-13, (m, n, eps, gamma, _rel(g, r))


def pin_pure_decay():
    """P = 0 and zero gradient: X is unchanged, P stays 0 and the factors
    decay exactly as dR/dt = -alpha R (the forcing [P]^2 vanishes)."""
    rng = np.random.default_rng(12)
    for eps in (0.0, 1e-8, 0.5):
        m, n = 5, 3
        X = rng.standard_normal((m, n))
        P = np.zeros((m, n))
        R0 = rng.uniform(0.1, 1.0, m)
        C0 = rng.uniform(0.1, 1.0, n)
        R, C, X1 = R0.copy(), C0.copy(), X.copy()
        h, alpha = 0.37, 0.9
        oracle.step_matrix(X1, P, R, C, np.zeros((m, n)), h, HParams(alpha, 2.0, 0.3, eps))
        assert np.array_equal(X1, X)
        assert np.all(P == 0.0)
        assert _rel(R, np.exp(-alpha * h) * R0) < 1e-15
        assert _rel(C, np.exp(-alpha * h) * C0) < 1e-15
        x, p, xi = X[0].copy(), np.zeros(n), C0.copy()
        oracle.step_vector(x, p, xi, np.zeros(n), h, HParams(alpha, 2.0, 0.3))
        assert np.array_equal(x, X[0]) and np.all(p == 0.0)
        assert _rel(xi, np.exp(-alpha * h) * C0) < 1e-15


def pin_factor_filter_ode():
    """With the friction negligible (huge eps_stab) the momentum after the
    first half-damp is P^(B) = P - h G, and the factors must equal the
    solution of dR/dt = [P^(B)]^2 1_n / mu - alpha R, dC/dt = ([P^(B)]^2)^T 1_m / mu
    - alpha C over one step, integrated numerically."""
    rng = np.random.default_rng(13)
    m, n = 4, 6
    X, P, R0, C0, G = _random_state(rng, m, n)
    h, alpha, mu = 0.21, 0.8, 1.7
    R, C, P1 = R0.copy(), C0.copy(), P.copy()
    oracle.step_matrix(X.copy(), P1, R, C, G, h, HParams(alpha, mu, 0.0, 1e300))
    PB = P - h * G
    q_row, q_col = (PB ** 2).sum(axis=1), (PB ** 2).sum(axis=0)

    def rhs(t, y):
        return np.concatenate([q_row / mu - alpha * y[:m], q_col / mu - alpha * y[m:]])

    sol = solve_ivp(rhs, (0.0, h), np.concatenate([R0, C0]), method="DOP853", rtol=1e-13,
                    atol=1e-15)
    ref = sol.y[:, -1]
    assert _rel(R, ref[:m]) < 1e-10, _rel(R, ref[:m])
    assert _rel(C, ref[m:]) < 1e-10, _rel(C, ref[m:])
    assert _rel(P1, PB) < 1e-14


def _c_field(m, n, alpha, mu, eps):
    def rhs(t, y):
        P = y[:m * n].reshape(m, n)
        R = y[m * n:m * n + m]
        C = y[m * n + m:]
        xi = np.outer(R, C) / (R.sum() + eps)
        return np.concatenate([(-xi * P).ravel(), (P ** 2).sum(axis=1) / mu - alpha * R,
                               (P ** 2).sum(axis=0) / mu - alpha * C])
    return rhs


def _order(errs):
    e = np.asarray(errs)
    return np.log2(e[:-1] / e[1:])


def pin_substep_c_local_order():
    """With zero gradient and gamma = 0 one step leaves (P, R, C) at the
    symmetric approximation of the flow of the C vector field (Section 2,
    splitting): its local error must shrink like h^3.  Factors start with
    sum R != sum C so the placement of eps_stab (on 1^T R) matters."""
    rng = np.random.default_rng(14)
    m, n = 3, 4
    X, P0, R0, C0, _ = _random_state(rng, m, n)
    alpha, mu, eps = 0.7, 1.3, 0.3
    rhs = _c_field(m, n, alpha, mu, eps)
    errs = []
    for h in (0.2, 0.1, 0.05, 0.025):
        P, R, C = P0.copy(), R0.copy(), C0.copy()
        oracle.step_matrix(X.copy(), P, R, C, np.zeros((m, n)), h, HParams(alpha, mu, 0.0, eps))
        y = solve_ivp(rhs, (0.0, h), np.concatenate([P0.ravel(), R0, C0]), method="DOP853",
                      rtol=1e-13, atol=1e-15).y[:, -1]
        errs.append(np.linalg.norm(np.concatenate([P.ravel(), R, C]) - y))
    orders = _order(errs)
    assert np.all((orders > 2.7) & (orders < 3.3)), (errs, orders)


def _full_field(a, Xs, alpha, mu, gamma, eps):
    m, n = a.shape

    def rhs(t, y):
        X = y[:m * n].reshape(m, n)
        P = y[m * n:2 * m * n].reshape(m, n)
        R = y[2 * m * n:2 * m * n + m]
        C = y[2 * m * n + m:]
        xi = np.outer(R, C) / (R.sum() + eps)
        dP = -a * (X - Xs) - xi * P - gamma * P
        return np.concatenate([P.ravel(), dP.ravel(), (P ** 2).sum(axis=1) / mu - alpha * R,
                               (P ** 2).sum(axis=0) / mu - alpha * C])
    return rhs


def pin_full_step_first_order():
    """The BACD map converges at first order to the continuous R-iKFAD system
    (Eqs. rikfad_x to rikfad_C) on f = 1/2 sum a (.) (X - X*)^2."""
    rng = np.random.default_rng(15)
    m, n = 3, 4
    a = rng.uniform(0.5, 2.0, (m, n))
    Xs = rng.standard_normal((m, n))
    X0, P0, R0, C0, _ = _random_state(rng, m, n)
    alpha, mu, gamma, eps, T = 0.7, 1.3, 0.25, 0.3, 1.0
    y0 = np.concatenate([X0.ravel(), P0.ravel(), R0, C0])
    ref = solve_ivp(_full_field(a, Xs, alpha, mu, gamma, eps), (0.0, T), y0, method="DOP853",
                    rtol=1e-13, atol=1e-14).y[:, -1]
    errs = []
    for N in (50, 100, 200, 400):
        h = T / N
        X, P, R, C = X0.copy(), P0.copy(), R0.copy(), C0.copy()
        for _ in range(N):
            oracle.step_matrix(X, P, R, C, a * (X - Xs), h, HParams(alpha, mu, gamma, eps))
        errs.append(np.linalg.norm(np.concatenate([X.ravel(), P.ravel(), R, C]) - ref))
    orders = _order(errs)
    assert np.all((orders > 0.9) & (orders < 1.1)), (errs, orders)
    assert errs[-1] < 0.02, errs


def pin_vector_rule_orders():
    """The element-wise rule for 1-D parameters converges at first order to
    continuous iKFAD (Eqs. ikfad_1 to ikfad_3), and its friction sub-step has
    third-order local error."""
    rng = np.random.default_rng(16)
    L = 5
    a = rng.uniform(0.5, 2.0, L)
    xs = rng.standard_normal(L)
    x0, p0 = rng.standard_normal(L), rng.standard_normal(L)
    xi0 = rng.uniform(0.1, 1.0, L)
    alpha, mu, gamma, T = 0.7, 1.3, 0.25, 1.0

    def full(t, y):
        x, p, xi = y[:L], y[L:2 * L], y[2 * L:]
        return np.concatenate([p, -a * (x - xs) - (gamma + xi) * p, p * p / mu - alpha * xi])

    ref = solve_ivp(full, (0.0, T), np.concatenate([x0, p0, xi0]), method="DOP853", rtol=1e-13,
                    atol=1e-14).y[:, -1]
    errs = []
    for N in (50, 100, 200, 400):
        h = T / N
        x, p, xi = x0.copy(), p0.copy(), xi0.copy()
        for _ in range(N):
            oracle.step_vector(x, p, xi, a * (x - xs), h, HParams(alpha, mu, gamma))
        errs.append(np.linalg.norm(np.concatenate([x, p, xi]) - ref))
    orders = _order(errs)
    assert np.all((orders > 0.9) & (orders < 1.1)), (errs, orders)

    def cfield(t, y):
        p, xi = y[:L], y[L:]
        return np.concatenate([-xi * p, p * p / mu - alpha * xi])

    errs = []
    for h in (0.2, 0.1, 0.05, 0.025):
        x, p, xi = x0.copy(), p0.copy(), xi0.copy()
        oracle.step_vector(x, p, xi, np.zeros(L), h, HParams(alpha, mu, 0.0))
        y = solve_ivp(cfield, (0.0, h), np.concatenate([p0, xi0]), method="DOP853", rtol=1e-13,
                      atol=1e-15).y[:, -1]
        errs.append(np.linalg.norm(np.concatenate([p, xi]) - y))
    orders = _order(errs)
    assert np.all((orders > 2.7) & (orders < 3.3)), (errs, orders)


def pin_heavy_ball_closed_form():
    """With the friction switched off (mu = inf keeps R = C = 0) the step is
    kick, drift with the kicked momentum, then damping by e^{-gamma h}: on
    f = 1/2 a (x - x*)^2 each entry follows the linear recurrence
        [x - x*, p]_{k+1} = M [x - x*, p]_k,
        M = [[1 - h^2 a, h], [-e^{-gamma h} h a, e^{-gamma h}]],
    whose k-th power gives the state in closed form."""
    rng = np.random.default_rng(17)
    m, n, h, K = 2, 3, 0.1, 60
    a = rng.uniform(0.5, 3.0, (m, n))
    Xs = rng.standard_normal((m, n))
    for gamma in (0.0, 0.3):
        for rule in ("matrix", "vector"):
            X0, P0 = rng.standard_normal((m, n)), rng.standard_normal((m, n))
            X, P = X0.copy(), P0.copy()
            hp = HParams(0.5, np.inf, gamma, 1e-8)
            if rule == "matrix":
                R, C = np.zeros(m), np.zeros(n)
                for _ in range(K):
                    oracle.step_matrix(X, P, R, C, a * (X - Xs), h, hp)
            else:
                x, p, xi = X.ravel().copy(), P.ravel().copy(), np.zeros(m * n)
                for _ in range(K):
                    oracle.step_vector(x, p, xi, (a * (x.reshape(m, n) - Xs)).ravel(), h, hp)
                X, P = x.reshape(m, n), p.reshape(m, n)
            e = np.exp(-gamma * h)
            for i in range(m):
                for j in range(n):
                    M = np.array([[1 - h * h * a[i, j], h], [-e * h * a[i, j], e]])
                    v = np.linalg.matrix_power(M, K) @ np.array([X0[i, j] - Xs[i, j], P0[i, j]])
                    assert abs(X[i, j] - Xs[i, j] - v[0]) < 1e-12, (rule, gamma)
                    assert abs(P[i, j] - v[1]) < 1e-12, (rule, gamma)


def pin_symplectic_invariant():
    """gamma = 0 and no friction: kick-then-drift on f = 1/2 w^2 x^2 is the
    symplectic Euler map, which conserves p^2 + w^2 x^2 - h w^2 x p exactly."""
    w2, h = 2.5, 0.05
    X, P = np.array([[0.7]]), np.array([[-0.3]])
    R, C = np.zeros(1), np.zeros(1)
    q0 = P[0, 0] ** 2 + w2 * X[0, 0] ** 2 - h * w2 * X[0, 0] * P[0, 0]
    for _ in range(2000):
        oracle.step_matrix(X, P, R, C, w2 * X, h, HParams(1.0, np.inf, 0.0, 1e-8))
    q = P[0, 0] ** 2 + w2 * X[0, 0] ** 2 - h * w2 * X[0, 0] * P[0, 0]
    assert abs(q - q0) < 1e-12 * abs(q0), (q, q0)


def pin_rank1_equivalence():
    """From R = C = 0 with eps_stab = 0, a rank-1 squared momentum makes the
    factored friction equal element-wise iKFAD's (Eq. xi_def against Eqs.
    ikfad_1 to ikfad_3): after one step R_i C_j / 1^T R = k P1_ij^2 = xi_ij, so
    the matrix rule and the element-wise rule give the same X and P."""
    rng = np.random.default_rng(18)
    for m, n in ((1, 1), (3, 5), (6, 2)):
        a, b = rng.standard_normal(m), rng.standard_normal(n)
        X = rng.standard_normal((m, n))
        P = np.outer(a, b)
        hp = HParams(0.4, 0.7, 0.2, 0.0)
        h = 0.3
        Xm, Pm, R, C = X.copy(), P.copy(), np.zeros(m), np.zeros(n)
        oracle.step_matrix(Xm, Pm, R, C, np.zeros((m, n)), h, hp)
        x, p, xi = X.ravel().copy(), P.ravel().copy(), np.zeros(m * n)
        oracle.step_vector(x, p, xi, np.zeros(m * n), h, hp)
        assert _rel(Xm.ravel(), x) < 1e-14
        assert _rel(Pm.ravel(), p) < 1e-13
        assert _rel(np.outer(R, C).ravel() / R.sum(), xi) < 1e-13


def pin_invariants():
    """Along a random run from R = C = 0: R, C >= 0, 0 <= xi~_ij <= C_j
    (Lemma 1) and sum R = sum C (the two totals obey the same scalar
    equation, rates appendix)."""
    rng = np.random.default_rng(19)
    m, n = 5, 7
    X, P = rng.standard_normal((m, n)), rng.standard_normal((m, n))
    R, C = np.zeros(m), np.zeros(n)
    hp = HParams(0.3, 0.5, 0.0, 1e-3)
    for _ in range(60):
        oracle.step_matrix(X, P, R, C, rng.standard_normal((m, n)), 0.05, hp)
        assert np.all(R >= 0) and np.all(C >= 0)
        xi = np.outer(R, C) / (R.sum() + hp.eps_stab)
        assert np.all(xi <= C[None, :] * (1 + 1e-15))
        assert abs(R.sum() - C.sum()) <= 1e-12 * R.sum()


FAST_PINS = [pin_explicit_agreement, pin_pure_decay, pin_factor_filter_ode,
             pin_substep_c_local_order, pin_full_step_first_order, pin_vector_rule_orders,
             pin_heavy_ball_closed_form, pin_symplectic_invariant, pin_rank1_equivalence,
             pin_invariants]
