"""Pins of the diagnostic oracle (oracle/diagnostics.py), CPU only."""
import numpy as np

import oracle
from oracle import HParams
from oracle.diagnostics import friction_metrics, shadow_step


def test_shadow_step_is_elementwise_ikfad():
    """X, P and the friction follow the C oracle's element-wise rule (itself
    pinned to continuous iKFAD)."""
    rng = np.random.default_rng(31)
    m, n = 6, 9
    X, P, G = (rng.standard_normal((m, n)) for _ in range(3))
    XI = rng.uniform(0, 2, (m, n))
    hp = HParams(0.4, 0.3, 0.2)
    X1, P1, XI1, _, _ = shadow_step(X, P, XI, np.zeros(m), np.zeros(n), G, 0.17, hp)
    x, p, xi = X.ravel().copy(), P.ravel().copy(), XI.ravel().copy()
    oracle.step_vector(x, p, xi, G.ravel().copy(), 0.17, hp)
    for a, b in ((X1, x), (P1, p), (XI1, xi)):
        assert np.max(np.abs(a.ravel() - b)) < 1e-13 * np.max(np.abs(b))


def test_shadow_factors_match_rikfad_factors_on_first_step():
    """From zero friction and zero factors, both methods damp nothing in the
    first half-step, so the shadow factors equal R-iKFAD's own factors."""
    rng = np.random.default_rng(32)
    m, n = 5, 7
    X, P, G = (rng.standard_normal((m, n)) for _ in range(3))
    hp = HParams(0.4, 0.3, 0.1, 1e-8)
    _, _, _, R, C = shadow_step(X, P, np.zeros((m, n)), np.zeros(m), np.zeros(n), G, 0.2, hp)
    Rr, Cr = np.zeros(m), np.zeros(n)
    oracle.step_matrix(X.copy(), P.copy(), Rr, Cr, G, 0.2, hp)
    assert np.max(np.abs(R - Rr)) < 1e-14 * np.max(Rr)
    assert np.max(np.abs(C - Cr)) < 1e-14 * np.max(Cr)


def test_eckart_young_floor_is_the_best_rank1_error():
    """The floor sqrt(1 - sigma1^2/||xi||^2) equals the error of the truncated
    SVD sigma1 u1 v1^T, computed separately."""
    rng = np.random.default_rng(33)
    XI = rng.uniform(0, 1, (12, 8)) ** 3
    _, floor, sr, s1, frob = friction_metrics(XI, np.ones(12), np.ones(8), 0.0)
    U, S, Vt = np.linalg.svd(XI)
    best = S[0] * np.outer(U[:, 0], Vt[0])
    assert abs(floor - np.linalg.norm(XI - best) / np.linalg.norm(XI)) < 1e-12
    assert abs(sr - np.sum(S ** 2) / S[0] ** 2) < 1e-12


def test_metrics_closed_forms():
    """Rank-1 friction: floor 0, stable rank 1, and zero error for factors
    that reproduce it; k x k identity: stable rank k, floor sqrt(1 - 1/k)."""
    a, b = np.array([1.0, 2.0, 0.5]), np.array([0.3, 1.0, 2.0, 4.0])
    XI = np.outer(a, b)
    err, floor, sr, s1, frob = friction_metrics(XI, a, b * a.sum(), 0.0)
    assert err < 1e-15 and floor < 1e-7 and abs(sr - 1) < 1e-12
    assert abs(s1 - np.linalg.norm(a) * np.linalg.norm(b)) < 1e-12
    for k in (2, 5):
        err, floor, sr, s1, frob = friction_metrics(np.eye(k), np.ones(k), np.ones(k), 0.0)
        assert abs(sr - k) < 1e-12 and abs(floor - np.sqrt(1 - 1 / k)) < 1e-12
        assert abs(err - np.linalg.norm(np.eye(k) - np.ones((k, k)) / k) / np.sqrt(k)) < 1e-12
    assert friction_metrics(np.zeros((3, 3)), np.zeros(3), np.zeros(3), 0.0) == (0, 0, 0, 0, 0)


def test_rank1_momentum_gives_zero_construction_error():
    """Rank-1 momentum from zero friction and factors (eps_stab = 0): after one
    step the shadow rank-1 friction equals the element-wise friction."""
    rng = np.random.default_rng(34)
    a, b = rng.standard_normal(6), rng.standard_normal(4)
    P = np.outer(a, b)
    hp = HParams(0.5, 0.8, 0.0, 0.0)
    _, _, XI, R, C = shadow_step(np.zeros((6, 4)), P, np.zeros((6, 4)), np.zeros(6), np.zeros(4),
                                 np.zeros((6, 4)), 0.3, hp)
    err, floor, sr, _, _ = friction_metrics(XI, R, C, 0.0)
    assert err < 1e-14 and floor < 1e-7 and abs(sr - 1) < 1e-10
