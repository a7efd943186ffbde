"""The oracle against the paper and the mathematics (CPU only)."""
import os

import numpy as np
import pytest

import oracle
from oracle import HParams
from paper_2609_30342_gb300 import workloads

import pins
from oracle import explicit

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _table(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


@pytest.mark.parametrize("pin", pins.FAST_PINS, ids=lambda p: p.__name__)
def test_fast_pin(pin):
    pin()


def _slopes(m, n, eps, seed, T, h=0.02):
    """Local slopes of log E vs log t on [1e3, 1e4] (and [1e4, 1e5] if T >= 1e5)
    for the dense quadratic of the paper's numerical-validation section."""
    A, X, P = workloads.dense_quadratic_instance(m, n, seed)
    nsteps = int(round(T / h))
    rec = np.unique(np.round(np.logspace(2, np.log10(T), 300) / h).astype(np.int64))
    E = oracle.dense_quadratic_run(A, X, P, np.zeros(m), np.zeros(n), h, HParams(1.0, 1.0, 0.0, eps),
                                   nsteps, rec)
    t = rec * h
    out = []
    for lo in (1e3, 1e4):
        if lo * 10 <= T * (1 + 1e-12):
            sel = (t >= lo) & (t <= 10 * lo)
            out.append(np.polyfit(np.log(t[sel]), np.log(E[sel]), 1)[0])
    return out


@pytest.mark.parametrize("row", _table("g0_slopes.txt"), ids=lambda r: "eps%s_%sx%s" % tuple(r[:3]))
def test_energy_decay_slopes_match_paper_table(row):
    """Table tab:g0_slopes: the oracle's BACD run on a fresh random instance
    (MATLAB's random streams cannot be reproduced) must reproduce the printed
    slopes.  The paper states the exponents are instance independent; the
    finite-window slopes still move with the instance, most for 2 x 2."""
    eps, m, n = float(row[0]), int(row[1]), int(row[2])
    paper = [float(v) for v in row[3:5]]
    T = 1e5 if m * n <= 12 else 1e4
    got = _slopes(m, n, eps, seed=1, T=T)
    tol = 0.04 if m * n == 4 else 0.02
    for g, p in zip(got, paper):
        assert abs(g - p) < tol, (row, got)


def test_scalar_prefactors_match_paper():
    """Prefactor appendix: m = n = 1, alpha = mu = 1, h = 0.02, t = 1e5 gives
    t E/(alpha mu) = 0.909 (eps_stab = 0) and E sqrt(t)/(alpha mu sqrt(eps/2)) =
    0.884 (eps_stab > 0), within ~10% of the averaging value 1 for any
    instance.  Ours is another random instance: within 6% of the paper's."""
    vals = dict((r[0], float(r[1])) for r in _table("prefactors.txt"))
    h, T = 0.02, 1e5
    n = int(round(T / h))
    for eps, key in ((0.0, "tE_over_alpha_mu_eps0"), (0.1, "E_sqrt_t_over_alpha_mu_sqrt_half_eps")):
        rng = np.random.default_rng(1)
        B = rng.standard_normal((1, 1))
        A = B @ B.T + 0.8 * np.eye(1)
        X = 0.4 * rng.standard_normal((1, 1))
        P = 0.3 * rng.standard_normal((1, 1))
        E = oracle.dense_quadratic_run(A, X, P, np.zeros(1), np.zeros(1), h,
                                       HParams(1.0, 1.0, 0.0, eps), n, [n])[0]
        q = T * E if eps == 0.0 else E * np.sqrt(T) / np.sqrt(eps / 2)
        assert abs(q / vals[key] - 1.0) < 0.06, (key, q)


def test_prefactor_table_parameter_dependence():
    """Table tab:g0_prefactors (m = 3, n = 2, t = 1e4): over the printed
    (alpha, mu) grid, t E/(alpha mu) at eps_stab = 0 moves by less than 30%
    (the caption's claim; printed spread 1.29) and E sqrt(t)/(alpha mu
    sqrt(eps/2)) by less than 20% (printed 1.14), while alpha mu spans a
    factor of 16 (4).  The means depend on the instance (ours is another
    random draw, and the paper integrated the flow, not the map): within 15%
    of the printed 4.69 and 2.31."""
    rows = {r[0]: r for r in _table("g0_prefactor_table.txt")}
    h, T = 0.02, 1e4
    n = int(round(T / h))
    A, X, P = workloads.dense_quadratic_instance(3, 2, 1)

    def energy(al, mu, ep):
        return oracle.dense_quadratic_run(A, X.copy(), P.copy(), np.zeros(3), np.zeros(2), h,
                                          HParams(al, mu, 0.0, ep), n, [n])[0]
    r1 = rows["tE_over_alpha_mu"]
    q1 = np.array([T * energy(al, mu, 0.0) / (al * mu)
                   for al in map(float, r1[2].split(",")) for mu in map(float, r1[2].split(","))])
    r2 = rows["E_sqrt_t_over_alpha_mu_sqrt_half_eps"]
    q2 = np.array([energy(al, mu, ep) * np.sqrt(T) / (al * mu * np.sqrt(ep / 2))
                   for al in map(float, r2[2].split(",")) for mu in map(float, r2[2].split(","))
                   for ep in map(float, r2[1].split(","))])
    assert q1.max() / q1.min() < 1.3, q1
    assert q2.max() / q2.min() < 1.2, q2
    assert abs(q1.mean() / float(r1[3]) - 1) < 0.15, q1.mean()
    assert abs(q2.mean() / float(r2[3]) - 1) < 0.15, q2.mean()


def test_state_size_matches_paper_memory_table():
    """Table tab:memory, GPT2-S row: R-iKFAD 475.4 MiB vs iKFAD/Adam 948.9 MiB
    (fp32).  Our GPT2-S list (separate q/k/v, 74 matrices) must land within
    1 MiB of both and reproduce the printed 2.0x ratio."""
    row = _table("memory_table.txt")[0]
    adam, rikfad = float(row[2]), float(row[6])
    shapes = [s for _, s in workloads.gpt2_small()]
    N = workloads.count(shapes)[0]
    mib = 4.0 / 2 ** 20
    ours = oracle.state_scalars(shapes) * mib
    full = 2 * N * mib
    assert abs(ours - rikfad) < 1.0, ours
    assert abs(full - adam) < 1.0, full
    assert round(full / ours, 1) == 2.0


@pytest.mark.parametrize("gamma", [0.0, 0.1])
def test_energy_decreases_on_convex_quadratic(gamma):
    """f = 1/2 sum A (.) (X - X*)^2 with A ~ U[0.1, 10]: the paper's energy
    E = f - f* + 1/2 ||P||^2 is non-increasing in continuous time (Lemma 1,
    Eq. E_decay); the discrete BACD trajectory must not increase it either
    (to rounding), and must reduce it over 2000 steps."""
    prob = workloads.QuadraticProblem(48, 40, seed=1)
    A = prob.A.astype(np.float64)
    Xs = prob.Xstar.astype(np.float64)
    X, P = prob.X0.astype(np.float64), prob.P0.astype(np.float64)
    R, C = np.zeros(48), np.zeros(40)
    hp = HParams(0.01, 1.0, gamma, 1e-8)
    E_prev = E0 = oracle.diag_quadratic_energy(A, Xs, X, P)
    for _ in range(2000):
        oracle.step_matrix(X, P, R, C, A * (X - Xs), 1e-3, hp)
        E = oracle.diag_quadratic_energy(A, Xs, X, P)
        assert E <= E_prev * (1 + 1e-12)
        E_prev = E
    assert E_prev < 0.2 * E0


@pytest.mark.parametrize("shape", [(1, 1), (4, 3), (7, 5), (33, 17)])
def test_half_damped_momentum_output(shape):
    """The oracle's optional P^(1) output (the stored form of the GPU step):
    equal to the kick P_n - h g when the factors are zero (no friction yet,
    so the first half-damp is the identity), and to the independent numpy
    variant's P^(1) from non-zero factors; the main outputs are unchanged by
    asking for it."""
    m, n = shape
    rng = np.random.default_rng(m * 100 + n)
    X = rng.standard_normal((m, n))
    P = rng.standard_normal((m, n))
    G = rng.standard_normal((m, n))
    hp = HParams(0.7, 0.3, 0.2, 1e-3)
    h = 0.1
    # zero factors: P^(1) = P^(B) exactly
    P1 = np.empty((m, n))
    Xa, Pa, Ra, Ca = X.copy(), P.copy(), np.zeros(m), np.zeros(n)
    oracle.step_matrix(Xa, Pa, Ra, Ca, G, h, hp, P1=P1)
    assert np.array_equal(P1, P - h * G)
    Xb, Pb, Rb, Cb = X.copy(), P.copy(), np.zeros(m), np.zeros(n)
    oracle.step_matrix(Xb, Pb, Rb, Cb, G, h, hp)
    for a, b in ((Xa, Xb), (Pa, Pb), (Ra, Rb), (Ca, Cb)):
        assert np.array_equal(a, b)
    # non-zero factors: against the explicit-friction variant
    R0 = rng.uniform(0.1, 2.0, m)
    C0 = rng.uniform(0.1, 2.0, n)
    Xc, Pc, Rc, Cc = X.copy(), P.copy(), R0.copy(), C0.copy()
    oracle.step_matrix(Xc, Pc, Rc, Cc, G, h, hp, P1=P1)
    ref = explicit.step_matrix_explicit(X, P, R0, C0, G, h, hp.alpha, hp.mu, hp.gamma, hp.eps_stab,
                                        return_p1=True)
    assert np.allclose(P1, ref[4], rtol=1e-13, atol=0.0)
    assert not np.allclose(P1, P - h * G)      # the friction acted
