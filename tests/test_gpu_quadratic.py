"""Batched BACD integration on small dense quadratics (rikfad_quadratic_run)
against the oracle and the paper's Table tab:g0_slopes (GPU).

Tolerance: the kernel integrates in float32, the oracle in float64 from the
same float32 inputs.  The gamma = 0 dynamics are dissipative, so float32
rounding does not compound along the trajectory: a float32 re-statement of
the steps (numpy, float32 at every operation) stays within 3e-5 of the
float64 energies and within 3e-5 of the state's rms, from a few steps to
2e4 steps.  The bounds below are about eight times that: energies within
2e-4 relative, states within 2e-4 * (|ref| + rms(ref)).
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import HParams
from paper_2609_30342_gb300 import g0_table, rikfad, workloads

from gpu_helpers import compare

pytestmark = pytest.mark.gpu

E_RTOL = 2e-4
S_RTOL = 2e-4
H = 0.02


def _gpu_state(A, X, P, R=None, C=None):
    dev = torch.device("cuda")
    b, m, n = X.shape
    st = dict(A=torch.from_numpy(np.ascontiguousarray(A, np.float32)).to(dev),
              X=torch.from_numpy(np.ascontiguousarray(X, np.float32)).to(dev),
              P=torch.from_numpy(np.ascontiguousarray(P, np.float32)).to(dev),
              R=torch.zeros(b, m, device=dev) if R is None else torch.from_numpy(R).to(dev),
              C=torch.zeros(b, n, device=dev) if C is None else torch.from_numpy(C).to(dev))
    return st


def _run(st, nsteps, rec, hp):
    recd = torch.as_tensor(np.asarray(rec, np.int64)).to("cuda")
    E = torch.full((len(rec), st["X"].shape[0]), float("nan"), device="cuda")
    rikfad.quadratic_run(st["A"], st["X"], st["P"], st["R"], st["C"], H, hp.alpha, hp.mu, hp.gamma,
                         hp.eps_stab, nsteps, recd if len(rec) else None, E if len(rec) else None)
    torch.cuda.synchronize()
    return E.cpu().numpy()


def _oracle(A, X, P, nsteps, rec, hp, R=None, C=None):
    m, n = X.shape
    X, P = X.astype(np.float64).copy(), P.astype(np.float64).copy()
    R = np.zeros(m) if R is None else R.astype(np.float64).copy()
    C = np.zeros(n) if C is None else C.astype(np.float64).copy()
    E = oracle.dense_quadratic_run(A.astype(np.float64), X, P, R, C, H, hp, nsteps, rec)
    return E, X, P, R, C


SHAPES = [(1, 1), (2, 2), (4, 3), (6, 5), (3, 7), (4, 8), (1, 32), (32, 1), (5, 1), (2, 9)]


@pytest.mark.parametrize("m,n", SHAPES)
@pytest.mark.parametrize("eps,gamma", [(0.0, 0.0), (0.1, 0.0), (1e-3, 0.05)])
def test_quadratic_run_matches_oracle(m, n, eps, gamma):
    """Seven instances per shape (a ragged last warp for every packing of
    systems per warp), 3000 steps: energies at the recorded steps and the
    final X, P, R, C against the float64 oracle."""
    seeds = list(range(11, 18))
    A, X, P = workloads.dense_quadratic_batch(m, n, seeds)
    hp = HParams(1.0, 1.0, gamma, eps)
    rec = [0, 1, 2, 10, 100, 1000, 2999, 3000]
    st = _gpu_state(A, X, P)
    Eg = _run(st, 3000, rec, hp)
    for s in range(len(seeds)):
        E, Xo, Po, Ro, Co = _oracle(A[s], X[s], P[s], 3000, rec, hp)
        assert np.all(np.abs(Eg[:, s] - E) <= E_RTOL * E), (s, Eg[:, s], E)
        compare("X", st["X"][s].cpu().numpy(), Xo, S_RTOL, 1.0)
        compare("P", st["P"][s].cpu().numpy(), Po, S_RTOL, 1.0)
        compare("R", st["R"][s].cpu().numpy(), Ro, S_RTOL, 1.0)
        compare("C", st["C"][s].cpu().numpy(), Co, S_RTOL, 1.0)


def test_first_step_matches_oracle_per_element():
    """One step from non-zero factors, so the friction, the half-damps and the
    factor filter all act: element-wise against the oracle at the one-step
    bound of the multi-tensor path (1e-5, floor 1e-2 rms)."""
    m, n = 6, 5
    A, X, P = workloads.dense_quadratic_batch(m, n, [3, 4, 5])
    rng = np.random.default_rng(7)
    R = rng.uniform(0.01, 1.0, (3, m)).astype(np.float32)
    C = rng.uniform(0.01, 1.0, (3, n)).astype(np.float32)
    hp = HParams(1.0, 1.0, 0.02, 1e-3)
    st = _gpu_state(A, X, P, R.copy(), C.copy())
    Eg = _run(st, 1, [0, 1], hp)
    for s in range(3):
        E, Xo, Po, Ro, Co = _oracle(A[s], X[s], P[s], 1, [0, 1], hp, R[s], C[s])
        assert np.all(np.abs(Eg[:, s] - E) <= 1e-5 * E)
        for name, g, r in (("X", st["X"], Xo), ("P", st["P"], Po), ("R", st["R"], Ro), ("C", st["C"], Co)):
            compare(name, g[s].cpu().numpy(), r, 1e-5, 1e-2)


def test_split_run_at_launch_boundary_is_bit_identical():
    """70000 steps in one call (launches of 65536 steps) equal 65536 + 4464
    steps in two calls bit for bit (state and the energies recorded in both
    halves); a split inside a launch (400 + 600 of 1000 steps) agrees to
    float32 rounding."""
    A, X, P = workloads.dense_quadratic_batch(4, 3, range(1, 40))
    hp = HParams(1.0, 1.0, 0.0, 0.1)
    one = _gpu_state(A, X, P)
    E1 = _run(one, 70000, [0, 150, 65536, 69999, 70000], hp)
    two = _gpu_state(A, X, P)
    Ea = _run(two, 65536, [0, 150, 65536], hp)
    Eb = _run(two, 4464, [0, 4463, 4464], hp)
    for k in "XPRC":
        assert torch.equal(one[k], two[k]), k
    assert np.array_equal(E1, np.concatenate([Ea, Eb[1:]]))
    one, two = _gpu_state(A, X, P), _gpu_state(A, X, P)
    E1 = _run(one, 1000, [1000], hp)
    _run(two, 400, [], hp)
    E2 = _run(two, 600, [600], hp)
    assert np.allclose(E1, E2, rtol=1e-5, atol=0)
    for k in "XPRC":
        compare(k, two[k].cpu().numpy(), one[k].cpu().numpy(), 1e-4, 1.0)


def test_zero_steps_and_record_handling():
    """nsteps = 0 leaves the state untouched and records E(0); records out of
    range leave their energies untouched; duplicates repeat the value."""
    A, X, P = workloads.dense_quadratic_batch(2, 2, [1, 2, 3])
    hp = HParams(1.0, 1.0, 0.0, 0.0)
    st = _gpu_state(A, X, P)
    X0 = st["X"].clone()
    E = _run(st, 0, [-5, 0, 0, 3], hp)
    assert torch.equal(st["X"], X0)
    assert np.all(np.isnan(E[0])) and np.all(np.isnan(E[3]))
    assert np.array_equal(E[1], E[2])
    for s in range(3):
        ref = oracle.dense_quadratic_run(A[s].astype(np.float64), X[s].astype(np.float64),
                                         P[s].astype(np.float64), np.zeros(2), np.zeros(2), H, hp, 0, [0])
        assert abs(E[1, s] - ref[0]) <= 1e-6 * ref[0]


def test_large_batch_sampled_against_oracle():
    """20000 systems of 6 x 5 (several waves of blocks) for 200 steps; a
    sample of systems against the oracle."""
    seeds = np.arange(20000)
    A, X, P = workloads.dense_quadratic_batch(6, 5, seeds)
    hp = HParams(1.0, 1.0, 0.0, 0.1)
    st = _gpu_state(A, X, P)
    Eg = _run(st, 200, [0, 200], hp)
    for s in (0, 1, 4095, 12345, 19999):
        E, Xo, _, _, _ = _oracle(A[s], X[s], P[s], 200, [0, 200], hp)
        assert np.all(np.abs(Eg[:, s] - E) <= E_RTOL * E)
        compare("X", st["X"][s].cpu().numpy(), Xo, S_RTOL, 1.0)


def test_bad_arguments_raise():
    A, X, P = workloads.dense_quadratic_batch(6, 6, [1])
    st = _gpu_state(A, X, P)
    with pytest.raises(rikfad.RikfadError):   # m n = 36 > 32
        _run(st, 1, [], HParams(1.0, 1.0, 0.0, 0.0))
    A, X, P = workloads.dense_quadratic_batch(2, 2, [1])
    st = _gpu_state(A, X, P)
    with pytest.raises(rikfad.RikfadError):
        _run(st, 1, [], HParams(-1.0, 1.0, 0.0, 0.0))


def _paper_rows():
    import os
    rows = []
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "g0_slopes.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                v = line.split()
                rows.append((float(v[0]), int(v[1]), int(v[2]), [float(x) for x in v[3:]]))
    return rows


def test_decade_slope_matches_oracle():
    """The first decade's slope [1e3, 1e4] of the seed-1 instance, from the
    GPU run and from the float64 oracle run of the same instance, agree to
    1e-3 for every row of the table."""
    for eps, m, n, _ in _paper_rows():
        run = g0_table.Run(m, n, eps, [1], 1e4, H)
        run.launch()
        t, E = run.energies()
        got = g0_table.decade_slopes(t, E, [1e3])[0, 0]
        A, X, P = workloads.dense_quadratic_batch(m, n, [1])
        k = workloads.log_records(1e4, H)
        Eo, *_ = _oracle(A[0], X[0], P[0], int(round(1e4 / H)), k, HParams(1.0, 1.0, 0.0, eps))
        ref = g0_table.decade_slopes(k * H, Eo[:, None], [1e3])[0, 0]
        assert abs(got - ref) < 1e-3, (eps, m, n, got, ref)


def test_chunked_run_is_bit_identical_to_one_call():
    """g0_table issues a long run as calls of 2^19 steps (interleaved with
    other runs); a run cut into calls at multiples of the launch length
    equals one call bit for bit, energies included."""
    one = g0_table.Run(4, 3, 0.1, [1, 2, 3], 4000.0, H)     # 200000 steps
    one.launch()
    t, E1 = one.energies()
    two = g0_table.Run(4, 3, 0.1, [1, 2, 3], 4000.0, H)
    parts = two.chunks(1 << 16)
    assert len(parts) == 4
    for c in parts:
        c()
    _, E2 = two.energies()
    assert np.array_equal(E1, E2)
    for k in ("X", "P", "R", "C"):
        assert torch.equal(getattr(one, k), getattr(two, k)), k


def test_slopes_reproduce_paper_table_to_1e6():
    """Table tab:g0_slopes, first three decades (t to 1e6, 5e7 steps): the
    seed-1 instance of every row lands within 0.04 (2 x 2) or 0.02 of the
    printed slopes (the paper's MATLAB instance cannot be reproduced, and
    the finite-window slopes move with the instance, most for 2 x 2), and
    the median over 8 instances within the same bounds."""
    res, _ = g0_table.run_table(T=1e6, seeds=range(1, 9))
    for eps, m, n, paper in _paper_rows():
        lows, s = res[(eps, m, n)]
        tol = 0.04 if m * n == 4 else 0.02
        for r in range(len(lows)):
            assert abs(s[r, 0] - paper[r]) < tol, (eps, m, n, lows[r], s[r, 0], paper[r])
            assert abs(np.median(s[r]) - paper[r]) < tol, (eps, m, n, lows[r], np.median(s[r]))


def test_slopes_independent_of_step_size():
    """Numerical-setup appendix: repeating the fits at h = 0.01 instead of
    0.02 moved each slope by less than 8.9e-4 on the paper's instance.  Ours
    (seed 1, decades to 1e5): within 2e-3."""
    for eps, m, n in ((0.0, 4, 3), (0.1, 4, 3), (0.1, 6, 5)):
        sl = []
        for h in (0.02, 0.01):
            run = g0_table.Run(m, n, eps, [1], 1e5, h)
            run.launch()
            t, E = run.energies()
            sl.append(g0_table.decade_slopes(t, E, [1e3, 1e4])[:, 0])
        assert np.all(np.abs(sl[0] - sl[1]) < 2e-3), (eps, m, n, sl)


def test_prefactor_table_matches_oracle_and_paper():
    """Table tab:g0_prefactors on the GPU (m = 3, n = 2, t = 1e4, 17 (alpha,
    mu, eps) settings x 16 instances): the seed-1 values equal the float64
    oracle's to 1e-3, and over the instances the median spread stays under
    the paper's bounds (t E/(alpha mu) moves by less than 30% while alpha mu
    spans 16x; E sqrt(t)/(alpha mu sqrt(eps/2)) by less than 20%)."""
    res = g0_table.prefactor_table(1e4, 3, 2, range(1, 17), H)
    A, X, P = workloads.dense_quadratic_batch(3, 2, [1])
    n = int(round(1e4 / H))
    for name, (cfgs, v) in res.items():
        for (al, mu, ep), q in zip(cfgs, v):
            E, *_ = _oracle(A[0], X[0], P[0], n, [n], HParams(al, mu, 0.0, ep))
            ref = 1e4 * E[0] / (al * mu) if ep == 0.0 else E[0] * 100.0 / (al * mu * np.sqrt(ep / 2))
            assert abs(q[0] / ref - 1) < 1e-3, (name, al, mu, ep, q[0], ref)
        spread = np.median(v.max(axis=0) / v.min(axis=0))
        assert spread < (1.3 if name == "tE_over_alpha_mu" else 1.2), (name, spread)
