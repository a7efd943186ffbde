"""The per-element rounding bound of the parity tests (tests/error_bound.c),
checked on the CPU: a float32 evaluation of one step in the kernels' order of
operations (every operation rounded to float32; the two fused multiply-adds
rounded once) must stay within the bound the model carries along the oracle's
float64 trajectory, over 100 steps, on shapes with cancelling sums.  A bound
that misses a rounding (a dropped term, a wrong factor) fails here.

The float32 evaluation below is test scaffolding for the bound only: it is not
the oracle (which stays float64 and in the paper's order) and not the CUDA path.
"""
import numpy as np
import pytest

import error_model as em
import oracle
from oracle import HParams
from paper_2609_30342_gb300 import workloads

F = np.float32
LOG2E = 1.4426950408889634


def _fma(a, b, c):
    """a * b + c rounded once to float32 (exact in float64 for float32 inputs)."""
    return (a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64)).astype(F)


def _exp_factor(scale, R, C, eps):
    """exp2(scale * (R_i / (sum R + eps)) * C_j) with float32 roundings at each operation."""
    s = np.sum(R, dtype=F)
    den = F(s + F(eps))
    inv = F(0) if den == 0 else F(F(1) / den)
    a = (F(scale) * (R * inv).astype(F)).astype(F)
    return np.exp2((a[:, None] * C[None, :]).astype(F)).astype(F)


def _step32(X, Phat, R, C, G, h, h_prev, hp):
    """One step in the kernels' stored form (Phat = P^(1) of the last step)."""
    e_prev = _exp_factor(-0.5 * h_prev * LOG2E, R, C, hp.eps_stab)
    e_cur = _exp_factor(-0.5 * h * LOG2E, R, C, hp.eps_stab)
    p_n = ((Phat * e_prev).astype(F) * F(np.exp(-hp.gamma * h_prev))).astype(F)
    p_b = _fma(np.full_like(G, -F(h)), G, p_n)
    X = _fma(np.full_like(G, F(h)), p_b, X)
    p1 = (p_b * e_cur).astype(F)
    q = (p1 * p1).astype(F)
    d = F(np.exp(-hp.alpha * h))
    k = F(-np.expm1(-hp.alpha * h) / (hp.mu * hp.alpha))
    R = _fma(np.full_like(R, k), np.sum(q, axis=1, dtype=F), (d * R).astype(F))
    C = _fma(np.full_like(C, k), np.sum(q, axis=0, dtype=F), (d * C).astype(F))
    return X, p1, R, C


def _canonical32(Phat, R, C, h, hp):
    e = _exp_factor(-0.5 * h * LOG2E, R, C, hp.eps_stab)
    return ((Phat * e).astype(F) * F(np.exp(-hp.gamma * h))).astype(F)


@pytest.mark.parametrize("shape,gamma", [((96, 64), 0.0), ((33, 40), 0.1), ((257, 1), 0.0),
                                         ((1, 24), 0.05)])
def test_float32_evaluation_stays_within_the_bound(shape, gamma):
    m, n = shape
    rng = np.random.default_rng(m * 7 + n)
    hp = HParams(0.0579, 1.3637e-6, gamma, 1e-16)
    h = 0.0918
    X0 = (0.02 * rng.standard_normal(shape)).astype(F)
    Xe, Pe, Re, Ce = X0.copy(), np.zeros(shape, F), np.zeros(m, F), np.zeros(n, F)
    Xo, Po, Ro, Co = X0.astype(np.float64), np.zeros(shape), np.zeros(m), np.zeros(n)
    bound = em.TensorBound(shape, n / 8 + 40, m + 40)
    dF0, h_prev, worst, needed = None, 0.0, 0.0, 0
    for k in range(100):
        # gradients of the same size as h g P-cancellation needs: bf16 values
        g = workloads.bf16_round((1e-3 * rng.standard_normal(shape)).astype(F))
        Xe, Pe, Re, Ce = _step32(Xe, Pe, Re, Ce, g, h, h_prev, hp)
        h_prev = h
        X_, P_, F0 = Xo.copy(), Po.copy(), (Ro.copy(), Co.copy())
        oracle.step_matrix(Xo, Po, Ro, Co, g.astype(np.float64), h, hp)
        dF1 = (np.abs(Re - Ro), np.abs(Ce - Co))
        bound.step(h, hp, X_, P_, g, Xo, Po, F0, (Ro, Co), dF0, dF1)
        dF0 = dF1
        if k in (0, 1, 9, 99):
            Pc = _canonical32(Pe, Re, Ce, h, hp)
            for name, gv, ref, E in (("X", Xe, Xo, bound.EX), ("P", Pc, Po, bound.EP),
                                     ("R", Re, Ro, bound.ER), ("C", Ce, Co, bound.EC)):
                err = np.abs(gv.astype(np.float64) - ref).ravel()
                E = E.ravel()
                assert np.all(err <= em.KAPPA * E + 1e-300), (name, k, float(np.max(err / E)))
                worst = max(worst, float(np.max(err / (em.KAPPA * E + 1e-300))))
                needed += int(np.sum(err > 1e-5 * np.abs(ref).ravel()))
    # The bound is not vacuous: the evaluation uses a sizeable part of it,
    # and some elements do need it (their relative error exceeds 1e-5).
    assert worst > 0.05
    assert needed > 0 or m * n < 100


@pytest.mark.parametrize("shape", [(64, 48), (300, 1), (1, 200)])
def test_first_step_bound_is_tight_where_sums_cancel(shape):
    """One step from a momentum of the same size as h g, so that P_n - h g
    (and with it X_n + h P^(B)) cancels for many elements: the float32
    evaluation must stay within the bound, and must use more than a tenth of
    it on the cancelling elements (a bound that dropped the cancellation
    terms would fail the first check; a vacuous one the second)."""
    m, n = shape
    rng = np.random.default_rng(m + 3 * n)
    hp = HParams(0.0579, 1.3637e-6, 0.0, 1e-16)
    h = 0.0918
    g = workloads.bf16_round((1e-3 * rng.standard_normal(shape)).astype(F))
    P0 = (h * g.astype(np.float64) * (1.0 + 1e-3 * rng.standard_normal(shape))).astype(F)
    PB = P0.astype(np.float64) - h * g.astype(np.float64)
    X0 = (-h * PB * (1.0 + 1e-3 * rng.standard_normal(shape))).astype(F)
    Xe, Pe, Re, Ce = _step32(X0.copy(), P0.copy(), np.zeros(m, F), np.zeros(n, F), g, h, 0.0, hp)
    Xo, Po, Ro, Co = X0.astype(np.float64), P0.astype(np.float64), np.zeros(m), np.zeros(n)
    oracle.step_matrix(Xo, Po, Ro, Co, g.astype(np.float64), h, hp)
    bound = em.TensorBound(shape, n / 8 + 40, m + 40)
    bound.step(h, hp, X0, P0, g, Xo, Po, (np.zeros(m), np.zeros(n)), (Ro, Co), None,
               (np.abs(Re - Ro), np.abs(Ce - Co)))
    Pc = _canonical32(Pe, Re, Ce, h, hp)
    for name, gv, ref, E in (("X", Xe, Xo, bound.EX), ("P", Pc, Po, bound.EP)):
        err = np.abs(gv.astype(np.float64) - ref).ravel()
        E = E.ravel()
        cancel = err > 1e-5 * np.abs(ref).ravel()          # beyond the pure relative bound
        assert cancel.sum() > 0, name
        assert np.all(err <= em.KAPPA * E), (name, float(np.max(err / E)))
        assert float(np.max(err[cancel] / (em.KAPPA * E[cancel]))) > 0.1, name


def test_bound_is_zero_for_exact_steps():
    """With X = P = g = 0 every operation is exact, and so is the bound's start."""
    hp = HParams(0.3, 1.0, 0.0, 1e-8)
    b = em.TensorBound((4, 3), 8, 8)
    z = np.zeros((4, 3))
    b.step(0.1, hp, z, z, z, z, z, (np.zeros(4), np.zeros(3)), (np.zeros(4), np.zeros(3)))
    assert not b.EX.any() and not b.EP.any() and not b.ER.any() and not b.EC.any()
