"""Oracle for the R-iKFAD optimiser step: plain, slow, float64, on the CPU.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product
library (``paper_2609_30342_gb300``) never imports, links or executes it, and
shares no code with it.

Two independent implementations live here:

* ``rikfad_oracle.c`` (loaded through ctypes): the BACD step of the paper's
  Appendix A table, loop by loop, for matrix parameters (rank-1 friction,
  Eq. xi_def) and for 1-D parameters (element-wise iKFAD, Section 2
  "Memory Complexity"), plus the dense-quadratic test problem of Section 3.2.
* ``explicit.py`` (numpy): the same step written with the m x n friction
  tensor materialised, used as a cross-check on small matrices.

Everything is pinned by ``tests/test_oracle_pins.py`` (see the header of the
C file for the list); nothing is parity-unpinned.
"""
import ctypes

import numpy as np

from . import build as _build

_lib = None


def load(path):
    """Load a compiled oracle library from ``path`` and declare its signatures."""
    L = ctypes.CDLL(path)
    i64 = ctypes.c_int64
    dp = ctypes.POINTER(ctypes.c_double)
    d = ctypes.c_double
    L.orc_step_matrix.argtypes = [i64, i64, dp, dp, dp, dp, dp, d, d, d, d, d, dp, dp, dp]
    L.orc_step_matrix.restype = ctypes.c_int
    L.orc_step_vector.argtypes = [i64, dp, dp, dp, dp, d, d, d, d]
    L.orc_step_vector.restype = ctypes.c_int
    L.orc_dense_quadratic_energy.argtypes = [i64, dp, dp, dp]
    L.orc_dense_quadratic_energy.restype = d
    L.orc_dense_quadratic_run.argtypes = [i64, i64, dp, dp, dp, dp, dp, d, d, d, d, d,
                                          i64, ctypes.POINTER(ctypes.c_int64), i64, dp, dp]
    L.orc_dense_quadratic_run.restype = ctypes.c_int
    return L


def lib():
    """The C oracle (built on first use)."""
    global _lib
    if _lib is None:
        _lib = load(_build.build())
    return _lib


def _f64(a, name):
    if not (isinstance(a, np.ndarray) and a.dtype == np.float64 and a.flags.c_contiguous):
        raise TypeError("%s must be a C-contiguous float64 numpy array" % name)
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


class HParams:
    """Hyperparameters of Eqs. rikfad_x to rikfad_C and Eq. xi_def."""

    def __init__(self, alpha, mu, gamma=0.0, eps_stab=1e-16):
        self.alpha = float(alpha)
        self.mu = float(mu)
        self.gamma = float(gamma)
        self.eps_stab = float(eps_stab)


def step_matrix(X, P, R, C, G, h, hp, P1=None):
    """One BACD step (Appendix A table) for an m x n matrix, in place.  If
    ``P1`` (an m x n float64 array) is given it receives the half-damped
    momentum P^(1) of sub-step C."""
    m, n = X.shape
    if P.shape != (m, n) or G.shape != (m, n) or R.shape != (m,) or C.shape != (n,):
        raise ValueError("shape mismatch")
    if P1 is not None and P1.shape != (m, n):
        raise ValueError("shape mismatch")
    rowsq = np.empty(max(m, 1))
    colsq = np.empty(n)
    rc = lib().orc_step_matrix(m, n, _f64(X, "X"), _f64(P, "P"), _f64(R, "R"), _f64(C, "C"),
                               _f64(G, "G"), float(h), hp.alpha, hp.mu, hp.gamma, hp.eps_stab,
                               _f64(rowsq, "rowsq"), _f64(colsq, "colsq"),
                               None if P1 is None else _f64(P1, "P1"))
    if rc != 0:
        raise ValueError("orc_step_matrix rejected its arguments")


def step_vector(x, p, xi, g, h, hp):
    """One BACD step of element-wise iKFAD (1-D parameters), in place."""
    L = x.size
    if p.size != L or xi.size != L or g.size != L:
        raise ValueError("shape mismatch")
    rc = lib().orc_step_vector(L, _f64(x, "x"), _f64(p, "p"), _f64(xi, "xi"), _f64(g, "g"),
                               float(h), hp.alpha, hp.mu, hp.gamma)
    if rc != 0:
        raise ValueError("orc_step_vector rejected its arguments")


class ModelState:
    """Optimiser state of a whole parameter list, float64.

    ``shapes`` is a list of ``(rows, cols)``; ``cols == 0`` marks a tensor
    that is not a matrix (it follows the element-wise rule with ``rows``
    elements).  Factors and 1-D friction start at zero (Lemma 1's setting,
    R(0) = C(0) = 0); X and P are given by the caller.
    """

    def __init__(self, shapes, X, P):
        self.shapes = [tuple(int(v) for v in s) for s in shapes]
        self.X = [np.ascontiguousarray(x, dtype=np.float64).copy() for x in X]
        self.P = [np.ascontiguousarray(p, dtype=np.float64).copy() for p in P]
        self.R, self.C, self.xi = [], [], []
        for (m, n), x in zip(self.shapes, self.X):
            if n == 0:
                self.R.append(None)
                self.C.append(None)
                self.xi.append(np.zeros(m))
            else:
                self.R.append(np.zeros(m))
                self.C.append(np.zeros(n))
                self.xi.append(None)
        for (m, n), x, p in zip(self.shapes, self.X, self.P):
            want = (m,) if n == 0 else (m, n)
            if x.shape != want or p.shape != want:
                raise ValueError("state shape %s does not match %s" % (x.shape, want))

    def step(self, grads, h, hp):
        """Advance every tensor by one step; ``grads`` are float64 arrays."""
        for t, (m, n) in enumerate(self.shapes):
            g = np.ascontiguousarray(grads[t], dtype=np.float64)
            if n == 0:
                step_vector(self.X[t], self.P[t], self.xi[t], g, h, hp)
            else:
                step_matrix(self.X[t], self.P[t], self.R[t], self.C[t], g, h, hp)


def dense_quadratic_energy(A, X, P):
    """E = 1/2 vec(X)^T A vec(X) + 1/2 ||P||^2 (Section 3 energy, f* = 0)."""
    d = X.size
    return lib().orc_dense_quadratic_energy(d, _f64(A, "A"), _f64(X, "X"), _f64(P, "P"))


def dense_quadratic_run(A, X, P, R, C, h, hp, nsteps, record):
    """BACD on f = 1/2 x^T A x from the given state; returns E at ``record`` steps."""
    m, n = X.shape
    rec = np.ascontiguousarray(np.asarray(record, dtype=np.int64))
    if rec.size and (np.any(np.diff(rec) < 0) or rec[0] < 0 or rec[-1] > nsteps):
        raise ValueError("record steps must be ascending within [0, nsteps]")
    energy = np.empty(rec.size)
    work = np.empty(m * n + m + n)
    rc = lib().orc_dense_quadratic_run(
        m, n, _f64(A, "A"), _f64(X, "X"), _f64(P, "P"), _f64(R, "R"), _f64(C, "C"), float(h),
        hp.alpha, hp.mu, hp.gamma, hp.eps_stab, int(nsteps),
        rec.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), rec.size, _f64(energy, "energy"),
        _f64(work, "work"))
    if rc != 0:
        raise ValueError("orc_dense_quadratic_run rejected its arguments")
    return energy


def diag_quadratic_energy(A, Xstar, X, P):
    """E = 1/2 sum A (.) (X - X*)^2 + 1/2 ||P||^2 for f = 1/2 sum A (.) (X - X*)^2."""
    D = np.asarray(X, np.float64) - np.asarray(Xstar, np.float64)
    return 0.5 * float(np.sum(np.asarray(A, np.float64) * D * D)) + \
        0.5 * float(np.sum(np.asarray(P, np.float64) ** 2))


def state_scalars(shapes):
    """Optimiser auxiliary state in scalars, Section 2 "Memory Complexity":
    momentum for every parameter (N), plus m + n factor entries per matrix,
    plus one friction scalar per element of every non-matrix parameter."""
    total = 0
    for m, n in shapes:
        if n == 0:
            total += 2 * m
        else:
            total += m * n + m + n
    return total
