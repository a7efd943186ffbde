"""Per-element error bounds for the GPU parity tests (test infrastructure).

The stated parity target is a per-element relative error of 1e-5 after one
step and 1e-4 after 100 steps.  Two float32 sums of the step can cancel:
X_n + h P^(B) and P_n - h g.  Where they do, the result is tiny but any
float32 evaluation carries a rounding of the larger terms, which a pure
relative bound on the tiny result cannot accept.  ``error_bound.c`` carries
a first-order bound on |float32 kernel - float64 oracle| for every element
along the oracle's trajectory (its header derives it).  An element passes if

    |gpu - ref| <= max(rtol |ref|, KAPPA * E)

i.e. within the stated relative tolerance, or, for the elements beyond it,
within KAPPA times the element's own bound (KAPPA covers the second-order
terms the first-order bound drops).  Every comparison records how many
elements needed the bound ("beyond pure") and the largest |gpu - ref| / E
among them; ``summary_lines`` feeds the end-of-session report.
"""
import ctypes
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "error_bound.c")
OUTDIR = os.path.join(HERE, "_build")
KAPPA = 2.0
U = 2.0 ** -24

_lib = None
_lock = threading.Lock()
STATS = []          # (test tag, elements, beyond_pure, worst err/E among them, max rel)


def lib():
    """The compiled helper (built with gcc into tests/_build on first use)."""
    global _lib
    with _lock:
        if _lib is None:
            os.makedirs(OUTDIR, exist_ok=True)
            so = os.path.join(OUTDIR, "liberror_bound_%d.so" % os.getpid())
            r = subprocess.run(["gcc", "-O2", "-std=c99", "-shared", "-fPIC", SRC, "-o", so, "-lm"],
                               capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError("gcc failed on error_bound.c:\n" + r.stderr)
            L = ctypes.CDLL(so)
            os.unlink(so)
            dp = ctypes.POINTER(ctypes.c_double)
            i64, d = ctypes.c_int64, ctypes.c_double
            L.eb_matrix_step.argtypes = [i64, i64, d, d, d, d] + [dp] * 13 + [d, d] + [dp] * 5
            L.eb_matrix_step.restype = ctypes.c_int
            L.eb_vector_step.argtypes = [i64, d, d, d] + [dp] * 10
            L.eb_vector_step.restype = None
            _lib = L
    return _lib


def _p(a):
    if a is None:
        return None
    assert a.dtype == np.float64 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _f64(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float64)


def filter_constants(h, hp):
    """e^{-alpha h} and (1 - e^{-alpha h})/(mu alpha), as the update defines them."""
    d = float(np.exp(-hp.alpha * h))
    k = 0.0 if np.isinf(hp.mu) else float(-np.expm1(-hp.alpha * h) / (hp.mu * hp.alpha))
    return d, k


class TensorBound:
    """The carried bound of one tensor: EX, EP (and Exi for element-wise
    tensors; ER, EC after the last step for matrices)."""

    def __init__(self, shape, depth_row=0.0, depth_col=0.0):
        m, n = shape
        self.matrix = n != 0
        size = m * n if self.matrix else m
        self.shape = (m, n)
        self.EX = np.zeros(size)
        self.EP = np.zeros(size)
        self.EXI = None if self.matrix else np.zeros(size)
        self.ER = np.zeros(m) if self.matrix else None
        self.EC = np.zeros(n) if self.matrix else None
        self.EP1 = np.zeros(size) if self.matrix else None     # the stored form P^(1)
        self.depth_row = float(depth_row)
        self.depth_col = float(depth_col)

    def step(self, h, hp, X0, P0, G, X1, P1, F0, F1, dF0=None, dF1=None):
        """Advance over one step.  X0, P0 (canonical) and the factors F0 =
        (R, C) or (xi, None) are the oracle's before the step, X1, P1, F1
        after it; dF0, dF1 = (|dR|, |dC|) the measured deviations of the
        kernel's factors (matrices only; None = zero)."""
        d, k = filter_constants(h, hp)
        X0, P0, G, X1, P1 = (_f64(a).ravel() for a in (X0, P0, G, X1, P1))
        if not self.matrix:
            lib().eb_vector_step(self.shape[0], h, d, k, _p(X0), _p(P0), _p(_f64(F0[0])), _p(G), _p(X1),
                                 _p(P1), _p(_f64(F1[0])), _p(self.EX), _p(self.EP), _p(self.EXI))
            return
        m, n = self.shape
        dR0, dC0 = (None, None) if dF0 is None else (_f64(dF0[0]), _f64(dF0[1]))
        dR1, dC1 = (None, None) if dF1 is None else (_f64(dF1[0]), _f64(dF1[1]))
        rc = lib().eb_matrix_step(m, n, h, hp.eps_stab, d, k, _p(X0), _p(P0), _p(G), _p(X1), _p(P1),
                                  _p(_f64(F0[0])), _p(_f64(F0[1])), _p(_f64(F1[0])), _p(_f64(F1[1])),
                                  _p(dR0), _p(dC0), _p(dR1), _p(dC1), self.depth_row, self.depth_col,
                                  _p(self.EX), _p(self.EP), _p(self.ER), _p(self.EC), _p(self.EP1))
        if rc != 0:
            raise MemoryError("eb_matrix_step could not allocate")


def check(name, gpu, ref, E, rtol, atol=0.0, tag=None):
    """|gpu - ref| <= max(rtol |ref|, KAPPA E) + atol element by element;
    returns and records (elements, beyond pure, worst err/E beyond pure, max rel)."""
    gpu = np.asarray(gpu, np.float64).ravel()
    ref = np.asarray(ref, np.float64).ravel()
    E = np.zeros_like(ref) if E is None else np.asarray(E, np.float64).ravel()
    assert gpu.shape == ref.shape == E.shape, name
    if ref.size == 0:
        return (0, 0, 0.0, 0.0)
    if not np.all(np.isfinite(gpu)):
        raise AssertionError("%s: non-finite values" % name)
    err = np.abs(gpu - ref)
    pure = rtol * np.abs(ref)
    beyond = err > pure + atol
    with np.errstate(divide="ignore", invalid="ignore"):
        ratio = np.where(beyond, err / (KAPPA * E), 0.0)
    bad = beyond & (err > KAPPA * E + atol)
    with np.errstate(divide="ignore", invalid="ignore"):
        rel = np.where(ref != 0, err / np.abs(ref), np.where(err == 0, 0.0, np.inf))
    nb = int(beyond.sum())
    worst = float(np.max(ratio)) if nb else 0.0
    if np.any(bad):
        i = int(np.argmax(np.where(bad, err - KAPPA * E, -np.inf)))
        raise AssertionError(
            "%s: %d of %d elements beyond max(rtol |ref|, %g E) (rtol %g); worst at %d: gpu %.9g ref "
            "%.9g |err| %.3g rtol|ref| %.3g E %.3g" % (name, int(bad.sum()), ref.size, KAPPA, rtol, i,
                                                      gpu[i], ref[i], err[i], pure[i], E[i]))
    out = (ref.size, nb, worst, float(np.max(rel)))
    if tag is not None:
        STATS.append((tag,) + out)
    return out


def summary_lines():
    """One line per recorded test tag: elements, beyond pure, worst err/(KAPPA E), max rel."""
    agg = {}
    for tag, n, nb, worst, mrel in STATS:
        a = agg.setdefault(tag, [0, 0, 0.0, 0.0])
        a[0] += n
        a[1] += nb
        a[2] = max(a[2], worst)
        a[3] = max(a[3], mrel)
    return ["%s: %d elements, %d beyond the pure relative tolerance, worst |err|/(%g E) %.3g, "
            "max rel %.3g" % (tag, n, nb, KAPPA, worst, mrel) for tag, (n, nb, worst, mrel) in agg.items()]
