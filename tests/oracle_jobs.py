"""Oracle runs executed in worker processes (spawned, so they never inherit a
CUDA context) while the GPU side of a test runs."""
import os

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


def _load(d, name):
    return np.load(os.path.join(d, name + ".npy"))


def tensor_trajectory(job):
    """One tensor of a model-sized parity run, in a worker process: the
    oracle's trajectory from the seeded initial state through ``steps``
    steps (the gradients regenerated from the tensor's own streams), the
    per-element bound carried along it (``error_model``), and the comparison
    with the GPU's arrays saved in ``job["dir"]`` at the steps of
    ``compare_at``.  Returns the recorded comparison statistics; raises
    AssertionError on a mismatch."""
    import error_model as em
    shape = tuple(job["shape"])
    t = job["t"]
    d = job["dir"]
    hp = HParams(*job["hp"])
    inp = workloads.ModelInputs(job["shapes"], seed=job["seed"], draw_x=False,
                                g_std=job.get("g_std", 1e-3), grad_bf16=job.get("grad_bf16", True))
    m, n = shape
    X = np.ascontiguousarray(inp.x(t), dtype=np.float64)
    P = np.zeros_like(X)
    bound = em.TensorBound(shape, job.get("depth_row", 0.0), job.get("depth_col", 0.0))
    if n:
        R, C = np.zeros(m), np.zeros(n)
        Rg = _load(d, "%d_R" % t).astype(np.float64)   # (steps, m): the GPU's factors after each step
        Cg = _load(d, "%d_C" % t).astype(np.float64)
    else:
        xi = np.zeros(m)
    dF0 = None
    first = len(em.STATS)
    for k in range(1, job["steps"] + 1):
        h = job["hs"][k - 1]
        g = np.ascontiguousarray(inp.grad(k - 1, t), dtype=np.float64).reshape(X.shape)
        X0, P0 = X.copy(), P.copy()
        if n:
            F0 = (R.copy(), C.copy())
            oracle.step_matrix(X, P, R, C, g, h, hp)
            dF1 = (np.abs(Rg[k - 1] - R), np.abs(Cg[k - 1] - C))
            bound.step(h, hp, X0, P0, g, X, P, F0, (R, C), dF0, dF1)
            dF0 = dF1
        else:
            F0 = (xi.copy(), None)
            oracle.step_vector(X, P, xi, g, h, hp)
            bound.step(h, hp, X0, P0, g, X, P, F0, (xi, None))
        if k in job["compare_at"]:
            rtol = job["rtol"][k]
            tag = "%s step %d (rtol %g)" % (job["tag"], k, rtol)
            name = "%s step%d tensor %d %s" % (job["tag"], k, t, job.get("name", ""))
            Xg = _load(d, "%d_%d_X" % (k, t))
            Pg = _load(d, "%d_%d_P" % (k, t))
            em.check(name + " X", Xg, X, bound.EX, rtol, tag=tag)
            em.check(name + " P", Pg, P, bound.EP, rtol, tag=tag)
            if n:
                em.check(name + " R", Rg[k - 1], R, bound.ER, rtol, tag=tag)
                em.check(name + " C", Cg[k - 1], C, bound.EC, rtol, tag=tag)
            else:
                em.check(name + " xi", _load(d, "%d_%d_xi" % (k, t)), xi, bound.EXI, rtol, tag=tag)
    return em.STATS[first:]
