"""Glue for the GPU tests: run the CUDA path through the C ABI on seeded
inputs and compare with the oracle.

Tolerance.  The stated target is a per-element relative error of 1e-5 after
one step and 1e-4 after 100 steps.  The parity tests of the optimiser step
apply it as

    |gpu - ref| <= max(rtol |ref|, 2 E)                        per element,

where E is the element's own first-order bound on the float32 rounding of
the kernels, carried along the oracle's trajectory (``error_model``,
``error_bound.c``).  E matters only where two terms of a float32 sum nearly
cancel (X_n + h P^(B), P_n - h g): there the result is tiny, but its error is
a rounding of the larger terms, which no pure relative bound on the result
can accept.  Every comparison records how many elements needed E.

``compare`` keeps the older form rtol (|ref| + floor rms(ref)) for the
tests whose inputs do not come from a step of the oracle alone: the 2000-step
quadratic trajectories (the gradient is computed from the GPU's own X, so
rounding differences feed back) and the limits of the hyperparameters (where
exp underflows).  It records the count of elements that needed the floor.
"""
import os

import numpy as np
import torch

import error_model as em
import oracle
from paper_2609_30342_gb300 import rikfad, workloads


CHECKED = []        # failed-check counts of the handles closed on the checked build


def _test_tag():
    return os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]


def compare(name, gpu, ref, rtol, floor, atol=0.0):
    """Element-wise |gpu - ref| <= rtol (|ref| + floor rms(ref)) + atol."""
    gpu = np.asarray(gpu, np.float64).ravel()
    ref = np.asarray(ref, np.float64).ravel()
    assert gpu.shape == ref.shape, name
    if ref.size == 0:
        return {"max_rel": 0.0, "beyond_pure": 0}
    assert np.all(np.isfinite(gpu)), "%s: non-finite values" % name
    rms = float(np.sqrt(np.mean(ref * ref)))
    err = np.abs(gpu - ref)
    bound = rtol * (np.abs(ref) + floor * rms) + atol
    bad = err > bound
    with np.errstate(divide="ignore", invalid="ignore"):
        rel = np.where(ref != 0, err / np.abs(ref), np.where(err == 0, 0.0, np.inf))
    if np.any(bad):
        i = int(np.argmax(err - bound))
        raise AssertionError("%s: %d of %d elements beyond tolerance (rtol %g, floor %g); worst at "
                             "%d: gpu %.9g ref %.9g |err| %.3g bound %.3g; max rel %.3g"
                             % (name, int(bad.sum()), ref.size, rtol, floor, i, gpu[i], ref[i],
                                err[i], bound[i], float(np.max(rel))))
    beyond = rel > rtol
    worst = float(np.max(np.where(beyond, err / np.maximum(bound, 1e-300), 0.0))) if beyond.any() else 0.0
    em.STATS.append(("%s (rtol %g, floor %g rms)" % (_test_tag(), rtol, floor), ref.size,
                     int(beyond.sum()), worst, float(np.max(rel))))
    return {"max_rel": float(np.max(rel)), "beyond_pure": int(beyond.sum())}


class DeviceRun:
    """R-iKFAD on the GPU through the C ABI, with host-side inputs."""

    def __init__(self, shapes, hp, grad_bf16, X, P, device="cuda", method="rikfad"):
        self.shapes = [tuple(s) for s in shapes]
        self.grad_bf16 = grad_bf16
        self.opt = rikfad.RIKFAD(self.shapes, hp.alpha, hp.mu, hp.gamma, hp.eps_stab,
                                 "bf16" if grad_bf16 else "f32", method=method)
        gdt = torch.bfloat16 if grad_bf16 else torch.float32
        self.x = [torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device) for a in X]
        self.p = [torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device) for a in P]
        self.g = [torch.zeros(workloads.array_shape(s), dtype=gdt, device=device) for s in self.shapes]
        self.out = [torch.empty_like(a) for a in self.p]
        self.ptrs = self.opt.pack(self.x, self.g, self.p)
        self.gdt = gdt

    def set_grads(self, grads):
        for dst, src in zip(self.g, grads):
            t = torch.from_numpy(np.ascontiguousarray(src, np.float32))
            dst.copy_(t.to(self.gdt).to(dst.device))

    def step(self, h):
        self.opt.step(h, ptrs=self.ptrs)

    def canonical_P(self):
        self.opt.canonical_momentum(self.p, self.out)
        torch.cuda.synchronize()
        return [o.double().cpu().numpy() for o in self.out]

    def X(self):
        torch.cuda.synchronize()
        return [x.double().cpu().numpy() for x in self.x]

    def factors(self):
        out = []
        for t in range(len(self.shapes)):
            R, C = self.opt.get_factors(t)
            out.append((R.astype(np.float64), None if C is None else C.astype(np.float64)))
        return out

    def close(self):
        if os.environ.get("RIKFAD_EXPECT_CHECKED"):
            # Run on the checked build: no device-side check may have failed.
            n, code = self.opt.debug_check_failures()
            assert n == 0, "device-side plan checks failed: %d (first code %d)" % (n, code)
            CHECKED.append(n)
        self.opt.close()


# ------------------------------------------------ per-element error model

def summation_depths(shapes, nblocks):
    """Longest chain of float32 additions in the kernels' row and column sums
    of every matrix, from the host planner's pieces (the same planner the
    library runs): {t: (depth_row, depth_col)}.  A lane adds its own
    columns of a panel row (8 per 256/RPW-column chunk, or every 32nd column
    on the scalar path), a 32-lane butterfly follows, and the finalise kernel
    adds the panels; a column sum runs over a warp's rows of a piece, the 8
    warps (times RPW lane groups) and the panel's slots."""
    plan = rikfad.plan_query(shapes, "bf16", nblocks)
    out = {}
    for t, (m, n) in enumerate(shapes):
        if n == 0:
            continue
        rows = plan[(plan[:, 1] == t) & (plan[:, 2] == 0)]
        if rows.size == 0:
            out[t] = (8.0, 8.0)
            continue
        npanels = len(np.unique(rows[:, 3]))
        drow = dcol = 0
        for col0 in np.unique(rows[:, 3]):
            pr = rows[rows[:, 3] == col0]
            w = int(pr[0, 4])
            if n % 8 == 0:
                rpw = 1 if (w % 256 == 0 or w > 512) else (4 if w <= 64 else 2)
                lane = 8 * -(-w * rpw // 256)
            else:
                rpw, lane = 1, -(-w // 32)
            drow = max(drow, lane + 5)
            piece_rows = int(np.max(pr[:, 6] - pr[:, 5]))
            dcol = max(dcol, -(-piece_rows // (8 * rpw)) + 8 * rpw + len(pr) + 2)
        out[t] = (float(drow + npanels + 2), float(dcol))
    return out


def _nblocks():
    return 2 * torch.cuda.get_device_properties(0).multi_processor_count


def model_parity(tag, named, seed, hp, h, steps, compare_at, rtol, tensors=None, workers=None, hs=None):
    """A parity run at model size, in the launch configuration the benchmark
    times: the whole list steps on the GPU (gradients ~ N(0, 1e-3^2), bf16,
    from the tensors' own streams); the tensors in ``tensors`` (default all)
    get fresh gradients every step and are compared with the oracle at the
    steps of ``compare_at`` (rtol[k] at step k, per-element bound beyond it);
    the others keep their first gradients.  The oracle runs per tensor in
    spawned worker processes after the GPU run (``oracle_jobs.tensor_trajectory``),
    from the GPU's saved arrays and per-step factors.  ``hs`` (default: h at
    every step) gives the step size of each step."""
    import multiprocessing as mp
    import os
    import shutil
    import tempfile
    from concurrent.futures import ThreadPoolExecutor

    import error_model as em
    import oracle_jobs

    shapes = [s for _, s in named]
    names = [nm for nm, _ in named]
    T = len(shapes)
    tensors = list(range(T)) if tensors is None else list(tensors)
    hs = [h] * steps if hs is None else list(hs)
    assert len(hs) == steps
    inp = workloads.ModelInputs(shapes, seed=seed, draw_x=False)
    pool_t = ThreadPoolExecutor(8)
    X0 = list(pool_t.map(inp.x, range(T)))
    P0 = [np.zeros(workloads.array_shape(s), np.float32) for s in shapes]
    run = DeviceRun(shapes, hp, True, X0, P0)
    del X0, P0
    d = tempfile.mkdtemp(prefix="rikfad_parity_")
    depths = summation_depths(shapes, _nblocks())
    try:
        fac = {t: ([], []) for t in tensors if shapes[t][1] != 0}
        for k in range(1, steps + 1):
            sel = range(T) if k == 1 else tensors
            gs = list(pool_t.map(lambda t: (t, inp.grad(k - 1, t)), sel))
            for t, g in gs:
                run.g[t].copy_(torch.from_numpy(g).to(run.gdt).to(run.g[t].device))
            del gs
            run.step(hs[k - 1])
            torch.cuda.synchronize()
            for t in fac:
                R, C = run.opt.get_factors(t)
                fac[t][0].append(R)
                fac[t][1].append(C)
            if k in compare_at:
                out = [torch.empty_like(p) for p in run.p]
                run.opt.canonical_momentum(run.p, out)
                torch.cuda.synchronize()
                for t in tensors:
                    np.save(os.path.join(d, "%d_%d_X.npy" % (k, t)), run.x[t].cpu().numpy())
                    np.save(os.path.join(d, "%d_%d_P.npy" % (k, t)), out[t].cpu().numpy())
                    if shapes[t][1] == 0:
                        np.save(os.path.join(d, "%d_%d_xi.npy" % (k, t)), run.opt.get_factors(t)[0])
                del out
        for t, (Rs, Cs) in fac.items():
            np.save(os.path.join(d, "%d_R.npy" % t), np.stack(Rs))
            np.save(os.path.join(d, "%d_C.npy" % t), np.stack(Cs))
        del fac
        run.close()
        pool_t.shutdown()
        jobs = []
        for t in sorted(tensors, key=lambda t: -workloads.numel(shapes[t])):
            dr, dc = depths.get(t, (0.0, 0.0))
            jobs.append(dict(shapes=shapes, shape=shapes[t], t=t, name=names[t], seed=seed,
                             hp=(hp.alpha, hp.mu, hp.gamma, hp.eps_stab), hs=hs, steps=steps,
                             compare_at=sorted(compare_at), rtol=rtol, dir=d, tag=tag,
                             depth_row=dr, depth_col=dc))
        nw = workers or max(1, min(len(jobs), (os.cpu_count() or 2) - 1, 16))
        ctx = mp.get_context("spawn")
        with ctx.Pool(nw) as pool:
            for stats in pool.imap_unordered(oracle_jobs.tensor_trajectory, jobs):
                em.STATS.extend(stats)
    finally:
        shutil.rmtree(d, ignore_errors=True)


class Tracked:
    """The oracle's state of a tensor list with the carried per-element
    bounds, stepped in this process alongside a DeviceRun (small cases).  The
    GPU's factors after every step give the deviations the bound takes for
    the exponents of the next step (the factors themselves are compared too)."""

    def __init__(self, shapes, X, P, factors=None, depths=None):
        self.shapes = [tuple(s) for s in shapes]
        self.st = oracle.ModelState(self.shapes, X, P)
        if factors is not None:
            for t, (R, C) in enumerate(factors):
                if self.shapes[t][1] == 0:
                    self.st.xi[t] = np.asarray(R, np.float64).copy()
                else:
                    self.st.R[t] = np.asarray(R, np.float64).copy()
                    self.st.C[t] = np.asarray(C, np.float64).copy()
        depths = depths or {}
        self.bounds = [em.TensorBound(s, *depths.get(t, (64.0, 64.0))) for t, s in enumerate(self.shapes)]
        self.dF = [None] * len(self.shapes)

    @classmethod
    def from_gpu(cls, run, depths=None):
        """A fresh track from the GPU run's current state (bounds zero)."""
        return cls(run.shapes, run.X(), run.canonical_P(), run.factors(), depths)

    def step(self, grads, h, hp, gpu_factors):
        st = self.st
        for t, (m, n) in enumerate(self.shapes):
            g = np.ascontiguousarray(grads[t], dtype=np.float64)
            X0, P0 = st.X[t].copy(), st.P[t].copy()
            if n == 0:
                F0 = (st.xi[t].copy(), None)
                oracle.step_vector(st.X[t], st.P[t], st.xi[t], g, h, hp)
                self.bounds[t].step(h, hp, X0, P0, g, st.X[t], st.P[t], F0, (st.xi[t], None))
            else:
                F0 = (st.R[t].copy(), st.C[t].copy())
                oracle.step_matrix(st.X[t], st.P[t], st.R[t], st.C[t], g, h, hp)
                Rg, Cg = gpu_factors[t]
                dF1 = (np.abs(Rg - st.R[t]), np.abs(Cg - st.C[t]))
                self.bounds[t].step(h, hp, X0, P0, g, st.X[t], st.P[t], F0, (st.R[t], st.C[t]),
                                    self.dF[t], dF1)
                self.dF[t] = dF1

    def check(self, run, rtol, label, gpu=None, atol=0.0):
        """Compare the GPU state (X, canonical P, factors) with the tracked
        oracle state within max(rtol |ref|, 2 E)."""
        Xg, Pg, F = gpu if gpu is not None else (run.X(), run.canonical_P(), run.factors())
        tag = "%s (rtol %g)" % (_test_tag(), rtol)
        for t, (m, n) in enumerate(self.shapes):
            b = self.bounds[t]
            nm = "%s tensor %d %s" % (label, t, self.shapes[t])
            em.check(nm + " X", Xg[t], self.st.X[t], b.EX, rtol, atol, tag)
            em.check(nm + " P", Pg[t], self.st.P[t], b.EP, rtol, atol, tag)
            if n == 0:
                em.check(nm + " xi", F[t][0], self.st.xi[t], b.EXI, rtol, atol, tag)
            else:
                em.check(nm + " R", F[t][0], self.st.R[t], b.ER, rtol, atol, tag)
                em.check(nm + " C", F[t][1], self.st.C[t], b.EC, rtol, atol, tag)
