"""Glue for the GPU tests: run the CUDA path through the C ABI on seeded
inputs and compare with the oracle.

Tolerance (the reading of the stated "per-element relative error <= 1e-5
after 1 step, <= 1e-4 after 100 steps" used throughout):

    |gpu - ref| <= rtol * (|ref| + floor * rms(ref))          per element,

with ``floor = 1e-2``.  Two updates of the step are float32 sums whose terms
can nearly cancel: X_n + h P^(B) (already in the first step, where |X_n| is
tiny) and P_n - h g.  Where they cancel, any float32 implementation carries an
absolute error of about one ulp of the larger term, which a pure relative
bound on the tiny result cannot accept; the floor (1% of the tensor's rms)
is that scale.  Elements beyond the pure relative bound are counted in the
returned statistics.  Long trajectories (thousands of steps) are judged
against the tensor's scale (``floor = 1``) because float32 rounding of the
state accumulates along them.
"""
import numpy as np
import torch

import oracle
from paper_2609_30342_gb300 import rikfad, workloads


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
    return {"max_rel": float(np.max(rel)), "beyond_pure": int(np.sum(rel > rtol))}


class GpuRun:
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
        self.opt.close()


def oracle_from_gpu(run):
    """A fresh oracle state holding the GPU run's current (canonical) state."""
    st = oracle.ModelState(run.shapes, run.X(), run.canonical_P())
    for t, (R, C) in enumerate(run.factors()):
        if C is None:
            st.xi[t] = R.copy()
        else:
            st.R[t] = R.copy()
            st.C[t] = C.copy()
    return st


def compare_state(run, st, rtol, floor, tag="", tensors=None, atol=0.0):
    """Compare GPU X, canonical P and factors with the oracle state."""
    Xg, Pg, F = run.X(), run.canonical_P(), run.factors()
    stats = {}
    idx = range(len(run.shapes)) if tensors is None else tensors
    for t in idx:
        n = run.shapes[t][1]
        stats[("X", t)] = compare("%sX[%d]" % (tag, t), Xg[t], st.X[t], rtol, floor, atol)
        stats[("P", t)] = compare("%sP[%d]" % (tag, t), Pg[t], st.P[t], rtol, floor, atol)
        if n == 0:
            stats[("xi", t)] = compare("%sxi[%d]" % (tag, t), F[t][0], st.xi[t], rtol, floor, atol)
        else:
            stats[("R", t)] = compare("%sR[%d]" % (tag, t), F[t][0], st.R[t], rtol, floor, atol)
            stats[("C", t)] = compare("%sC[%d]" % (tag, t), F[t][1], st.C[t], rtol, floor, atol)
    return stats
