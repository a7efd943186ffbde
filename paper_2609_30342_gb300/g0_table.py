"""Energy-decay slopes of R-iKFAD with gamma = 0 on small dense quadratics,
integrated on the GPU (the experiment behind Table tab:g0_slopes of Section
3.2: BACD splitting at h = 0.02, alpha = mu = 1, to t = 1e7, local slopes of
log E against log t by least squares on successive decades).

Every (m, n, eps_stab) row integrates a batch of seeded instances with
``rikfad_quadratic_run`` on its own CUDA stream; the rows are issued as
interleaved chunks of 2^19 steps, so they run on the GPU at the same time.
Slopes are fitted to energies recorded at points spread evenly in log t.

    python -m paper_2609_30342_gb300.g0_table --T 1e7 --seeds 16
    python -m paper_2609_30342_gb300.g0_table --prefactors --seeds 16

The second form measures the parameter dependence of the energy prefactors
(Table tab:g0_prefactors, m = 3, n = 2, t = 1e4).
"""
import argparse
import json
import time

import numpy as np

from . import rikfad, workloads

ROWS = ((0.0, 2, 2), (0.0, 4, 3), (0.0, 6, 5), (0.1, 2, 2), (0.1, 4, 3), (0.1, 6, 5))


def decades(T, first=1e3):
    """Lower ends of the decades [lo, 10 lo] inside [first, T]."""
    out, lo = [], first
    while lo * 10 <= T * (1 + 1e-12):
        out.append(lo)
        lo *= 10
    return out


def decade_slopes(t, E, lows):
    """Least-squares slope of log E against log t on each [lo, 10 lo].
    ``E`` is (len(t), batch); returns (len(lows), batch)."""
    out = np.empty((len(lows), E.shape[1]))
    for r, lo in enumerate(lows):
        sel = (t >= lo * (1 - 1e-9)) & (t <= 10 * lo * (1 + 1e-9))
        u = np.log(t[sel])
        u = u - u.mean()
        v = np.log(E[sel].astype(np.float64))
        out[r] = (u @ (v - v.mean(axis=0))) / (u @ u)
    return out


class Run:
    """One batched integration enqueued on its own stream."""

    def __init__(self, m, n, eps, seeds, T, h=0.02, alpha=1.0, mu=1.0, gamma=0.0, per_decade=60):
        import torch
        self.m, self.n, self.eps, self.h = m, n, eps, h
        self.seeds = list(seeds)
        A, X, P = workloads.dense_quadratic_batch(m, n, self.seeds)
        dev = torch.device("cuda")
        b = len(self.seeds)
        self.A = torch.from_numpy(A).to(dev)
        self.X = torch.from_numpy(X).to(dev)
        self.P = torch.from_numpy(P).to(dev)
        self.R = torch.zeros(b, m, device=dev)
        self.C = torch.zeros(b, n, device=dev)
        self.k = workloads.log_records(T, h, per_decade)
        self.rec = torch.from_numpy(self.k).to(dev)
        self.E = torch.full((len(self.k), b), float("nan"), device=dev)
        self.nsteps = int(round(T / h))
        self.stream = torch.cuda.Stream()
        self.stream.wait_stream(torch.cuda.current_stream())
        self.args = (alpha, mu, gamma, eps)

    def launch(self):
        """The whole run as one call."""
        alpha, mu, gamma, eps = self.args
        rikfad.quadratic_run(self.A, self.X, self.P, self.R, self.C, self.h, alpha, mu, gamma, eps,
                             self.nsteps, self.rec, self.E, stream=self.stream)

    def chunks(self, chunk_steps=1 << 19):
        """The run as consecutive calls of ``chunk_steps`` steps (a multiple of
        the library's launch length, so the result is bit-identical to one
        call), each with its own slice of the record list; returns one
        callable per chunk.  Interleaving the chunks of several runs keeps
        the GPU's launch queue shared between their streams, so the runs
        proceed at the same time."""
        import torch
        alpha, mu, gamma, eps = self.args
        out = []
        k0 = 0
        while True:
            k1 = min(k0 + chunk_steps, self.nsteps)
            last = k1 == self.nsteps
            sel = np.nonzero((self.k >= k0) & ((self.k <= k1) if last else (self.k < k1)))[0]
            if sel.size:
                r0, r1 = int(sel[0]), int(sel[-1]) + 1
                rec = torch.from_numpy(self.k[r0:r1] - k0).to(self.rec.device)
                energy = self.E[r0:r1]
            else:
                rec, energy = None, None

            def call(k0=k0, k1=k1, rec=rec, energy=energy):
                rikfad.quadratic_run(self.A, self.X, self.P, self.R, self.C, self.h, alpha, mu, gamma,
                                     eps, k1 - k0, rec, energy, stream=self.stream)
            out.append(call)
            if last:
                return out
            k0 = k1

    def energies(self):
        self.stream.synchronize()
        return self.k * self.h, self.E.cpu().numpy()


def run_table(T=1e7, seeds=range(1, 17), h=0.02, rows=ROWS, per_decade=60):
    """Slopes for every row of ``rows``: {(eps, m, n): (lows, slopes (decades x seeds))}."""
    import torch
    runs = [Run(m, n, eps, seeds, T, h, per_decade=per_decade) for eps, m, n in rows]
    parts = [r.chunks() for r in runs]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for c in range(max(len(p) for p in parts)):
        for p in parts:
            if c < len(p):
                p[c]()
    out = {}
    for (eps, m, n), r in zip(rows, runs):
        t, E = r.energies()
        lows = decades(T)
        out[(eps, m, n)] = (lows, decade_slopes(t, E, lows))
    return out, time.perf_counter() - t0


PREFACTOR_GRID = {
    # quantity: (eps values, alpha and mu values), Table tab:g0_prefactors
    "tE_over_alpha_mu": ((0.0,), (0.5, 1.0, 2.0)),
    "E_sqrt_t_over_alpha_mu_sqrt_half_eps": ((0.05, 0.2), (0.5, 1.0)),
}


def prefactor_table(T=1e4, m=3, n=2, seeds=range(1, 17), h=0.02):
    """The parameter dependence of the energy prefactors (Table
    tab:g0_prefactors): t E/(alpha mu) with eps_stab = 0 over alpha, mu in
    {1/2, 1, 2}, and E sqrt(t)/(alpha mu sqrt(eps/2)) over alpha, mu in
    {1/2, 1}, eps in {0.05, 0.2}, at t = T.  Every (alpha, mu, eps) is one
    batched run over the seeds, all on their own streams at once.  Returns
    {quantity: (configs, values (configs x seeds))}."""
    import torch
    jobs = []
    for name, (epss, ams) in PREFACTOR_GRID.items():
        for al in ams:
            for mu in ams:
                for ep in epss:
                    jobs.append((name, al, mu, ep, Run(m, n, ep, seeds, T, h, alpha=al, mu=mu, per_decade=2)))
    parts = [j[-1].chunks() for j in jobs]
    torch.cuda.synchronize()
    for c in range(max(len(p) for p in parts)):
        for p in parts:
            if c < len(p):
                p[c]()
    out = {}
    for name, al, mu, ep, run in jobs:
        _, E = run.energies()
        e = E[-1].astype(np.float64)            # the last record is t = T
        q = T * e / (al * mu) if ep == 0.0 else e * np.sqrt(T) / (al * mu * np.sqrt(ep / 2))
        cfgs, vals = out.setdefault(name, ([], []))
        cfgs.append((al, mu, ep))
        vals.append(q)
    return {k: (c, np.array(v)) for k, (c, v) in out.items()}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--T", type=float, default=1e7)
    ap.add_argument("--h", type=float, default=0.02)
    ap.add_argument("--seeds", type=int, default=16, help="instances per row (seeds 1..N)")
    ap.add_argument("--json", action="store_true")
    ap.add_argument("--prefactors", action="store_true",
                    help="the prefactor table instead (m = 3, n = 2, t = 1e4 unless --T is given)")
    a = ap.parse_args()
    if a.prefactors:
        T = a.T if a.T != 1e7 else 1e4
        res = prefactor_table(T, 3, 2, range(1, a.seeds + 1), a.h)
        out = {}
        for name, (cfgs, v) in res.items():
            mean = v.mean(axis=0)                       # per seed, over the parameter grid
            spread = v.max(axis=0) / v.min(axis=0)
            out[name] = {"configs": cfgs, "seed1_mean": round(float(mean[0]), 4),
                         "seed1_spread": round(float(spread[0]), 4),
                         "median_mean": round(float(np.median(mean)), 4),
                         "median_spread": round(float(np.median(spread)), 4),
                         "spread_range": [round(float(spread.min()), 4), round(float(spread.max()), 4)]}
        print(json.dumps({"T": T, "h": a.h, "m": 3, "n": 2, "seeds": a.seeds, "prefactors": out}))
        return
    res, secs = run_table(a.T, range(1, a.seeds + 1), a.h)
    if a.json:
        print(json.dumps({"T": a.T, "h": a.h, "seconds": secs,
                          "rows": [{"eps_stab": e, "m": m, "n": n, "decades": lows,
                                    "seed1": s[:, 0].round(4).tolist(),
                                    "median": np.median(s, axis=1).round(4).tolist(),
                                    "min": s.min(axis=1).round(4).tolist(),
                                    "max": s.max(axis=1).round(4).tolist()}
                                   for (e, m, n), (lows, s) in res.items()]}))
        return
    print("T = %g, h = %g, %d seeds, %.1f s" % (a.T, a.h, a.seeds, secs))
    for (e, m, n), (lows, s) in res.items():
        head = "eps=%-4g %dx%d" % (e, m, n)
        cells = ["[%g,%g] seed1 %+.3f median %+.3f (%+.3f..%+.3f)"
                 % (lo, 10 * lo, s[r, 0], np.median(s[r]), s[r].min(), s[r].max())
                 for r, lo in enumerate(lows)]
        print(head + "\n  " + "\n  ".join(cells))


if __name__ == "__main__":
    main()
