"""The allocation-free single-matrix step against the handle API and the
oracle (GPU).

rikfad_step_matrix_noalloc exists for callers that cannot allocate device
memory themselves: programs whose framework allocator already owns the GPU's
memory, and services that forbid cudaMalloc after start-up because it can
stall the device.  It keeps its partial sums in an array compiled into the
library, so it must give the same results as the ordinary handle-based step
(which allocates its workspace in rikfad_create), call after call, and the
oracle's.

This file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

import error_model as em
import oracle
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad

from gpu_helpers import compare

pytestmark = pytest.mark.gpu

HP = dict(alpha=0.5, mu=1e-6, gamma=0.1, eps_stab=1e-8)
# The third call repeats the second's step size, so the pending factor and
# the first half-damp share one exponential (the reuse instantiation).
STEPS = (0.05, 0.03, 0.03)

# (rows, cols, grad dtype, also against the oracle): 8-wide and scalar rows
# with both gradient types, and the largest size the compiled-in array allows.
CASES = [(3000, 768, "bf16", True), (257, 129, "f32", True), (512, 256, "f32", True),
         (300, 100, "bf16", True), (65536, 1024, "bf16", False)]


def _inputs(rows, cols, grad):
    dev = torch.device("cuda")
    gdt = torch.bfloat16 if grad == "bf16" else torch.float32
    gen = torch.Generator(device="cpu").manual_seed(rows + cols)
    X0 = 0.02 * torch.randn(rows, cols, generator=gen)
    P0 = 0.01 * torch.randn(rows, cols, generator=gen)
    G = [(1e-3 * torch.randn(rows, cols, generator=gen)).to(gdt) for _ in STEPS]
    return dev, X0, P0, G


@pytest.mark.parametrize("rows,cols,grad,with_oracle", CASES,
                         ids=["%dx%d-%s" % c[:3] for c in CASES])
def test_noalloc_step_matches_handle_step_and_oracle(rows, cols, grad, with_oracle):
    """Three calls in a row (the second with a new step size, so the pending
    factor of the first is applied; the third with the same one): X, the
    stored momentum and both factors agree with rikfad_step within 1e-5, and
    with the oracle (X, the half-damped momentum P^(1) the call stores, R and
    C) within the parity tolerance of the tests: 1e-5 after the first call,
    1e-4 after the others, per-element rounding bound beyond it."""
    pkg_build.build()
    dev, X0, P0, G = _inputs(rows, cols, grad)
    Gd = [g.to(dev) for g in G]

    # the handle API (allocates its workspace in rikfad_create)
    opt = rikfad.RIKFAD([(rows, cols)], grad_dtype=grad, **HP)
    xa, pa = X0.to(dev), P0.to(dev)
    # the allocation-free entry point: caller-owned state, zero factors
    xb, pb = X0.to(dev), P0.to(dev)
    R = torch.zeros(rows, dtype=torch.float32, device=dev)
    C = torch.zeros(cols, dtype=torch.float32, device=dev)
    # the oracle and the per-element bound
    hp = oracle.HParams(**HP)
    Xo, Po = X0.double().numpy().copy(), P0.double().numpy().copy()
    Ro, Co = np.zeros(rows), np.zeros(cols)
    P1o = np.empty((rows, cols))
    bound = em.TensorBound((rows, cols), cols / 16 + 40, rows / 8 + 400)
    dF0 = None

    pending = 0.0
    for k, h in enumerate(STEPS):
        opt.step(h, [xa], [Gd[k]], [pa])
        rikfad.step_matrix_noalloc(rows, cols, h, pending, HP["alpha"], HP["mu"], HP["gamma"],
                                   HP["eps_stab"], grad, xb, Gd[k], pb, R, C)
        pending = h
        torch.cuda.synchronize()
        Ra, Ca = opt.get_factors(0)
        tag = "%dx%d call %d " % (rows, cols, k + 1)
        Xg, Pg = xb.double().cpu().numpy(), pb.double().cpu().numpy()
        Rg, Cg = R.double().cpu().numpy(), C.double().cpu().numpy()
        compare(tag + "X", Xg, xa.double().cpu().numpy(), 1e-5, 1e-2)
        compare(tag + "P", Pg, pa.double().cpu().numpy(), 1e-5, 1e-2)
        compare(tag + "R", Rg, Ra.astype(np.float64), 1e-5, 1e-2)
        compare(tag + "C", Cg, Ca.astype(np.float64), 1e-5, 1e-2)
        if with_oracle:
            g64 = G[k].double().numpy()
            X_, P_, F0 = Xo.copy(), Po.copy(), (Ro.copy(), Co.copy())
            oracle.step_matrix(Xo, Po, Ro, Co, g64, h, hp, P1=P1o)
            dF1 = (np.abs(Rg - Ro), np.abs(Cg - Co))
            bound.step(h, hp, X_, P_, g64, Xo, Po, F0, (Ro, Co), dF0, dF1)
            dF0 = dF1
            rtol = 1e-5 if k == 0 else 1e-4
            utag = "no-alloc step vs oracle (rtol %g)" % rtol
            em.check(tag + "X vs oracle", Xg, Xo, bound.EX, rtol, tag=utag)
            em.check(tag + "P^(1) vs oracle", Pg, P1o, bound.EP1, rtol, tag=utag)
            em.check(tag + "R vs oracle", Rg, Ro, bound.ER, rtol, tag=utag)
            em.check(tag + "C vs oracle", Cg, Co, bound.EC, rtol, tag=utag)
    assert float(R.sum()) > 0 and float(C.sum()) > 0
    opt.close()


def test_noalloc_rejects_oversize_requests():
    """Sizes beyond the compiled-in scratch are refused before any launch."""
    pkg_build.build()
    dev = torch.device("cuda")
    x = torch.zeros(8, device=dev)
    for rows, cols in ((65537, 8), (8, 1025), (8, 0)):
        with pytest.raises(rikfad.RikfadError) as e:
            rikfad.step_matrix_noalloc(rows, cols, 0.1, 0.0, 0.5, 1.0, 0.0, 1e-8, "f32", x, x, x,
                                       x, x)
        assert e.value.code == rikfad.ERR_ARG
        assert "rows" in str(e.value) or "cols" in str(e.value)


def test_noalloc_binding_checks_buffers():
    """The binding refuses buffers that do not match rows x cols (the C side
    cannot check sizes) before calling the library."""
    pkg_build.build()
    dev = torch.device("cuda")
    rows, cols = 64, 32
    ok = dict(x=torch.zeros(rows, cols, device=dev), grad=torch.zeros(rows, cols, device=dev),
              p=torch.zeros(rows, cols, device=dev), R=torch.zeros(rows, device=dev),
              C=torch.zeros(cols, device=dev))
    bad = [("R", torch.zeros(rows - 1, device=dev)), ("x", torch.zeros(rows, cols - 1, device=dev)),
           ("grad", torch.zeros(rows, cols, device=dev, dtype=torch.bfloat16)),
           ("p", torch.zeros(rows, cols, device=dev, dtype=torch.float64)),
           ("C", torch.zeros(cols)), ("x", torch.zeros(cols, rows, device=dev).t())]
    for name, t in bad:
        args = dict(ok, **{name: t})
        with pytest.raises(ValueError):
            rikfad.step_matrix_noalloc(rows, cols, 0.1, 0.0, 0.5, 1.0, 0.0, 1e-8, "f32", args["x"],
                                       args["grad"], args["p"], args["R"], args["C"])
    rikfad.step_matrix_noalloc(rows, cols, 0.1, 0.0, 0.5, 1.0, 0.0, 1e-8, "f32", ok["x"], ok["grad"],
                               ok["p"], ok["R"], ok["C"])
    torch.cuda.synchronize()
