"""The allocation-free single-matrix step against the handle API (GPU).

rikfad_step_matrix_noalloc exists for callers that cannot allocate device
memory themselves: programs whose framework allocator already owns the GPU's
memory, and services that forbid cudaMalloc after start-up because it can
stall the device.  It keeps its partial sums in an array compiled into the
library, so it must give the same results as the ordinary handle-based step
(which allocates its workspace in rikfad_create), call after call.

This file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad

from gpu_helpers import compare

pytestmark = pytest.mark.gpu

HP = dict(alpha=0.5, mu=1e-6, gamma=0.1, eps_stab=1e-8)
STEPS = (0.05, 0.03)


@pytest.mark.parametrize("rows,cols,grad", [(3000, 768, "bf16"), (257, 129, "f32"),
                                            (65536, 1024, "bf16")])
def test_noalloc_step_matches_handle_step(rows, cols, grad):
    """Two calls in a row (the second with a different step size, so the
    pending factor of the first is applied): X, the stored momentum and both
    factors agree with rikfad_step within the parity tolerance of the tests."""
    pkg_build.build()
    dev = torch.device("cuda")
    gdt = torch.bfloat16 if grad == "bf16" else torch.float32
    gen = torch.Generator(device="cpu").manual_seed(rows + cols)
    X0 = 0.02 * torch.randn(rows, cols, generator=gen)
    P0 = 0.01 * torch.randn(rows, cols, generator=gen)
    G = [(1e-3 * torch.randn(rows, cols, generator=gen)).to(gdt).to(dev) for _ in STEPS]

    # the handle API (allocates its workspace in rikfad_create)
    opt = rikfad.RIKFAD([(rows, cols)], grad_dtype=grad, **HP)
    xa, pa = X0.to(dev), P0.to(dev)
    # the allocation-free entry point: caller-owned state, zero factors
    xb, pb = X0.to(dev), P0.to(dev)
    R = torch.zeros(rows, dtype=torch.float32, device=dev)
    C = torch.zeros(cols, dtype=torch.float32, device=dev)

    pending = 0.0
    for k, h in enumerate(STEPS):
        opt.step(h, [xa], [G[k]], [pa])
        rikfad.step_matrix_noalloc(rows, cols, h, pending, HP["alpha"], HP["mu"], HP["gamma"],
                                   HP["eps_stab"], grad, xb, G[k], pb, R, C)
        pending = h
        torch.cuda.synchronize()
        Ra, Ca = opt.get_factors(0)
        tag = "%dx%d call %d " % (rows, cols, k + 1)
        compare(tag + "X", xb.double().cpu().numpy(), xa.double().cpu().numpy(), 1e-5, 1e-2)
        compare(tag + "P", pb.double().cpu().numpy(), pa.double().cpu().numpy(), 1e-5, 1e-2)
        compare(tag + "R", R.double().cpu().numpy(), Ra.astype(np.float64), 1e-5, 1e-2)
        compare(tag + "C", C.double().cpu().numpy(), Ca.astype(np.float64), 1e-5, 1e-2)
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
