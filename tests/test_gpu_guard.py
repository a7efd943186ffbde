"""Non-finite guard (GPU): a non-finite gradient element, written on the
host into the input buffer (an input value, not a device fault), is reported
as RIKFAD_ERR_NONFINITE naming its tensor; a clean run never reports; the
report blocks further steps until it is cleared, and a restored state steps
again.  The division of Eq. xi_def by 1^T R + eps_stab makes one non-finite
element poison its whole matrix, which is why the guard exists."""
import os

import pytest
import torch

from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad, workloads

pytestmark = pytest.mark.gpu

SHAPES = [(64, 256), (3, 0), (33, 40), (0, 8), (128, 0), (257, 129), (1, 1)]
HP = dict(alpha=0.0579, mu=1.3637e-6, gamma=0.0, eps_stab=1e-16)
H = 0.0918


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _setup(method="rikfad", seed=31):
    inp = workloads.ModelInputs(SHAPES, seed=seed)
    dev = torch.device("cuda")
    x = [torch.from_numpy(a).to(dev) for a in inp.X]
    p = [torch.zeros(workloads.array_shape(s), device=dev) for s in SHAPES]
    g = [torch.from_numpy(a).to(torch.bfloat16).to(dev) for a in inp.grads(0)]
    opt = rikfad.RIKFAD(SHAPES, grad_dtype="bf16", method=method, **HP)
    return inp, opt, x, g, p


@pytest.mark.parametrize("method", ["rikfad", "ikfad", "ikfad_shadow"])
def test_clean_run_never_reports(method):
    inp, opt, x, g, p = _setup(method)
    for k in range(5):
        for t, a in enumerate(inp.grads(k)):
            g[t].copy_(torch.from_numpy(a).to(torch.bfloat16))
        opt.step(H, x, g, p)
    opt.check_finite()
    opt.read_denominators()
    opt.close()


@pytest.mark.parametrize("method,tensor,value", [("rikfad", 5, float("nan")), ("rikfad", 0, float("inf")),
                                                 ("rikfad", 4, float("-inf")), ("rikfad", 6, float("nan")),
                                                 ("ikfad", 2, float("nan")),
                                                 ("ikfad_shadow", 0, float("inf"))])
def test_nonfinite_gradient_is_reported(method, tensor, value):
    """One non-finite gradient element of one tensor: the next syncing call
    reports RIKFAD_ERR_NONFINITE with that tensor's index; rikfad_step then
    refuses until the report is cleared; after restoring the checkpointed
    state the optimiser steps cleanly again."""
    inp, opt, x, g, p = _setup(method)
    opt.step(H, x, g, p)
    opt.check_finite()
    # checkpoint: factors (state image), positions and momenta
    img = torch.empty(opt.state_image_bytes(), dtype=torch.uint8, device="cuda")
    opt.export_state(img)
    xs = [a.clone() for a in x]
    ps = [a.clone() for a in p]
    pending = opt.pending_step
    # a non-finite value in the middle of the tensor's gradient
    flat = g[tensor].view(-1)
    flat[flat.numel() // 2] = value
    opt.step(H, x, g, p)
    torch.cuda.synchronize()
    with pytest.raises(rikfad.RikfadError) as e:
        opt.step(H, x, g, p)           # the report is visible: nothing more is enqueued
    assert e.value.code == rikfad.ERR_NONFINITE
    with pytest.raises(rikfad.RikfadError) as e:
        opt.read_denominators()
    assert e.value.code == rikfad.ERR_NONFINITE
    with pytest.raises(rikfad.RikfadError) as e:
        opt.check_finite()
    assert e.value.code == rikfad.ERR_NONFINITE
    assert "first tensor: %d" % tensor in str(e.value)
    # restore the checkpoint and a finite gradient: clean again
    opt.import_state(img)
    for a, b in zip(x, xs):
        a.copy_(b)
    for a, b in zip(p, ps):
        a.copy_(b)
    g[tensor].copy_(torch.from_numpy(inp.grads(0)[tensor]).to(torch.bfloat16))
    assert opt.pending_step == pending
    for _ in range(3):
        opt.step(H, x, g, p)
    opt.check_finite()
    for a in x + p:
        assert torch.isfinite(a).all()
    opt.close()


def test_nonfinite_momentum_is_reported_and_other_tensors_untouched():
    """A non-finite momentum element (a caller's corrupted buffer) is
    reported for its tensor only; the tensors before it in the list keep
    finite state (tensors are independent)."""
    inp, opt, x, g, p = _setup()
    opt.step(H, x, g, p)
    p[5].view(-1)[7] = float("nan")
    opt.step(H, x, g, p)
    with pytest.raises(rikfad.RikfadError) as e:
        opt.check_finite()
    assert e.value.code == rikfad.ERR_NONFINITE and "first tensor: 5" in str(e.value)
    for t in (0, 1, 2):
        assert torch.isfinite(x[t]).all() and torch.isfinite(p[t]).all()
    opt.close()


def test_guard_under_sweep_schedule():
    """The opt-in in-order schedule reports too (its in-kernel factor finish)."""
    os.environ["RIKFAD_SCHEDULE"] = "sweep"
    try:
        inp, opt, x, g, p = _setup()
    finally:
        del os.environ["RIKFAD_SCHEDULE"]
    assert opt.launches_per_step() == 1
    opt.step(H, x, g, p)
    opt.check_finite()
    g[0].view(-1)[100] = float("nan")
    opt.step(H, x, g, p)
    with pytest.raises(rikfad.RikfadError) as e:
        opt.check_finite()
    assert e.value.code == rikfad.ERR_NONFINITE and "first tensor: 0" in str(e.value)
    opt.close()


def test_guard_reports_from_graph_replay():
    """A step captured in a CUDA graph: replays enqueue the kernels without
    rikfad_step, so the report comes from the kernels alone.  A non-finite
    gradient written into the captured buffer between replays is reported by
    rikfad_check_finite after the next replay; clean replays before it are not."""
    inp, opt, x, g, p = _setup()
    opt.step(H, x, g, p)              # eager: pointer table uploaded, h_prev = h
    ptrs = opt.pack(x, g, p)
    opt.step(H, ptrs=ptrs)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            opt.step(H, ptrs=ptrs, stream=stream)
    # Replays go to the stream that check_finite waits on.
    with torch.cuda.stream(stream):
        for _ in range(3):
            graph.replay()
    opt.check_finite(stream)
    g[2].view(-1)[5] = float("inf")
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        graph.replay()
    with pytest.raises(rikfad.RikfadError) as e:
        opt.check_finite(stream)
    assert e.value.code == rikfad.ERR_NONFINITE and "first tensor: 2" in str(e.value)
    opt.close()
