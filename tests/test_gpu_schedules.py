"""The two work schedules of the step agree: the default static schedule
(step kernel + finalise kernel) and the in-order sweep schedule (one kernel,
RIKFAD_SCHEDULE=sweep at handle creation).  Both are checked against the
oracle and the sweep for bitwise reproducibility."""
import os

import numpy as np
import pytest
import torch

from oracle import HParams
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import workloads

from gpu_helpers import DeviceRun, Tracked, compare

pytestmark = pytest.mark.gpu

SHAPES = [(1500, 768), (3, 0), (64, 3072), (17, 40), (0, 16), (4097, 0), (257, 129), (96, 1024)]
HP = HParams(alpha=0.2, mu=1e-4, gamma=0.05, eps_stab=1e-8)


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _make(schedule, inp):
    old = os.environ.get("RIKFAD_SCHEDULE")
    os.environ["RIKFAD_SCHEDULE"] = schedule
    try:
        return DeviceRun(SHAPES, HP, True, inp.X, inp.P)
    finally:
        if old is None:
            del os.environ["RIKFAD_SCHEDULE"]
        else:
            os.environ["RIKFAD_SCHEDULE"] = old


def _steps(run, inp, hs):
    for k, h in enumerate(hs):
        run.set_grads(inp.grads(k))
        run.step(h)
    torch.cuda.synchronize()


@pytest.mark.parametrize("schedule", ["static", "sweep"])
def test_schedule_matches_oracle(schedule):
    inp = workloads.ModelInputs(SHAPES, seed=21, g_std=1e-2)
    run = _make(schedule, inp)
    assert run.opt.launches_per_step() == (1 if schedule == "sweep" else 2)
    ref = Tracked(SHAPES, inp.X, inp.P)
    hs = (0.1, 0.1, 0.05)
    for k, h in enumerate(hs):
        g = inp.grads(k)
        run.set_grads(g)
        run.step(h)
        ref.step(g, h, HP, run.factors())
        ref.check(run, 1e-5 if k == 0 else 1e-4, "%s step%d" % (schedule, k + 1))
    run.close()


def test_sweep_is_reproducible_and_close_to_static():
    inp = workloads.ModelInputs(SHAPES, seed=22, g_std=1e-2)
    hs = (0.1, 0.1, 0.07, 0.07)
    a, b, c = _make("sweep", inp), _make("sweep", inp), _make("static", inp)
    for r in (a, b, c):
        _steps(r, inp, hs)
    for t in range(len(SHAPES)):
        assert torch.equal(a.x[t], b.x[t]) and torch.equal(a.p[t], b.p[t])
        Ra, Ca = a.opt.get_factors(t)
        Rb, Cb = b.opt.get_factors(t)
        assert np.array_equal(Ra, Rb) and (Ca is None or np.array_equal(Ca, Cb))
        # the schedules differ only in the order of the column sums
        compare("x[%d]" % t, a.x[t].double().cpu().numpy(), c.x[t].double().cpu().numpy(), 1e-5, 1e-2)
        compare("p[%d]" % t, a.p[t].double().cpu().numpy(), c.p[t].double().cpu().numpy(), 1e-5, 1e-2)
        Rc, Cc = c.opt.get_factors(t)
        compare("R[%d]" % t, Ra, Rc, 1e-5, 1e-2)
        if Ca is not None:
            compare("C[%d]" % t, Ca, Cc, 1e-5, 1e-2)
    for r in (a, b, c):
        r.close()
