"""Failure of an allocation inside rikfad_create (GPU; the failure is
injected on the host, no memory is exhausted): every allocation site in
turn reports failure, and each time rikfad_create returns RIKFAD_ERR_OOM,
leaves *out NULL and holds no allocation afterwards."""
import ctypes
import os

import pytest
import torch

from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad

pytestmark = pytest.mark.gpu

SHAPES = [(300, 768), (5, 0), (4097, 0), (33, 40), (2, 3000), (0, 16)]


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _create(which, schedule=None):
    L = rikfad.lib()
    arr = rikfad._shapes(SHAPES)
    hp = rikfad.HParams(0.3, 1e-3, 0.1, 1e-8)
    out = ctypes.c_void_p(0x1234)
    fn = {"rikfad": L.rikfad_create, "ikfad": L.rikfad_create_ikfad,
          "ikfad_shadow": L.rikfad_create_ikfad_shadow}[which]
    old = os.environ.get("RIKFAD_SCHEDULE")
    if schedule:
        os.environ["RIKFAD_SCHEDULE"] = schedule
    try:
        rc = fn(arr, len(SHAPES), ctypes.byref(hp), rikfad.GRAD_BF16, ctypes.byref(out))
    finally:
        if schedule:
            if old is None:
                del os.environ["RIKFAD_SCHEDULE"]
            else:
                os.environ["RIKFAD_SCHEDULE"] = old
    return rc, out.value


@pytest.mark.parametrize("which,schedule", [("rikfad", None), ("ikfad", None), ("ikfad_shadow", None),
                                            ("rikfad", "sweep")])
def test_every_allocation_failure_is_clean(which, schedule):
    torch.cuda.synchronize()
    live0 = rikfad.debug_live_allocations()
    free0 = torch.cuda.mem_get_info()[0]
    sites = 0
    try:
        for n in range(1, 200):
            rikfad.debug_fail_allocation(n)
            rc, h = _create(which, schedule)
            if rc == rikfad.OK:
                # n passed the last allocation: the handle is complete
                assert h is not None
                rikfad.debug_fail_allocation(0)
                rikfad.lib().rikfad_destroy(h)
                break
            sites += 1
            msg = rikfad.lib().rikfad_last_error().decode()
            assert rc == rikfad.ERR_OOM, (n, rc, msg)
            assert h is None, "out must be NULL on failure"
            assert "out of memory" in msg
            assert rikfad.debug_live_allocations() == live0, "allocation %d leaked" % n
        else:
            pytest.fail("rikfad_create never succeeded")
    finally:
        rikfad.debug_fail_allocation(0)
    assert sites >= 10, sites
    assert rikfad.debug_live_allocations() == live0
    torch.cuda.synchronize()
    # no device memory kept either (the driver frees in pages: allow 4 MiB of noise)
    assert torch.cuda.mem_get_info()[0] >= free0 - (4 << 20)
    # a normal create afterwards works
    opt = rikfad.RIKFAD(SHAPES, 0.3, 1e-3, 0.1, 1e-8, "bf16", method=which)
    opt.close()
    assert rikfad.debug_live_allocations() == live0


def test_sweep_state_allocated_only_when_selected():
    """The in-order schedule's units, trees and partials exist only for a
    handle created with RIKFAD_SCHEDULE=sweep."""
    live0 = rikfad.debug_live_allocations()
    a = rikfad.RIKFAD(SHAPES, 0.3, 1e-3, 0.1, 1e-8, "bf16")
    na = rikfad.debug_live_allocations() - live0
    os.environ["RIKFAD_SCHEDULE"] = "sweep"
    try:
        b = rikfad.RIKFAD(SHAPES, 0.3, 1e-3, 0.1, 1e-8, "bf16")
    finally:
        del os.environ["RIKFAD_SCHEDULE"]
    nb = rikfad.debug_live_allocations() - live0 - na
    assert nb == na + 6, (na, nb)
    assert b.workspace_bytes() > a.workspace_bytes()
    assert a.launches_per_step() == 2 and b.launches_per_step() == 1
    a.close()
    b.close()
    assert rikfad.debug_live_allocations() == live0
