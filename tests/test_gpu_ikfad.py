"""Full-friction iKFAD (rikfad_create_ikfad) on the GPU: parity with the
oracle's element-wise rule, and the rank-1 cross-check against R-iKFAD."""
import numpy as np
import pytest

from oracle import HParams
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import workloads

from gpu_helpers import DeviceRun, Tracked, compare

pytestmark = pytest.mark.gpu

SHAPES = [(300, 768), (17, 40), (5, 0), (1000, 0), (64, 1032), (0, 8)]


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _flat(shapes):
    return [(m if n == 0 else m * n, 0) for m, n in shapes]


@pytest.mark.parametrize("grad_bf16", [True, False])
def test_ikfad_matches_oracle(grad_bf16):
    """Every tensor follows element-wise iKFAD (Eqs. ikfad_1 to ikfad_3 with the
    BACD sub-steps): 4 steps with a changing step size, against the oracle
    run alongside (1e-5 after the first step, 1e-4 after the others) and
    re-seeded from the GPU state every step (1e-5), per-element rounding
    bound beyond the relative tolerance."""
    hp = HParams(alpha=0.3, mu=1e-3, gamma=0.1, eps_stab=1e-8)
    inp = workloads.ModelInputs(SHAPES, seed=11, g_std=1e-2, grad_bf16=grad_bf16)
    run = DeviceRun(SHAPES, hp, grad_bf16, inp.X, inp.P, method="ikfad")
    flat = _flat(SHAPES)
    ref = Tracked(flat, [a.ravel() for a in inp.X], [a.ravel() for a in inp.P])

    def gpu_state():
        # the handle holds canonical momenta; every tensor is element-wise
        return ([x.ravel() for x in run.X()], [p.double().cpu().numpy().ravel() for p in run.p],
                run.factors())

    for k, h in enumerate((0.1, 0.1, 0.05, 0.2)):
        g = inp.grads(k)
        X0, P0, F0 = gpu_state()
        seeded = Tracked(flat, X0, P0, F0)
        run.set_grads(g)
        run.step(h)
        gflat = [a.ravel() for a in g]
        gpu = gpu_state()
        ref.step(gflat, h, hp, gpu[2])
        seeded.step(gflat, h, hp, gpu[2])
        seeded.check(run, 1e-5, "reseeded step%d" % (k + 1), gpu)
        ref.check(run, 1e-5 if k == 0 else 1e-4, "run step%d" % (k + 1), gpu)
    N = workloads.count(SHAPES)[0]
    assert run.opt.state_bytes(True) == 8 * N
    run.close()


@pytest.mark.parametrize("m,n", [(300, 768), (7, 5), (64, 1032)])
def test_rank1_momentum_gives_identical_friction(m, n):
    """From R = C = 0 with eps_stab = 0 and a rank-1 momentum P = a b^T (zero
    gradient), one R-iKFAD step equals one full-friction iKFAD step: the
    factored friction R_i C_j / 1^T R equals xi_ij = k P1_ij^2 (Eq. xi_def)."""
    hp = HParams(alpha=0.4, mu=0.7, gamma=0.2, eps_stab=0.0)
    rng = np.random.default_rng(m + n)
    a = rng.standard_normal(m).astype(np.float32)
    b = rng.standard_normal(n).astype(np.float32)
    X = rng.standard_normal((m, n)).astype(np.float32)
    P = np.outer(a, b).astype(np.float32)
    r1 = DeviceRun([(m, n)], hp, False, [X], [P], method="rikfad")
    fk = DeviceRun([(m, n)], hp, False, [X], [P], method="ikfad")
    for r in (r1, fk):
        r.set_grads([np.zeros((m, n), np.float32)])
        r.step(0.3)
    P_r1 = r1.canonical_P()[0]
    P_fk = fk.p[0].double().cpu().numpy()
    compare("rank1 P", P_r1, P_fk, 1e-5, 1e-2)
    compare("rank1 X", r1.X()[0], fk.X()[0], 1e-6, 1e-2)
    R, C = r1.factors()[0]
    xi_factored = np.outer(R, C) / R.sum()
    compare("rank1 friction", xi_factored.ravel(), fk.factors()[0][0], 1e-5, 1e-2)
    r1.close()
    fk.close()
