"""Full iKFAD with shadow R-iKFAD factors and the friction diagnostic on the
GPU (rikfad_create_ikfad_shadow, rikfad_friction_diagnostics) against the
oracle of the paper's Section 4.4 comparison."""
import numpy as np
import pytest

from oracle import HParams
from oracle.diagnostics import friction_metrics, shadow_step
import oracle
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import workloads

from gpu_helpers import DeviceRun, compare

pytestmark = pytest.mark.gpu

SHAPES = [(300, 768), (17, 40), (5, 0), (64, 1032), (0, 8), (129, 257), (2, 3072)]
HP = HParams(alpha=0.3, mu=1e-3, gamma=0.05, eps_stab=1e-8)


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


class ShadowRef:
    """Oracle state of a shadow run (matrices: X, P, XI, R, C; vectors: the
    C oracle's element-wise rule)."""

    def __init__(self, shapes, X, P, XI=None, RC=None):
        self.shapes = shapes
        self.X = [np.array(a, np.float64) for a in X]
        self.P = [np.array(a, np.float64) for a in P]
        self.XI = [np.zeros(workloads.array_shape(s)) for s in shapes] if XI is None else \
            [np.array(a, np.float64) for a in XI]
        self.R = [np.zeros(m) if n else None for m, n in shapes] if RC is None else [r for r, _ in RC]
        self.C = [np.zeros(n) if n else None for m, n in shapes] if RC is None else [c for _, c in RC]

    def step(self, grads, h):
        for t, (m, n) in enumerate(self.shapes):
            g = np.asarray(grads[t], np.float64)
            if n == 0:
                oracle.step_vector(self.X[t], self.P[t], self.XI[t], g.copy(), h, HP)
            else:
                self.X[t], self.P[t], self.XI[t], self.R[t], self.C[t] = shadow_step(
                    self.X[t], self.P[t], self.XI[t], self.R[t], self.C[t], g, h, HP)


def _gpu_state(run):
    X = run.X()
    P = [p.double().cpu().numpy() for p in run.p]
    XI = [run.opt.get_friction(t).astype(np.float64) for t in range(len(run.shapes))]
    RC = [tuple(None if a is None else a.astype(np.float64) for a in run.opt.get_factors(t))
          if n else (None, None) for t, (m, n) in enumerate(run.shapes)]
    return X, P, XI, RC


def _compare(run, ref, rtol, tag):
    X, P, XI, RC = _gpu_state(run)
    for t, (m, n) in enumerate(run.shapes):
        compare("%sX[%d]" % (tag, t), X[t], ref.X[t], rtol, 1e-2)
        compare("%sP[%d]" % (tag, t), P[t], ref.P[t], rtol, 1e-2)
        compare("%sxi[%d]" % (tag, t), XI[t], ref.XI[t], rtol, 1e-2)
        if n:
            compare("%sR[%d]" % (tag, t), RC[t][0], ref.R[t], rtol, 1e-2)
            compare("%sC[%d]" % (tag, t), RC[t][1], ref.C[t], rtol, 1e-2)


@pytest.mark.parametrize("grad_bf16", [True, False])
def test_shadow_run_matches_oracle(grad_bf16):
    inp = workloads.ModelInputs(SHAPES, seed=41, g_std=1e-2, grad_bf16=grad_bf16)
    run = DeviceRun(SHAPES, HP, grad_bf16, inp.X, inp.P, method="ikfad_shadow")
    ref = ShadowRef(SHAPES, inp.X, inp.P)
    for k, h in enumerate((0.1, 0.1, 0.05, 0.2)):
        X, P, XI, RC = _gpu_state(run)
        seeded = ShadowRef(SHAPES, X, P, XI, RC)
        g = inp.grads(k)
        run.set_grads(g)
        run.step(h)
        ref.step(g, h)
        seeded.step(g, h)
        _compare(run, seeded, 1e-5, "reseeded step%d " % (k + 1))
        _compare(run, ref, 1e-4, "step%d " % (k + 1))
    N, _, mn, one_d = workloads.count(SHAPES)
    assert run.opt.state_bytes(True) == 4 * (2 * N + mn)
    run.close()


def test_diagnostics_match_dense_linear_algebra():
    """On the GPU run's own state, the diagnostic equals the dense numpy
    computation (SVD for sigma_1): error, floor, stable rank, sigma_1, norm."""
    shapes = [(600, 768), (129, 257), (64, 1032), (2000, 64)]
    inp = workloads.ModelInputs(shapes, seed=42, g_std=1e-2)
    run = DeviceRun(shapes, HP, True, inp.X, inp.P, method="ikfad_shadow")
    for k in range(6):
        run.set_grads(inp.grads(k))
        run.step(0.1)
    for t, (m, n) in enumerate(shapes):
        err, floor, sr, s1, frob, iters = run.opt.friction_diagnostics(t, max_iters=500, tol=1e-12)
        XI = run.opt.get_friction(t).astype(np.float64)
        R, C = (a.astype(np.float64) for a in run.opt.get_factors(t))
        e_ref, f_ref, sr_ref, s1_ref, frob_ref = friction_metrics(XI, R, C, HP.eps_stab)
        assert abs(err - e_ref) <= 1e-4 * e_ref + 1e-7, (t, err, e_ref)
        assert abs(frob - frob_ref) <= 1e-5 * frob_ref, (t, frob, frob_ref)
        assert abs(s1 - s1_ref) <= 1e-5 * s1_ref, (t, s1, s1_ref, iters)
        assert abs(sr - sr_ref) <= 1e-4 * sr_ref, (t, sr, sr_ref)
        # the floor is a difference 1 - sigma_1^2/||xi||^2: compare its square absolutely
        assert abs(floor ** 2 - f_ref ** 2) <= 2e-5, (t, floor, f_ref)
        assert 1.0 <= sr and floor <= err + 1e-6      # no rank-1 friction beats the best one
    run.close()


def test_rank1_momentum_gives_zero_construction_error_on_gpu():
    """Rank-1 momentum, zero gradient, zero state, eps_stab = 0: after one
    step the shadow rank-1 friction equals the element-wise friction."""
    hp = HParams(alpha=0.5, mu=0.8, gamma=0.0, eps_stab=0.0)
    rng = np.random.default_rng(43)
    m, n = 256, 512
    a, b = rng.standard_normal(m).astype(np.float32), rng.standard_normal(n).astype(np.float32)
    run = DeviceRun([(m, n)], hp, False, [np.zeros((m, n), np.float32)], [np.outer(a, b)],
                 method="ikfad_shadow")
    run.set_grads([np.zeros((m, n), np.float32)])
    run.step(0.3)
    err, floor, sr, s1, frob, iters = run.opt.friction_diagnostics(0)
    assert err < 2e-5 and abs(sr - 1.0) < 1e-4 and floor < 1e-2, (err, floor, sr)
    run.close()


def test_diagnostics_refused_for_other_handles():
    from paper_2609_30342_gb300 import rikfad
    opt = rikfad.RIKFAD([(8, 8)], 0.1, 1.0)
    with pytest.raises(rikfad.RikfadError) as e:
        opt.friction_diagnostics(0)
    assert e.value.code == rikfad.ERR_STATE
    opt.close()
