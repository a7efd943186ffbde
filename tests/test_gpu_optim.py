"""The torch.optim front end (paper_2609_30342_gb300.optim): a small model
trained a few steps with RIKFADOptimizer takes bitwise the steps of the
pointer API on the same gradients (a parameter without a gradient steps with
a zero gradient), and its materialised momenta equal the pointer API's."""
import io
import os

import pytest
import torch

from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad
from paper_2609_30342_gb300.optim import RIKFADOptimizer

pytestmark = pytest.mark.gpu

HP = dict(alpha=0.2, mu=1e-3, gamma=0.05, eps_stab=1e-8)
H = 0.05


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _no_failed_checks(*handles):
    """On the checked build (its child run sets RIKFAD_EXPECT_CHECKED), no
    device-side plan check may have failed."""
    if os.environ.get("RIKFAD_EXPECT_CHECKED"):
        for h in handles:
            n, code = h.debug_check_failures()
            assert n == 0, "device-side plan checks failed: %d (first code %d)" % (n, code)


def _handles(opt):
    return [entry[0] for entry in opt._groups.values()]


def test_optimizer_matches_the_pointer_api():
    torch.manual_seed(0)
    model = torch.nn.Sequential(torch.nn.Linear(64, 96), torch.nn.GELU(), torch.nn.LayerNorm(96),
                                torch.nn.Linear(96, 10)).cuda()
    params = list(model.parameters())
    ref = [p.detach().clone() for p in params]
    mom = [torch.zeros_like(p) for p in params]
    shapes = [(p.shape[0], p.shape[1]) if p.dim() == 2 else (p.numel(), 0) for p in params]
    api = rikfad.RIKFAD(shapes, grad_dtype="f32", **HP)
    opt = RIKFADOptimizer(params, lr=H, **HP)
    x = torch.randn(32, 64, device="cuda")
    y = torch.randint(0, 10, (32,), device="cuda")
    for k in range(4):
        opt.zero_grad()
        torch.nn.functional.cross_entropy(model(x), y).backward()
        if k == 2:
            params[1].grad = None             # no gradient this step: a zero gradient
        grads = [torch.zeros_like(p) if p.grad is None else p.grad.detach().clone() for p in params]
        opt.step()
        api.step(H, ref, grads, mom)
        torch.cuda.synchronize()
        for a, b in zip(params, ref):
            assert torch.equal(a.detach(), b)
    opt.materialize()
    api.materialize(mom)
    torch.cuda.synchronize()
    for p, m in zip(params, mom):
        assert torch.equal(opt.state[p]["momentum"], m)
    opt.check_finite()
    _no_failed_checks(api, *_handles(opt))
    opt.close()
    api.close()



def test_state_dict_resumes_the_trajectory():
    """A checkpoint of the model and the optimiser (torch state plus the
    library's state image) taken after two steps and written with torch.save,
    loaded into a fresh optimiser over a fresh model, gives bitwise the same
    third step."""
    torch.manual_seed(1)
    model = torch.nn.Sequential(torch.nn.Linear(48, 80), torch.nn.Tanh(), torch.nn.Linear(80, 8)).cuda()
    opt = RIKFADOptimizer(model.parameters(), lr=H, **HP)
    x = torch.randn(16, 48, device="cuda")
    y = torch.randn(16, 8, device="cuda")

    def loss(m):
        return torch.nn.functional.mse_loss(m(x), y)

    for _ in range(2):
        opt.zero_grad()
        loss(model).backward()
        opt.step()
    buf = io.BytesIO()                     # a checkpoint: serialised, so nothing is shared
    torch.save({"model": model.state_dict(), "opt": opt.state_dict()}, buf)
    buf.seek(0)
    ckpt = torch.load(buf)
    clone = torch.nn.Sequential(torch.nn.Linear(48, 80), torch.nn.Tanh(), torch.nn.Linear(80, 8)).cuda()
    clone.load_state_dict(ckpt["model"])
    opt2 = RIKFADOptimizer(clone.parameters(), lr=H, **HP)
    opt2.load_state_dict(ckpt["opt"])
    for m, o in ((model, opt), (clone, opt2)):
        o.zero_grad()
        loss(m).backward()
        o.step()
    torch.cuda.synchronize()
    for a, b in zip(model.parameters(), clone.parameters()):
        assert torch.equal(a.detach(), b.detach())
    _no_failed_checks(*_handles(opt), *_handles(opt2))
    opt.close()
    opt2.close()
