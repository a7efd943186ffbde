"""The torch.optim front end's argument checks on the host (no GPU): they
raise before any handle is created or any library call is made."""
import pytest
import torch

from paper_2609_30342_gb300.optim import RIKFADOptimizer

HP = dict(alpha=0.2, mu=1e-3, gamma=0.05, eps_stab=1e-8)


def test_rejects_a_non_positive_step_size():
    with pytest.raises(ValueError):
        RIKFADOptimizer([torch.nn.Parameter(torch.zeros(4, 4))], lr=0.0, **HP)


def test_rejects_cpu_parameters_before_any_library_call():
    p = torch.nn.Parameter(torch.zeros(4, 4))
    opt = RIKFADOptimizer([p], lr=0.05, **HP)
    p.grad = torch.zeros(4, 4)
    with pytest.raises(ValueError):
        opt.step()
    assert opt._groups == {}
