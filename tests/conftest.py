import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_collection_modifyitems(config, items):
    # GPU tests need a device; on a CPU-only machine they are skipped rather than failed.
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


def pytest_terminal_summary(terminalreporter):
    # Per-element parity statistics of the GPU tests (how many elements
    # needed the rounding bound beyond the pure relative tolerance).
    gh = sys.modules.get("gpu_helpers")
    if gh is not None and os.environ.get("RIKFAD_EXPECT_CHECKED"):
        terminalreporter.write_line("checked handles: %d, failed device checks: %d"
                                    % (len(gh.CHECKED), sum(gh.CHECKED)))
    em = sys.modules.get("error_model")
    if em is None or not em.STATS:
        return
    terminalreporter.write_sep("-", "parity: elements beyond the pure relative tolerance")
    for line in em.summary_lines():
        terminalreporter.write_line(line)
