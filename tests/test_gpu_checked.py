"""The checked build (GPU): librikfad_checked.so, compiled with
RIKFAD_CHECKED, verifies in every kernel each plan index, range and buffer
offset and each pointer-table entry before using it, counting failures
instead of trapping.  The edge-shape, degenerate-hyperparameter,
Nano-shaped and full GPT2-S (the benchmark's launch configuration) parity
cases, the C-ABI behaviour tests, full iKFAD, the shadow
handle, the in-order schedule and the torch.optim front end run on it in a
child process (the library
is chosen when the binding first loads it), and every handle must end with
zero failed checks; the parity assertions themselves hold as on the
ordinary build."""
import os
import subprocess
import sys

import pytest

from paper_2609_30342_gb300 import build as pkg_build

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_parity_cases_on_checked_build():
    lib = pkg_build.build(checked=True)
    env = dict(os.environ, RIKFAD_LIBRARY=lib, RIKFAD_EXPECT_CHECKED="1")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
           "-k", "not test_gpu_parity or edge_shapes or degenerate or nano_shaped_full_model or "
                 "gpt2_small_full_size",
           os.path.join(HERE, "test_gpu_parity.py"), os.path.join(HERE, "test_gpu_api.py"),
           os.path.join(HERE, "test_gpu_ikfad.py"), os.path.join(HERE, "test_gpu_diagnostics.py"),
           os.path.join(HERE, "test_gpu_schedules.py"), os.path.join(HERE, "test_gpu_optim.py")]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    tail = (r.stdout + r.stderr)[-3000:]
    assert r.returncode == 0, tail
    assert " passed" in r.stdout and "checked handles: " in r.stdout, tail
