"""The C-ABI library on the host: it loads, exports what the header declares,
and its planner covers every element exactly once (CPU only, no GPU calls)."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import oracle
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad, workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rikfad.h")


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"RIKFAD_API\s+[\w\s\*]+?\b(rikfad_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for want in ("rikfad_create", "rikfad_step", "rikfad_state_bytes", "rikfad_destroy",
                 "rikfad_materialize", "rikfad_last_error"):
        assert want in names


def test_library_exports_every_declared_symbol():
    L = ctypes.CDLL(rikfad.LIB_PATH)
    for name in declared_symbols():
        assert hasattr(L, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", rikfad.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\b(rikfad_\w+)\b", out))
    assert exported == set(declared_symbols()), exported ^ set(declared_symbols())


def test_binding_covers_every_declared_symbol():
    bound = {name for name, _, _ in rikfad.SIGNATURES}
    assert bound == set(declared_symbols())


def test_abi_version_and_error_string():
    assert rikfad.lib().rikfad_abi_version() == 1
    assert isinstance(rikfad.lib().rikfad_last_error(), bytes)


GPT2S = [s for _, s in workloads.gpt2_small()]
NANO = [s for _, s in workloads.gpt2_nano()]
ODD = [(1, 1), (1, 7), (3, 5), (257, 129), (0, 4), (5, 0), (0, 0), (13, 0), (9, 2048),
       (2, 3000), (4096, 8), (100, 1032)]


# The planner's per-row cost of a matrix panel row, in bytes (kRowCost in
# csrc/rikfad_plan.hpp): blocks are balanced on bytes plus this per row.
ROW_COST = 256


def _bytes(shape, gb):
    m, n = shape
    return m * (gb + 24) if n == 0 else m * n * (gb + 16)


@pytest.mark.parametrize("shapes", [GPT2S, NANO, ODD, workloads.SWEEP_SHAPES[:2], [(256, 512)]],
                         ids=["gpt2s", "nano", "odd", "sweep", "single"])
@pytest.mark.parametrize("nblocks", [1, 7, 304, 1216])
@pytest.mark.parametrize("grad", ["bf16", "f32"])
def test_plan_covers_every_element_once(shapes, nblocks, grad):
    plan = rikfad.plan_query(shapes, grad, nblocks)
    gb = 2 if grad == "bf16" else 4
    blocks = plan[:, 0]
    assert np.all(np.diff(blocks) >= 0), "pieces out of block order"
    assert blocks.size == 0 or (blocks.min() >= 0 and blocks.max() < nblocks)
    # Coverage: mark every (row, column) of every matrix and every element of
    # every vector; each must be hit exactly once.
    hits = [np.zeros(workloads.array_shape(s), np.int32) for s in shapes]
    slots = []
    for b, t, kind, col0, width, beg, end, slot in plan:
        m, n = shapes[t]
        assert beg < end
        if kind == 0:
            assert n > 0 and 0 <= beg and end <= m and 0 <= col0 and col0 + width <= n
            assert width <= 1024
            if n % 8 == 0:
                assert col0 % 8 == 0 and width % 8 == 0
            hits[t][beg:end, col0:col0 + width] += 1
            slots.append(slot)
        else:
            assert n == 0 and 0 <= beg and end <= m and beg % 8 == 0
            hits[t][beg:end] += 1
    for t, hit in enumerate(hits):
        assert np.all(hit == 1), "tensor %d covered %s times" % (t, np.unique(hit))
    assert slots == list(range(len(slots))), "slots must be consecutive in piece order"
    # Balance: no block exceeds its fair share of the planner's cost (bytes,
    # plus ROW_COST per matrix panel row) by more than one unit of work; the
    # bytes of all pieces add up to the compulsory bytes of the list.
    if plan.size:
        total_bytes = sum(_bytes(s, gb) for s in shapes)
        used = int(blocks.max()) + 1
        per_block = np.zeros(used)
        bytes_sum = 0.0
        largest_unit = 0
        for b, t, kind, col0, width, beg, end, slot in plan:
            unit = width * (gb + 16) + ROW_COST if kind == 0 else 8 * (gb + 24)
            largest_unit = max(largest_unit, unit)
            per_block[b] += (end - beg) * unit / (1 if kind == 0 else 8)
            bytes_sum += (end - beg) * (width * (gb + 16) if kind == 0 else gb + 24)
        assert abs(bytes_sum - total_bytes) < 1e-6 * total_bytes
        fair = per_block.sum() / used
        assert per_block.max() <= fair + 2 * largest_unit + 1, (per_block.max(), fair)


def test_plan_rejects_bad_arguments():
    with pytest.raises(rikfad.RikfadError):
        rikfad.plan_query([(-1, 3)], "bf16", 10)
    with pytest.raises(rikfad.RikfadError):
        rikfad.plan_query([(3, 3)], "bf16", 0)


def test_state_bytes_match_oracle_count():
    for shapes in (GPT2S, NANO, ODD):
        assert rikfad.state_bytes_for(shapes, True) == 4 * oracle.state_scalars(shapes)
        N = workloads.count(shapes)[0]
        assert rikfad.state_bytes_for(shapes, False) == 4 * (oracle.state_scalars(shapes) - N)


def test_state_bytes_gpt2s_vs_full_friction():
    """R-iKFAD on GPT2-S (split q/k/v): 4 (N + sum(m + n) + 1-D) bytes; full
    iKFAD / Adam keep 2N floats."""
    N, mats, mn, one_d = workloads.count(GPT2S)
    assert (N, mats, mn, one_d) == (124439808, 74, 218705, 121344)
    assert rikfad.state_bytes_for(GPT2S, True) == 4 * (N + mn + one_d) == 499119428


def test_quadratic_run_rejects_bad_arguments_before_any_cuda_call():
    """rikfad_quadratic_run checks sizes, hyperparameters and pointers on the
    host and returns RIKFAD_ERR_ARG before touching the GPU."""
    L = rikfad.lib()
    hp = rikfad.HParams(1.0, 1.0, 0.0, 0.0)
    bad_hp = rikfad.HParams(1.0, 0.0, 0.0, 0.0)
    one = ctypes.c_void_p(64)
    cases = [
        (1, 6, 6, hp, 10, 0),          # m n = 36 > 32
        (1, 0, 3, hp, 10, 0),          # m = 0
        (1, 2, 2, hp, -1, 0),          # nsteps < 0
        (-1, 2, 2, hp, 10, 0),         # batch < 0
        (1, 2, 2, bad_hp, 10, 0),      # mu = 0
        (1, 2, 2, hp, 10, 3),          # record and energy NULL with nrecord > 0
    ]
    for batch, m, n, h, nsteps, nrec in cases:
        rc = L.rikfad_quadratic_run(batch, m, n, one, one, one, one, one, 0.02, ctypes.byref(h), nsteps,
                                    None, nrec, None, None)
        assert rc == rikfad.ERR_ARG, (batch, m, n, nsteps, nrec, rc)
    rc = L.rikfad_quadratic_run(1, 2, 2, None, one, one, one, one, 0.02, ctypes.byref(hp), 10, None, 0,
                                None, None)
    assert rc == rikfad.ERR_ARG
    rc = L.rikfad_quadratic_run(1, 2, 2, one, one, one, one, one, 0.0, ctypes.byref(hp), 10, None, 0,
                                None, None)
    assert rc == rikfad.ERR_ARG
    rc = L.rikfad_quadratic_run(1, 2, 2, ctypes.c_void_p(66), one, one, one, one, 0.02, ctypes.byref(hp),
                                10, None, 0, None, None)
    assert rc == rikfad.ERR_ALIGN
    # batch = 0 is a no-op that succeeds without a device.
    assert L.rikfad_quadratic_run(0, 2, 2, None, None, None, None, None, 0.02, ctypes.byref(hp), 10,
                                  None, 0, None, None) == rikfad.OK


@pytest.mark.parametrize("cols", [8, 40, 384, 576, 768, 800, 1032, 1536, 1600, 2048, 3000, 3072, 6400, 14336])
def test_panels_are_whole_chunks(cols):
    """On the 8-wide path (cols a multiple of 8) every column panel of a
    matrix but its last is a whole number of 256-column chunks and at most
    1024 wide, so a row takes the fewest chunk round trips, ceil(cols/256)."""
    plan = rikfad.plan_query([(64, cols)], "bf16", 4)
    panels = sorted({(int(c0), int(w)) for c0, w in zip(plan[:, 3], plan[:, 4])})
    assert sum(w for _, w in panels) == cols
    assert all(w <= 1024 for _, w in panels)
    assert all(w % 256 == 0 for _, w in panels[:-1]), panels
    assert sum(-(-w // 256) for _, w in panels) == -(-cols // 256)


C_CLIENT = r"""
#include <stdio.h>
#include "rikfad.h"
int main(void)
{
    rikfad_shape shapes[2] = {{768, 768}, {768, 0}};
    rikfad_hparams bad = {1.0, 0.0, 0.0, 0.0};
    size_t bytes = rikfad_state_bytes_for(shapes, 2, 1);
    int64_t rows = rikfad_plan_query(shapes, 2, RIKFAD_GRAD_BF16, 4, NULL, 0);
    int rc = rikfad_quadratic_run(1, 2, 2, NULL, NULL, NULL, NULL, NULL, 0.02, &bad, 10, NULL, 0,
                                  NULL, NULL);
    printf("%d %zu %lld %d\n", rikfad_abi_version(), bytes, (long long)rows, rc);
    return 0;
}
"""


def test_plain_c_client(tmp_path):
    """The boundary is a C ABI: include/rikfad.h compiles as strict C99 and a C
    program links against the library and calls it (host-only calls)."""
    import shutil
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(rikfad.LIB_PATH)
    subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I",
                    os.path.join(ROOT, "include"), str(src), "-L", libdir, "-lrikfad",
                    "-Wl,-rpath," + libdir, "-o", str(exe)], check=True, capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    assert int(out[0]) == rikfad.lib().rikfad_abi_version()
    assert int(out[1]) == 4 * (768 * 768 + 768 + 768 + 2 * 768)
    assert int(out[2]) > 0
    assert int(out[3]) == rikfad.ERR_ARG
