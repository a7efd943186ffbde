"""Behaviour of the C ABI on the GPU: determinism, stored-form semantics,
checkpoints, pointer changes, error codes, CUDA-graph replay."""
import numpy as np
import pytest
import torch

from oracle import HParams
from paper_2609_30342_gb300 import build as pkg_build
from paper_2609_30342_gb300 import rikfad, workloads

from gpu_helpers import DeviceRun, Tracked

pytestmark = pytest.mark.gpu

SHAPES = [(300, 768), (5, 0), (64, 1032), (17, 40), (1000, 0), (2, 3072)]
HP = HParams(alpha=0.2, mu=1e-4, gamma=0.05, eps_stab=1e-8)


@pytest.fixture(scope="module", autouse=True)
def built():
    pkg_build.build()
    yield


def _run(seed=0, grad_bf16=True):
    inp = workloads.ModelInputs(SHAPES, seed=seed, g_std=1e-2, grad_bf16=grad_bf16)
    return inp, DeviceRun(SHAPES, HP, grad_bf16, inp.X, inp.P)


def _state(run):
    return [x.clone() for x in run.x], [p.clone() for p in run.p], run.factors()


def test_bitwise_deterministic():
    """Two runs from identical inputs give bitwise-identical states (fixed
    reduction order, no atomics)."""
    outs = []
    for _ in range(2):
        inp, run = _run()
        for k, h in enumerate((0.1, 0.1, 0.07)):
            run.set_grads(inp.grads(k))
            run.step(h)
        torch.cuda.synchronize()
        outs.append(_state(run))
        run.close()
    (xa, pa, fa), (xb, pb, fb) = outs
    for a, b in zip(xa + pa, xb + pb):
        assert torch.equal(a, b)
    for (ra, ca), (rb, cb) in zip(fa, fb):
        assert np.array_equal(ra, rb)
        assert (ca is None and cb is None) or np.array_equal(ca, cb)


def test_materialize_keeps_the_trajectory():
    """Materialising between steps (P becomes canonical, pending factor
    cleared) changes only rounding: the trajectory stays on the oracle's."""
    inp, run = _run()
    ref = Tracked(SHAPES, inp.X, inp.P)
    for k in range(4):
        g = inp.grads(k)
        run.set_grads(g)
        run.step(0.1)
        ref.step(g, 0.1, HP, run.factors())
        if k == 1:
            assert run.opt.pending_step == pytest.approx(0.1)
            before = run.canonical_P()
            run.opt.materialize(run.p)
            assert run.opt.pending_step == 0.0
            after = [p.double().cpu().numpy() for p in run.p]
            for a, b in zip(before, after):
                assert np.array_equal(a, b)   # same expression, same rounding
    ref.check(run, 1e-4, "after materialize")
    run.close()


def test_canonical_momentum_leaves_state_alone():
    inp, run = _run()
    run.set_grads(inp.grads(0))
    run.step(0.1)
    p_before = [p.clone() for p in run.p]
    out1 = run.canonical_P()
    out2 = run.canonical_P()
    for a, b in zip(p_before, run.p):
        assert torch.equal(a, b)
    for a, b in zip(out1, out2):
        assert np.array_equal(a, b)
    assert run.opt.pending_step == pytest.approx(0.1)
    with pytest.raises(rikfad.RikfadError):
        run.opt.canonical_momentum(run.p, run.p)     # out must not alias p
    run.close()


def test_export_import_round_trip():
    """Checkpoint the factors and the pending step, run on, restore, rerun:
    bitwise the same continuation."""
    inp, run = _run()
    for k in range(2):
        run.set_grads(inp.grads(k))
        run.step(0.1)
    img = torch.empty(run.opt.state_image_bytes(), dtype=torch.uint8, device="cuda")
    run.opt.export_state(img)
    x0, p0, _ = _state(run)
    g2 = inp.grads(2)
    run.set_grads(g2)
    run.step(0.05)
    first = _state(run)
    # restore and repeat
    for dst, src in zip(run.x + run.p, x0 + p0):
        dst.copy_(src)
    run.opt.import_state(img)
    assert run.opt.pending_step == pytest.approx(0.1)
    run.set_grads(g2)
    run.step(0.05)
    second = _state(run)
    for a, b in zip(first[0] + first[1], second[0] + second[1]):
        assert torch.equal(a, b)
    for (ra, ca), (rb, cb) in zip(first[2], second[2]):
        assert np.array_equal(ra, rb)
    # a corrupted image is refused
    bad = img.clone()
    bad[:8] = 0
    with pytest.raises(rikfad.RikfadError):
        run.opt.import_state(bad)
    run.close()


def test_pointer_sets_may_change_between_steps():
    """Two parameter sets stepped alternately through one handle: the device
    pointer table follows the pointers of each call."""
    inp, run = _run()
    xb = [x.clone() for x in run.x]
    pb = [p.clone() for p in run.p]
    gb = [g.clone() for g in run.g]
    ptr_b = run.opt.pack(xb, gb, pb)
    run.set_grads(inp.grads(0))
    for g_dst, g_src in zip(gb, run.g):
        g_dst.copy_(g_src)
    run.opt.step(0.1, ptrs=run.ptrs)      # set A
    # set B sees the factors A just produced: a different (valid) trajectory
    run.opt.step(0.1, ptrs=ptr_b)
    torch.cuda.synchronize()
    # each set moved from its own X: both finite and changed
    for x0, xa, xbb in zip(inp.X, run.x, xb):
        if x0.size:
            assert torch.isfinite(xa).all() and torch.isfinite(xbb).all()
            assert not np.array_equal(xa.cpu().numpy(), x0)
            assert not np.array_equal(xbb.cpu().numpy(), x0)
    run.close()


def test_argument_errors_are_reported():
    inp, run = _run()
    opt = run.opt
    T = len(SHAPES)
    # misaligned pointer (16-byte alignment required on the vector path)
    xs = list(run.x)
    xs[0] = torch.zeros(300 * 768 + 1, device="cuda")[1:].view(300, 768)
    with pytest.raises(rikfad.RikfadError) as e:
        opt.step(0.1, xs, run.g, run.p)
    assert e.value.code == rikfad.ERR_ALIGN
    # NULL pointer for a non-empty tensor
    with pytest.raises(rikfad.RikfadError) as e:
        opt.step(0.1, [None] + run.x[1:], run.g, run.p)
    assert e.value.code == rikfad.ERR_ARG
    # bad step sizes
    for h in (0.0, -1.0, float("nan"), float("inf")):
        with pytest.raises(rikfad.RikfadError) as e:
            opt.step(h, run.x, run.g, run.p)
        assert e.value.code == rikfad.ERR_ARG
    # bad tensor index, bad factor values
    with pytest.raises(rikfad.RikfadError):
        opt.get_factors(T)
    buf = np.zeros(4096, np.float32)
    assert rikfad.lib().rikfad_get_factors(opt.handle, T, buf.ctypes.data, None) == rikfad.ERR_ARG
    assert rikfad.lib().rikfad_get_factors(opt.handle, -1, buf.ctypes.data, None) == rikfad.ERR_ARG
    with pytest.raises(rikfad.RikfadError):
        opt.set_factors(0, -np.ones(300, np.float32), np.ones(768, np.float32))
    # nothing was enqueued: the state still steps normally afterwards
    run.set_grads(inp.grads(0))
    run.step(0.1)
    torch.cuda.synchronize()
    for x in run.x:
        assert torch.isfinite(x).all()
    run.close()
    # bad hyperparameters and shapes at creation
    for kw in (dict(alpha=0.0, mu=1.0), dict(alpha=1.0, mu=0.0), dict(alpha=1.0, mu=1.0, gamma=-1.0),
               dict(alpha=1.0, mu=1.0, eps_stab=-1e-3)):
        with pytest.raises(rikfad.RikfadError):
            rikfad.RIKFAD([(4, 4)], **kw)
    with pytest.raises(rikfad.RikfadError):
        rikfad.RIKFAD([(4, -1)], 1.0, 1.0)


def test_empty_parameter_list():
    opt = rikfad.RIKFAD([], 0.1, 1.0)
    opt.step(0.1, [], [], [])
    assert opt.state_bytes() == 0
    assert opt.launches_per_step() == 0
    opt.close()


def test_cuda_graph_replay_matches_eager():
    """rikfad_step enqueues only kernels on the caller's stream, so a captured
    step replays in a CUDA graph.  With a constant step size (after one eager
    step with that size) replays match eager steps bitwise."""
    inp, run_e = _run()
    _, run_g = _run()
    g = inp.grads(0)
    run_e.set_grads(g)
    run_g.set_grads(g)
    run_e.step(0.1)
    run_g.step(0.1)          # eager: uploads the pointer table, sets h_prev = h
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            run_g.opt.step(0.1, ptrs=run_g.ptrs, stream=stream)
    torch.cuda.synchronize()
    for _ in range(3):
        run_e.step(0.1)
        graph.replay()
    torch.cuda.synchronize()
    # the capture itself does not run the kernels: 1 eager + 3 replays = 4 steps each
    (xe, pe, fe), (xg, pg, fg) = _state(run_e), _state(run_g)
    # run_e took 1 + 3 eager steps; the graph side 1 eager + 3 replays
    for a, b in zip(xe + pe, xg + pg):
        assert torch.equal(a, b)
    for (ra, ca), (rb, cb) in zip(fe, fg):
        assert np.array_equal(ra, rb)
    run_e.close()
    run_g.close()


def test_profile_counters():
    inp, run = _run()
    run.opt.profile_enable(True)
    run.set_grads(inp.grads(0))
    for _ in range(5):
        run.step(0.1)
    a, b, n = run.opt.profile_read()
    assert n == 5 and a > 0 and b >= 0
    # one kernel per step with the in-order schedule, step + finalise otherwise
    assert run.opt.launches_per_step() in (1, 2)
    run.opt.profile_enable(False)
    run.close()


def test_pinned_host_gradients_read_in_place():
    """Gradients may live in page-locked host memory: the step kernel reads
    them across the CPU-GPU link and gives bitwise the same step."""
    inp, run_d = _run()
    _, run_h = _run()
    g = inp.grads(0)
    run_d.set_grads(g)
    host_g = [torch.from_numpy(a).to(torch.bfloat16).pin_memory() for a in g]
    ptr_h = run_h.opt.pack(run_h.x, host_g, run_h.p)
    for h in (0.1, 0.1, 0.05):
        run_d.step(h)
        run_h.opt.step(h, ptrs=ptr_h)
    torch.cuda.synchronize()
    for a, b in zip(run_d.x + run_d.p, run_h.x + run_h.p):
        assert torch.equal(a, b)
    run_d.close()
    run_h.close()


def test_enqueued_denominators_match_the_synchronous_read():
    """rikfad_enqueue_denominators writes, once the stream passes it, the
    values rikfad_read_denominators returns; read back one step late (while
    the next step runs), every step's values equal 1^T R of that step's
    factors, and element-wise tensors read 0."""
    inp, run = _run()
    stream = torch.cuda.Stream()
    bufs = [torch.zeros(len(SHAPES), dtype=torch.float32).pin_memory() for _ in range(2)]
    events = [torch.cuda.Event() for _ in range(2)]
    expect = []
    with torch.cuda.stream(stream):
        for k, h in enumerate((0.1, 0.1, 0.05, 0.05)):
            run.set_grads(inp.grads(k))
            run.opt.step(h, ptrs=run.ptrs, stream=stream)
            run.opt.enqueue_denominators(bufs[k % 2], stream)
            events[k % 2].record(stream)
            if k > 0:
                events[(k - 1) % 2].synchronize()
                got = bufs[(k - 1) % 2].numpy().copy()
                assert np.array_equal(got, expect[-1])
            stream.synchronize()
            sync = run.opt.read_denominators(stream)
            F = run.factors()
            for t, (m, n) in enumerate(SHAPES):
                if n == 0:
                    assert sync[t] == 0.0
                else:
                    assert sync[t] == pytest.approx(float(np.sum(F[t][0], dtype=np.float64)), rel=1e-5)
            expect.append(sync)
    events[1].synchronize()
    assert np.array_equal(bufs[1].numpy(), expect[-1])
    with pytest.raises(ValueError):
        run.opt.enqueue_denominators(torch.zeros(len(SHAPES)))     # not page-locked
    # Through the C ABI, pageable host memory takes the copy path.
    pageable = np.full(len(SHAPES), -1.0, np.float32)
    assert rikfad.lib().rikfad_enqueue_denominators(run.opt.handle, pageable.ctypes.data, None) == rikfad.OK
    torch.cuda.synchronize()
    assert np.array_equal(pageable, expect[-1])
    run.close()


def test_host_pointers_are_checked_before_any_launch():
    """A changed pointer is checked on the host: pageable host memory for a
    gradient either works in place (a device that reads pageable memory
    through the host's page tables, as GB300 does) and gives bitwise the
    step of a device copy, or is refused with RIKFAD_ERR_ARG before any
    kernel runs; the handle stays usable either way."""
    inp, run_d = _run()
    _, run_h = _run()
    g = inp.grads(0)
    run_d.set_grads(g)
    run_h.set_grads(g)
    pageable = [np.ascontiguousarray(torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy())
                for a in g]
    ptrs = [a.ctypes.data for a in pageable]
    try:
        run_h.opt.step(0.1, run_h.x, ptrs, run_h.p)
    except rikfad.RikfadError as e:
        assert e.code == rikfad.ERR_ARG and "pageable host memory" in str(e)
        run_h.step(0.1)                      # the device gradients still step
    run_d.step(0.1)
    torch.cuda.synchronize()
    for a, b in zip(run_d.x + run_d.p, run_h.x + run_h.p):
        assert torch.equal(a, b)
    run_d.close()
    run_h.close()
