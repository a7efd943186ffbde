#!/usr/bin/env python
"""Benchmark of the R-iKFAD optimiser step on GB300.

One step = one R-iKFAD update (BACD splitting: kick, drift, symmetric rank-1
friction, damping) over every tensor of a GPT2-S-shaped parameter set
(196 tensors, 124,439,808 parameters; fp32 parameters and momenta, bf16
gradients), i.e. one fused step kernel plus one factor-finalise kernel.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  With N > 1 (launched by torchrun) every rank
runs its own replica of the step (the update has no exchange step); the
reported value is the total over ranks divided by the slowest rank's time.
"""
import argparse
import datetime
import hashlib
import json
import math
import os
import re
import shutil
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "R-iKFAD step Gparams/s and HBM GB/s vs peak, GPT2-S param set, 1 GB300"
UNIT = "Gparams/s"
# The paper's GPT2-S R-iKFAD0 hyperparameters (optimised-hyperparameter table).
HP = dict(alpha=0.0579, mu=1.3637e-6, gamma=0.0, eps_stab=1e-16)
STEP = 0.0918
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0      # GB300 HBM3e, nominal
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "rikfad_step_kernel__gpt2s.md")
KERNEL_SOURCES = ["paper_2609_30342_gb300/csrc/rikfad_kernels.cuh",
                  "paper_2609_30342_gb300/csrc/rikfad_plan.hpp",
                  "paper_2609_30342_gb300/csrc/rikfad_planner.cpp"]


# ------------------------------------------------------------ workloads

def workload(name):
    from paper_2609_30342_gb300 import workloads as W
    if name == "gpt2s":
        named = W.gpt2_small()
        desc = ("GPT2-S parameter set: 12 layers, width 768, vocab 50257 (tied), ctx 1024, "
                "separate q/k/v; 74 matrices + 122 vectors")
        seed = 3
    elif name in ("gpt2m", "gpt2xl"):
        layers, width = (24, 1024) if name == "gpt2m" else (48, 1600)
        named = W.gpt2_shapes(layers, width, 50257, 1024)
        desc = ("GPT2-%s-shaped parameter set: %d layers, width %d, vocab 50257 (tied), ctx 1024, "
                "separate q/k/v" % ("M" if name == "gpt2m" else "XL", layers, width))
        seed = 5
    elif name == "nano":
        named = W.gpt2_nano()
        desc = "GPT2-Nano-shaped parameter set: 6 layers, width 384, vocab 50304, ctx 256"
        seed = 2
    elif name.startswith("sweep"):
        i = int(name[5:] or 0)
        shp = W.SWEEP_SHAPES[i]
        named = [("W", shp)]
        desc = "single %d x %d matrix" % shp
        seed = 4
    else:
        raise SystemExit("unknown workload %r" % name)
    return named, desc, seed


def algorithmic_bytes(shapes, grad_bytes, method="rikfad"):
    """Compulsory HBM bytes of one step: every matrix element reads the
    gradient, X and P and writes X and P (grad + 16 bytes); every vector
    element also reads and writes its friction (grad + 24 bytes).  Under
    full-friction iKFAD every element is a vector element."""
    from paper_2609_30342_gb300 import workloads as W
    N, _, _, one_d = W.count(shapes)
    if method in ("ikfad", "ikfad_shadow"):
        return N * (grad_bytes + 24)
    return (N - one_d) * (grad_bytes + 16) + one_d * (grad_bytes + 24)


# ------------------------------------------------------- distributed glue

def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def init_dist(world, backend):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value, world, device="cpu"):
    """Maximum of a float over all ranks (identity when world == 1)."""
    if world == 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(units_per_rank, seconds_max, world):
    """Whole-job throughput: units processed by all ranks / slowest rank's time."""
    return units_per_rank * world / seconds_max


# ------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,timestamp")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id, period_ms=100):
        self.gpu_id = gpu_id
        self.period_ms = period_ms
        self.proc = None
        self.path = None
        self.err = None

    def start(self):
        smi = shutil.which("nvidia-smi")
        if smi is None:
            self.err = "nvidia-smi not found"
            return
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        cmd = [smi, "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
               "-lms", str(self.period_ms)]
        if self.gpu_id is not None:
            cmd += ["-i", str(self.gpu_id)]
        self.out = open(self.path, "w")
        self.proc = subprocess.Popen(cmd, stdout=self.out, stderr=subprocess.DEVNULL)

    def stop(self, window=None):
        """Stop sampling; summarise the samples taken within ``window`` (a
        (start, end) pair of time.time() values) if given."""
        if self.proc is None:
            return {"unavailable": self.err or "not started"}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        lines = open(self.path).read().strip().splitlines()
        os.unlink(self.path)
        sm, mx, pw, reasons = [], [], [], set()
        total = 0
        for ln in lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            total += 1
            if window is not None:
                try:
                    ts = datetime.datetime.strptime(f[9], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                except ValueError:
                    continue
                if not window[0] <= ts <= window[1]:
                    continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
                pw.append(float(f[3]))
            except ValueError:
                continue
            for name, val in zip(self.REASONS, f[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "samples_total": total}
        out = {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)),
               "reasons": sorted(reasons), "samples": len(sm), "power_w_max": float(max(pw)),
               "power_w_median": float(np.median(pw)), "sm_mhz_min": float(min(sm))}
        if window is not None:
            out["window_s"] = round(window[1] - window[0], 3)
            out["samples_total"] = total
        return out


# ------------------------------------------------------------ peaks & ncu

def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_digest():
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic():
    """DRAM bytes per launch of the step kernel from the committed ncu summary,
    or None if there is none or the kernel changed since it was taken."""
    try:
        text = open(PROFILE_SUMMARY).read()
    except OSError:
        return None
    m_sha = re.search(r"kernel_source_digest:\s*([0-9a-f]+)", text)
    m_b = re.search(r"dram_bytes_per_launch_gpt2s:\s*([0-9.eE+]+)", text)
    if not (m_sha and m_b) or m_sha.group(1) != kernel_source_digest():
        return None
    return float(m_b.group(1))


# ------------------------------------------------------------ oracle (CPU)

def oracle_sample(named, seed, budget_s):
    """Pick the largest sample of the workload that the oracle steps through
    within budget_s (one step), and the inputs for it."""
    from paper_2609_30342_gb300 import workloads as W
    import oracle
    names = [n for n, _ in named]
    cands = [("blocks h0-h1", lambda n: n.startswith("h0.") or n.startswith("h1.")),
             ("block h0", lambda n: n.startswith("h0.")),
             ("block h0 attention", lambda n: n.startswith("h0.attn.")),
             ("h0.attn.q", lambda n: n.startswith("h0.attn.q."))]
    if len(named) == 1:
        cands = [("whole workload", lambda n: True)]
    calib = [i for i, n in enumerate(names) if cands[-1][1](n)] or [0]
    shapes = [named[i][1] for i in calib]
    inp = W.ModelInputs(shapes, seed=seed)
    st = oracle.ModelState(shapes, inp.X, inp.P)
    g = [a.astype(np.float64) for a in inp.grads(0)]
    t0 = time.perf_counter()
    st.step(g, STEP, oracle.HParams(**HP))
    per_param = (time.perf_counter() - t0) / max(W.count(shapes)[0], 1)
    for label, pred in cands:
        idx = [i for i, n in enumerate(names) if pred(n)]
        n_par = W.count([named[i][1] for i in idx])[0]
        if n_par * per_param <= budget_s or label == cands[-1][0]:
            return label, idx
    return cands[-1][0], calib


def time_oracle(named, seed, idx, steps, warmup):
    """Seconds per oracle step over the tensors ``idx`` (float64, 1 thread)."""
    from paper_2609_30342_gb300 import workloads as W
    import oracle
    shapes = [named[i][1] for i in idx]
    inp = W.ModelInputs(shapes, seed=seed)
    st = oracle.ModelState(shapes, inp.X, inp.P)
    g = [a.astype(np.float64) for a in inp.grads(0)]
    hp = oracle.HParams(**HP)
    for _ in range(warmup):
        st.step(g, STEP, hp)
    t0 = time.perf_counter()
    for _ in range(steps):
        st.step(g, STEP, hp)
    return (time.perf_counter() - t0) / steps, W.count(shapes)[0]


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for ln in open("/proc/cpuinfo"):
            if ln.startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def _oracle_worker(args):
    """Worker of the all-cores baseline: step this worker's tensors ``steps``
    times with the unchanged oracle; returns (params, seconds)."""
    named, seed, idx, steps = args
    sec, n_par = time_oracle(named, seed, idx, steps, 1)
    return n_par, sec * steps


def cpu_baseline_all_cores(named, seed, target_s=10.0):
    """The oracle, unchanged, run by one spawned process per core, each
    stepping its share of the tensors (tensors are independent); throughput
    = all parameters stepped / the slowest worker's time."""
    import multiprocessing as mp
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    names = [n for n, _ in named]
    # every transformer block (the token and position embeddings would leave
    # one worker with a third of the parameters)
    idx = [i for i, n in enumerate(names) if n.startswith("h")] or list(range(len(named)))
    from paper_2609_30342_gb300 import workloads as W
    sizes = {i: W.numel(named[i][1]) for i in idx}
    shares = [[] for _ in range(cores)]
    load = [0] * cores
    for i in sorted(idx, key=lambda i: -sizes[i]):
        w = load.index(min(load))
        shares[w].append(i)
        load[w] += sizes[i]
    shares = [sh for sh in shares if sh]
    per_step = max(load) / 0.08e9            # ~0.08 Gparams/s per core (float64 C oracle)
    steps = int(min(30, max(2, target_s / max(per_step, 1e-6))))
    ctx = mp.get_context("spawn")
    with ctx.Pool(len(shares)) as pool:
        res = pool.map(_oracle_worker, [(named, seed, sh, steps) for sh in shares])
    n_par = sum(r[0] for r in res)
    slowest = max(r[1] for r in res)
    return {"value": n_par * steps / slowest / 1e9, "unit": UNIT, "cores": len(shares),
            "sample": "all %d transformer blocks (%d tensors, %d params), %d steps of the float64 C "
                      "oracle, one spawned process per core, tensors balanced by size"
                      % (len([n for n in names if n.endswith("ln_1.weight")]), len(idx), n_par, steps)}


def cpu_baseline(named, seed, target_s=12.0):
    label, idx = oracle_sample(named, seed, budget_s=target_s / 3)
    sec1, n_par = time_oracle(named, seed, idx, 1, 0)
    reps = int(min(30, max(2, math.ceil(target_s / max(sec1, 1e-6)))))
    sec, n_par = time_oracle(named, seed, idx, reps, 0)
    nproc = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    out = {"value": n_par / sec / 1e9, "unit": UNIT, "cores": 1, "kind": "oracle",
           "sample": "%s of the workload (%d tensors, %d params), %d steps of the float64 C "
                     "oracle, single thread" % (label, len(idx), n_par, reps),
           "nproc": nproc, "cpu_model": cpu_model()}
    try:
        out["all_cores"] = cpu_baseline_all_cores(named, seed)
    except Exception as e:                      # the single-thread figure stands on its own
        out["all_cores"] = {"unavailable": "%s: %s" % (type(e).__name__, e)}
    return out


# ------------------------------------------------------------ our arm

def run_ours(args, rank, world, local_rank):
    import torch
    from paper_2609_30342_gb300 import rikfad
    from paper_2609_30342_gb300 import workloads as W

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    init_dist(world, "nccl")
    rikfad.lib()

    named, desc, seed = workload(args.workload)
    shapes = [s for _, s in named]
    N, mats, mn, one_d = W.count(shapes)
    inp = W.ModelInputs(shapes, seed=seed)
    grads = inp.grads(0)

    # Gradients live in one flat bf16 buffer (device) with a pinned host twin,
    # which the end-to-end run reads from.
    offs, total = [], 0
    for s in shapes:
        offs.append(total)
        total += -(-W.numel(s) // 8) * 8
    g_dev = torch.zeros(max(total, 1), dtype=torch.bfloat16, device=dev)
    g_host = torch.zeros(max(total, 1), dtype=torch.bfloat16).pin_memory()
    g_views = []
    for s, o, a in zip(shapes, offs, grads):
        n = W.numel(s)
        g_host[o:o + n].copy_(torch.from_numpy(a.ravel()).to(torch.bfloat16))
        g_views.append(g_dev[o:o + n].view(W.array_shape(s)))
    g_dev.copy_(g_host)
    x = [torch.from_numpy(a).to(dev) for a in inp.X]
    p = [torch.zeros(W.array_shape(s), dtype=torch.float32, device=dev) for s in shapes]
    del inp, grads

    hp = dict(HP, gamma=args.gamma)
    opt = rikfad.RIKFAD(shapes, grad_dtype="bf16", method=args.method, **hp)
    ptrs = opt.pack(x, g_views, p)
    stream = torch.cuda.current_stream(dev)
    alg_bytes = algorithmic_bytes(shapes, 2, args.method)
    # --vary-h alternates the step size, so every step applies a pending
    # factor of a different h (two exponentials per matrix element).
    hs = (STEP, 0.9 * STEP) if args.vary_h else (STEP, STEP)
    # --canonical: every step is followed by the materialise pass, so the
    # stored momentum is always the paper's P_{n+1} (8 more bytes per matrix
    # element: P read and written once more).
    p_arr = rikfad.pointer_array(p)
    if args.canonical:
        alg_bytes += 8 * (N - one_d)

    def do_step(i, pt):
        opt.step(hs[i % 2], ptrs=pt, stream=stream)
        if args.canonical:
            opt.materialize(p_arr, stream=stream)

    # NVTX ranges mark the phases (ncu --nvtx --nvtx-include "timed/" selects
    # the timed steps); one push and pop per phase or repeat, none per step.
    nvtx = torch.cuda.nvtx
    w0 = torch.cuda.Event(enable_timing=True)
    w1 = torch.cuda.Event(enable_timing=True)
    nvtx.range_push("warmup")
    w0.record(stream)
    for i in range(args.warmup):
        do_step(i, ptrs)
    w1.record(stream)
    torch.cuda.synchronize(dev)
    nvtx.range_pop()
    warm_ms = w0.elapsed_time(w1) / max(args.warmup, 1)

    # ---- device-timed region: inputs resident in HBM (2.24 GB > 129 MB L2).
    # The K steps are timed R times back to back, each repeat exactly K steps
    # between a barrier and a device synchronisation on both sides; R is
    # chosen so the repeats keep the GPU loaded for about a second, long
    # enough for the clock sampler to see the load; the reported time per
    # step is the median over the repeats.
    reps = args.repeats or int(min(2000, max(3, math.ceil(1000.0 / max(warm_ms * args.steps, 1e-3)))))
    reps = int(max_over_ranks(reps, world, dev))
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        uuid = None
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.4)       # nvidia-smi starts before the load does
    rep_ms = []
    t_win0 = time.time()
    for r in range(reps):
        ev0 = torch.cuda.Event(enable_timing=True)
        ev1 = torch.cuda.Event(enable_timing=True)
        barrier(world)
        torch.cuda.synchronize(dev)
        nvtx.range_push("timed")
        ev0.record(stream)
        for i in range(args.steps):
            do_step(i, ptrs)
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        nvtx.range_pop()
        barrier(world)
        rep_ms.append(max_over_ranks(ev0.elapsed_time(ev1), world, dev))
    t_win1 = time.time()
    clocks = sampler.stop(window=(t_win0, t_win1))
    # Kernel durations: the same steps again with CUDA events around each
    # launch (events between the kernels stop them from overlapping, so this
    # pass is kept out of the headline timing above).
    nvtx.range_push("kernel events")
    opt.profile_enable(True)
    for i in range(args.steps):
        do_step(i, ptrs)
    torch.cuda.synchronize(dev)
    nvtx.range_pop()
    step_ms, fin_ms, nrec = opt.profile_read()
    opt.profile_enable(False)
    opt.check_finite(stream)          # the timed steps produced finite factors
    ms_max = float(np.median(rep_ms))
    ms_per_step = ms_max / args.steps
    value = aggregate(N, ms_per_step / 1e3, world) / 1e9
    kern_ms = step_ms / max(nrec, 1)
    peak, peak_src = hbm_peak()
    kern_bytes = algorithmic_bytes(shapes, 2, args.method)     # the step kernel's own bytes
    achieved = kern_bytes / (kern_ms / 1e3) / 1e9
    traffic = ncu_traffic() if args.workload == "gpt2s" and args.method == "rikfad" else None

    # ---- end to end: every step brings its bf16 gradients in from pinned host
    # memory and reads the friction denominators (one float per tensor) back.
    # The read-back is pipelined as in a training loop that logs a metric:
    # step i's values land in one of two page-locked buffers and the host
    # reads them (and checks that they are finite) after enqueueing step i + 1.
    # The step kernel loads the gradients directly from the pinned host buffer
    # (zero-copy over the coherent CPU-GPU link); measured on GB300 this moves
    # them faster than staging copies (one copy stream: ~120-180 GB/s, two or
    # more: ~205 GB/s, zero-copy loads: ~200 GB/s with no copy to overlap).
    host_views = [g_host[o:o + W.numel(s)].view(W.array_shape(s)) for s, o in zip(shapes, offs)]
    ptrs_host = opt.pack(x, host_views, p)
    # The same W untimed warm-up steps as the device-timed leg: the first
    # kernel to touch the pinned buffer pays a one-time mapping cost (7.9 ms
    # against 1.2 ms in the ncu launch list).
    den_bufs = [torch.zeros(len(shapes), dtype=torch.float32).pin_memory() for _ in range(2)]
    den_ready = [torch.cuda.Event() for _ in range(2)]

    def e2e_steps(n):
        bad = 0
        for i in range(n):
            do_step(i, ptrs_host)
            opt.enqueue_denominators(den_bufs[i % 2], stream)
            den_ready[i % 2].record(stream)
            if i > 0:
                den_ready[(i - 1) % 2].synchronize()
                bad += int(not torch.isfinite(den_bufs[(i - 1) % 2]).all())
        den_ready[(n - 1) % 2].synchronize()
        return bad + int(not torch.isfinite(den_bufs[(n - 1) % 2]).all())

    e2e_steps(args.warmup)
    barrier(world)
    torch.cuda.synchronize(dev)
    nvtx.range_push("end to end")
    t0 = time.perf_counter()
    e2e_bad = e2e_steps(args.steps)
    torch.cuda.synchronize(dev)
    e2e_s = max_over_ranks(time.perf_counter() - t0, world, dev)
    if e2e_bad:
        raise RuntimeError("non-finite friction denominators in the end-to-end leg")
    nvtx.range_pop()
    barrier(world)
    e2e = {"value": aggregate(N, e2e_s / args.steps, world) / 1e9, "unit": UNIT,
           "h2d_bytes_per_step": int(sum(v.numel() for v in host_views) * 2),
           "d2h_bytes_per_step": 4 * len(shapes),
           "h2d_path": "step kernel loads the bf16 gradients from pinned host memory (zero-copy)",
           "d2h_path": "denominators copied to page-locked memory every step; the host reads step i's "
                       "after enqueueing step i + 1"}

    diag = None
    if args.diagnostics and args.method == "ikfad_shadow":
        # Per-layer comparison of the paper's Section 4.4 on the final state:
        # error of the shadow rank-1 friction vs the Eckart-Young floor, and
        # the stable rank of the element-wise friction.
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        rows = []
        for t, (m, n) in enumerate(shapes):
            if n and m:
                rows.append(opt.friction_diagnostics(t, stream=stream))
        dt = time.perf_counter() - t0
        gaps = [100.0 * (r[0] - r[1]) for r in rows]
        diag = {"layers": len(rows), "seconds": round(dt, 3),
                "median_gap_pp": round(float(np.median(gaps)), 4),
                "max_gap_pp": round(float(np.max(gaps)), 4),
                "stable_rank_min_max": [round(min(r[2] for r in rows), 4),
                                        round(max(r[2] for r in rows), 4)],
                "mean_power_iterations": round(float(np.mean([r[5] for r in rows])), 1)}

    launches = opt.launches_per_step() * args.steps * reps
    state = opt.state_bytes(True)
    full_state = 8 * N
    opt.close()

    if rank != 0:
        return None
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "repeats": {"count": reps, "ms_per_step_median": round(ms_per_step, 5),
                    "ms_per_step_min": round(min(rep_ms) / args.steps, 5),
                    "ms_per_step_max": round(max(rep_ms) / args.steps, 5),
                    "timing": "the K steps timed R times back to back (each between a barrier and "
                              "a device synchronisation), median reported"},
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded): X ~ N(0, 0.02^2) fp32, P = 0 fp32, grad ~ N(0, 1e-3^2) bf16",
        "config": {"workload": desc, "params": N, "tensors": len(shapes), "matrices": mats,
                   "vector_elements": one_d, "grad_dtype": "bf16", "state_dtype": "f32",
                   "hyperparameters": dict(hp, h=STEP), "method": args.method,
                   "step_size": "alternating %g / %g" % hs if args.vary_h else "constant",
                   "momentum_form": "canonical after every step (3-pass)" if args.canonical
                                    else "deferred (P^(1) stored)",
                   "l2": "no flush: %.2f GB of inputs per step > 129 MB L2" % (alg_bytes / 1e9),
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "hbm_gbs_step": round(alg_bytes / (ms_per_step / 1e3) / 1e9, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                     "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": traffic,
                     "kernel": "rikfad_step_kernel", "peak_source": peak_src,
                     "peak_nominal": NOMINAL_HBM_GBS,
                     "frac_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                     "algorithmic_bytes_per_launch": kern_bytes,
                     "kernel_ms": round(kern_ms, 5),
                     "finalize_kernel_ms": round(fin_ms / max(nrec, 1), 5),
                     "timing": "CUDA events around every launch on the launching stream, "
                               "over a second pass of the same %d steps" % args.steps},
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": clocks,
        "state_bytes": {args.method: state, "full_friction_ikfad": full_state,
                        "ratio": round(full_state / state, 3)},
    }
    if diag is not None:
        line["friction_diagnostics"] = diag
    if world == 1 and not args.no_cpu_baseline and args.method == "rikfad":
        line["cpu_baseline"] = cpu_baseline(named, seed)
    return line


# ------------------------------------------------------------ NEXT-4: dense quadratics

G0_M, G0_N, G0_BATCH, G0_STEPS_PER_CALL, G0_H = 6, 5, 65536, 1000, 0.02
G0_HP = dict(alpha=1.0, mu=1.0, gamma=0.0, eps_stab=0.1)
G0_METRIC = ("batched BACD integration of R-iKFAD on dense quadratics (Table tab:g0_slopes "
             "problem), 6x5 systems, system-steps/s, 1 GB300")
G0_UNIT = "Gsystem-steps/s"
# FP32 peak of the SMs: 152 SMs x 128 FP32 lanes x 2 flop per FMA x 2.07 GHz.
FP32_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def g0_flops(m, n):
    """Algorithmic flops of one BACD step of one m x n system (an exponential
    counts as one): A vec(X) 2 d^2; per element the friction R^_i C_j and its
    scale (2), two damping exponentials and their products (4), kick (2),
    drift (2), square (1), row and column sums (2); per row the division
    R_i / (s + eps) and its share of s (2) and the filter (3); per column the
    filter (3)."""
    d = m * n
    return 2 * d * d + 13 * d + 5 * m + 3 * n


def g0_oracle_rate(budget_s, steps_hint=2000):
    """System-steps/s of the float64 C oracle on single 6x5 systems (one thread)."""
    import oracle
    from paper_2609_30342_gb300 import workloads as W
    A, X, P = W.dense_quadratic_instance(G0_M, G0_N, 1)
    hp = oracle.HParams(**G0_HP)
    t0 = time.perf_counter()
    oracle.dense_quadratic_run(A, X.copy(), P.copy(), np.zeros(G0_M), np.zeros(G0_N), G0_H, hp,
                               steps_hint, [steps_hint])
    per = (time.perf_counter() - t0) / steps_hint
    steps = int(max(steps_hint, min(5e7, budget_s / max(per, 1e-9))))
    t0 = time.perf_counter()
    oracle.dense_quadratic_run(A, X.copy(), P.copy(), np.zeros(G0_M), np.zeros(G0_N), G0_H, hp, steps,
                               [steps])
    sec = time.perf_counter() - t0
    return steps / sec, steps, sec


def run_g0(args, rank, world, local_rank):
    import torch
    from paper_2609_30342_gb300 import rikfad
    from paper_2609_30342_gb300 import workloads as W

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    init_dist(world, "nccl")
    rikfad.lib()
    m, n, B, K = G0_M, G0_N, G0_BATCH, G0_STEPS_PER_CALL
    # 64 seeded instances tiled over the batch (instance generation is host
    # numpy); each system is integrated independently.
    A64, X64, P64 = W.dense_quadratic_batch(m, n, range(1000 * rank, 1000 * rank + 64))
    reps = B // 64
    A_h = torch.from_numpy(np.tile(A64, (reps, 1, 1))).pin_memory()
    X_h = torch.from_numpy(np.tile(X64, (reps, 1, 1))).pin_memory()
    P_h = torch.from_numpy(np.tile(P64, (reps, 1, 1))).pin_memory()
    R_h = torch.zeros(B, m).pin_memory()
    C_h = torch.zeros(B, n).pin_memory()
    A, X, P, R, C = (t.to(dev) for t in (A_h, X_h, P_h, R_h, C_h))
    rec = torch.tensor([K], dtype=torch.int64, device=dev)
    E = torch.zeros(1, B, device=dev)
    hp = G0_HP
    stream = torch.cuda.current_stream(dev)

    def call(a, x, p, r, c, e, nsteps=K):
        rikfad.quadratic_run(a, x, p, r, c, G0_H, hp["alpha"], hp["mu"], hp["gamma"], hp["eps_stab"],
                             nsteps, rec, e, stream=stream)

    for _ in range(args.warmup):
        call(A, X, P, R, C, E)
    torch.cuda.synchronize(dev)
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        uuid = None
    sampler = ClockSampler(uuid)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    sampler.start()
    time.sleep(0.4)
    t_win0 = time.time()
    ev0.record(stream)
    for _ in range(args.steps):
        call(A, X, P, R, C, E)
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    t_win1 = time.time()
    barrier(world)
    clocks = sampler.stop(window=(t_win0, t_win1))
    ms_total = ev0.elapsed_time(ev1)
    ms_max = max_over_ranks(ms_total, world, dev)
    ms_per_call = ms_max / args.steps
    value = aggregate(B * K, ms_per_call / 1e3, world) / 1e9
    flops = g0_flops(m, n) * B * K
    achieved = flops / (ms_total / args.steps / 1e3) / 1e12

    # End to end through the same call with host buffers: every call copies
    # A, X, P, R, C in from pinned host memory and X, P, R, C and the energy
    # back out.
    outs = [torch.empty_like(t).pin_memory() for t in (X_h, P_h, R_h, C_h)]
    E_h = torch.empty(1, B).pin_memory()

    def e2e_call():
        for d_t, h_t in zip((A, X, P, R, C), (A_h, X_h, P_h, R_h, C_h)):
            d_t.copy_(h_t, non_blocking=True)
        call(A, X, P, R, C, E)
        for h_t, d_t in zip(outs + [E_h], (X, P, R, C, E)):
            h_t.copy_(d_t, non_blocking=True)

    for _ in range(args.warmup):        # untimed, as for the device-timed leg
        e2e_call()
    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_call()
    torch.cuda.synchronize(dev)
    e2e_s = max_over_ranks(time.perf_counter() - t0, world, dev)
    h2d = sum(t.numel() * 4 for t in (A_h, X_h, P_h, R_h, C_h))
    d2h = sum(t.numel() * 4 for t in outs) + E_h.numel() * 4
    e2e = {"value": round(aggregate(B * K, e2e_s / args.steps, world) / 1e9, 4), "unit": G0_UNIT,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    # Latency of one step of a single system (what bounds a long run such as
    # the paper's t = 1e7 table): 2^16 steps of one system, per table size.
    lat = {}
    for (mm, nn) in ((2, 2), (4, 3), (6, 5)):
        a1, x1, p1 = (torch.from_numpy(v).to(dev) for v in W.dense_quadratic_batch(mm, nn, [1]))
        r1, c1 = torch.zeros(1, mm, device=dev), torch.zeros(1, nn, device=dev)
        rikfad.quadratic_run(a1, x1, p1, r1, c1, G0_H, 1.0, 1.0, 0.0, 0.1, 1000, stream=stream)
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        rikfad.quadratic_run(a1, x1, p1, r1, c1, G0_H, 1.0, 1.0, 0.0, 0.1, 1 << 16, stream=stream)
        s1.record(stream)
        torch.cuda.synchronize(dev)
        lat["%dx%d" % (mm, nn)] = round(s0.elapsed_time(s1) * 1e6 / (1 << 16), 1)

    if rank != 0:
        return None
    line = {
        "metric": G0_METRIC, "value": round(value, 4), "unit": G0_UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_call, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded): A = B B^T/d + 0.8 I, X(0) ~ N(0, 0.4^2), P(0) ~ N(0, 0.3^2), "
                "R(0) = C(0) = 0 (the paper's construction)",
        "config": {"workload": "%d systems of %d x %d, %d BACD steps per call (one bench step = "
                               "one call)" % (B, m, n, K),
                   "hyperparameters": dict(hp, h=G0_H),
                   "l2": "no flush: A alone is %.0f MB > 129 MB L2, read once per launch"
                         % (A_h.numel() * 4 / 1e6),
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "alu", "achieved": round(achieved, 3), "peak": round(FP32_PEAK_TFLOPS, 1),
                     "unit": "TFLOP/s", "frac": round(achieved / FP32_PEAK_TFLOPS, 4), "traffic": None,
                     "kernel": "rikfad_quadratic_kernel<8,8>",
                     "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 flop x 2.07 GHz",
                     "flops_per_system_step": g0_flops(m, n)},
        "e2e": e2e,
        "gpu_launches": args.steps,
        "clocks": clocks,
        "single_system_ns_per_step": lat,
    }
    if world == 1 and not args.no_cpu_baseline:
        rate, steps, sec = g0_oracle_rate(10.0)
        line["cpu_baseline"] = {"value": rate / 1e9, "unit": G0_UNIT, "cores": 1, "kind": "oracle",
                                "sample": "one 6x5 system, %d steps of the float64 C oracle "
                                          "(%.1f s), single thread" % (steps, sec)}
    return line


# ------------------------------------------------------------ reference arm

def run_reference(args, rank, world):
    """The oracle (plain float64 C, one thread) on a bounded sample of the
    same workload, timed per step on the host cores."""
    if rank != 0:
        return None
    if args.workload == "g0":
        budget = 150.0 / max(args.steps + args.warmup, 1)
        rate, steps, sec = g0_oracle_rate(budget)
        sample = "one 6x5 system, %d steps of the float64 C oracle per bench step, single thread" % steps
        value = rate / 1e9
        return {
            "impl": "reference", "metric": G0_METRIC, "value": value, "unit": G0_UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": G0_BATCH * G0_STEPS_PER_CALL / rate * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
            "config": {"workload": "%d systems of %d x %d, %d BACD steps per call"
                                   % (G0_BATCH, G0_M, G0_N, G0_STEPS_PER_CALL)},
            "cpu_baseline": {"value": value, "unit": G0_UNIT, "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": G0_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }
    named, desc, seed = workload(args.workload)
    budget = 150.0 / max(args.steps + args.warmup, 1)
    label, idx = oracle_sample(named, seed, budget_s=budget)
    sec, n_par = time_oracle(named, seed, idx, args.steps, args.warmup)
    value = n_par / sec / 1e9
    sample = ("%s of the workload (%d tensors, %d params) per step, float64 C oracle, single "
              "thread" % (label, len(idx), n_par))
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded)", "config": {"workload": desc},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="gpt2s",
                    help="gpt2s (default), nano, gpt2m, gpt2xl, sweep0..sweep3, or g0 (batched "
                         "BACD on the paper's dense quadratics)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--method", choices=("rikfad", "ikfad", "ikfad_shadow"), default="rikfad",
                    help="rikfad (default), full-friction ikfad, or ikfad with shadow R-iKFAD factors")
    ap.add_argument("--diagnostics", action="store_true",
                    help="with --method ikfad_shadow: per-layer friction diagnostics after timing")
    ap.add_argument("--gamma", type=float, default=HP["gamma"],
                    help="linear damping gamma (default 0, R-iKFAD0)")
    ap.add_argument("--canonical", action="store_true",
                    help="materialise P after every step (the 3-pass canonical form, 26 B per "
                         "matrix element)")
    ap.add_argument("--vary-h", action="store_true",
                    help="alternate the step size between h and 0.9 h")
    ap.add_argument("--repeats", type=int, default=0,
                    help="times the K timed steps are repeated (default: enough for ~1 s of load)")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    rank, world, local_rank = dist_env()
    if world != args.gpus:
        if world == 1 and args.gpus > 1:
            raise SystemExit("--gpus %d needs torchrun with %d processes" % (args.gpus, args.gpus))
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    elif args.workload == "g0":
        line = run_g0(args, rank, world, local_rank)
    else:
        line = run_ours(args, rank, world, local_rank)
    if line is not None:
        print(json.dumps(line), flush=True)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist
        if dist.is_initialized():
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
