"""bench.py's multi-rank plumbing on the CPU with gloo, world size 2: the
max-over-ranks timing, the barrier, the whole-job aggregate, and the
reference arm printing from rank 0 only."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    assert bench.dist_env() == (rank, world, rank)
    t = bench.max_over_ranks(1.5 * (rank + 1), world)
    bench.barrier(world)
    agg = bench.aggregate(100.0, t, world)

    class Args:
        workload = "gpt2s"
        steps = 3
        warmup = 3
    ref = bench.run_reference(Args, rank, world) if rank != 0 else "skipped"
    q.put((rank, t, agg, ref))
    dist.destroy_process_group()


def test_max_over_ranks_and_aggregate_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    for rank, t, agg, ref in out:
        assert t == pytest.approx(3.0)          # slowest rank's time
        assert agg == pytest.approx(200.0 / 3.0)  # all ranks' units / slowest time
    assert out[1][3] is None                    # only rank 0 runs the reference arm


def test_single_process_helpers():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(2.5, 1) == 2.5
    assert bench.aggregate(10.0, 2.0, 1) == 5.0
    from paper_2609_30342_gb300 import workloads
    shapes = [s for _, s in workloads.gpt2_small()]
    assert bench.algorithmic_bytes(shapes, 2) == 124318464 * 18 + 121344 * 26 == 2240887296
