"""Multi-process host logic of bench.py on CPU (gloo, world size 2): the batch is
replicated per rank with no data-path collective, the timed region's length is the max
over ranks, the throughput is the whole job's, and the reference arm runs on rank 0
only."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    from paper_2509_05512_gb300 import inputs
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r "measured" (r + 1) ms for 10 steps of a 2-unit step
        ms = bench.max_over_ranks(float(rank + 1), dist, torch, "cpu")
        value = bench.job_throughput(2.0, 10, world, ms)

        class Args:
            workload = "c1"
            steps = 1
            warmup = 0
        # non-zero ranks leave the reference arm at once, with no work and no output
        ref_rc = bench.reference_arm(Args, rank, world, inputs) if rank != 0 else None
        dist.barrier()
        q.put((rank, ms, value, ref_rc))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_time_is_max_and_value_is_whole_job():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        rank, ms, value, ref_rc = q.get(timeout=120)
        res[rank] = (ms, value, ref_rc)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # both ranks agree on the slowest rank's 2 ms
    assert res[0][0] == res[1][0] == 2.0
    # 2 units/step * 10 steps * 2 ranks / 2 ms
    assert res[0][1] == pytest.approx(2.0 * 10 * 2 / 2e-3)
    assert res[1][2] == 0


def test_single_process_helpers_without_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, None, torch, "cpu") == 3.5
    assert bench.job_throughput(1.0, 4, 1, 2.0) == pytest.approx(2000.0)
