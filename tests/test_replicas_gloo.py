"""The N > 1 path of the benchmark, on CPU with two gloo ranks: each rank
quantizes its own replica of the block (no data-path collective), the job
time is the slowest rank's, and the throughput counts every rank's columns.
The reference arm runs on rank 0 only."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = [120.0, 80.0][rank]
        ms = bench.max_over_ranks(local_ms, dist, "cpu")
        dist.barrier()
        q.put((rank, ms, bench.job_throughput(10240, 5, world, ms)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_and_count_every_replica():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[1] for o in out] == [120.0, 120.0]
    # 2 replicas x 5 steps x 10240 columns in 120 ms
    assert out[0][2] == pytest.approx(2 * 5 * 10240 / 0.120)


def test_single_rank_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(42.0) == 42.0
    assert bench.job_throughput(10240, 10, 1, 113.2) == pytest.approx(10240 * 10 / 0.1132)


def test_reference_arm_runs_on_rank_zero_only():
    sys.path.insert(0, ROOT)
    import argparse
    import bench
    import synth
    args = argparse.Namespace(steps=1, warmup=0)
    assert bench.reference_arm(args, synth.workloads()["qwen3-0.6b"], 1, 2) is None
