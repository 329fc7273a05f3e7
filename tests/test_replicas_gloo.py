"""Multi-process path of the benchmark on CPU (gloo, world size 2): the path shards as
independent replicas (no exchange step), so the only cross-rank operation is the
max-over-ranks of the timed region; whole-job throughput counts every rank's units over the
slowest rank's time.  The reference arm runs on rank 0 only."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local = [12.5, 40.0][rank]
        ms = bench.max_over_ranks(local, world, torch.device("cpu"))
        q.put((rank, ms, bench.replica_throughput(100, 3, world, ms / 1e3)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_replica_throughput_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, v in got:
        assert ms == 40.0                       # both ranks see the slowest rank's time
        assert v == pytest.approx(2 * 100 * 3 / 0.040)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(7.0, 1, torch.device("cpu")) == 7.0
    assert bench.replica_throughput(10, 2, 1, 0.5) == 40.0


def test_reference_arm_runs_on_rank_zero_only():
    class A:
        steps, warmup, gpus = 1, 0, 2
    assert bench.reference_arm(A(), 1, 2) is None
