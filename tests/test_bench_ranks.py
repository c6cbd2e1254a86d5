"""The multi-rank path of bench.py on the host (gloo, world size 2): the
job's time is the slowest rank's, the whole-job throughput counts every
rank's units, and every rank runs its own seeded replica of the workload
(the batch's sequences are independent, so the path shards with no
data-path collective)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        ms = [3.0, 5.0][rank]  # this rank's own timed region
        job_ms = bench.max_over_ranks(ms, world, torch)
        rate = bench.job_rate(world, 1000 * 25, job_ms)
        c = bench.workload(1, rank, 0)  # config 1: small enough for the host
        out.put((rank, job_ms, rate, c.q[:8].tobytes(), c.cache_len.tolist()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_time_rate_and_replicas():
    world = 2
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()  # both ranks rendezvous on it
    procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        rank, job_ms, rate, q8, cl = out.get(timeout=120)
        res[rank] = (job_ms, rate, q8, cl)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(world):
        job_ms, rate, _, _ = res[r]
        assert job_ms == 5.0  # the slowest rank
        assert rate == pytest.approx(world * 1000 * 25 / 5e-3)
    # replicas: the same workload shape with each rank's own draws
    assert res[0][3] == res[1][3]
    assert res[0][2] != res[1][2]


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(4.0, 1, torch) == 4.0
    assert bench.job_rate(1, 50, 2.0) == pytest.approx(25000.0)
    a, b = bench.workload(1, 0, 0), bench.workload(1, 0, 1)
    assert not np.array_equal(a.q, b.q)  # the two alternating input sets differ
