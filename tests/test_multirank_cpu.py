"""The benchmark's multi-rank path on the CPU (gloo, world size 2): every rank has
its own independent restarts of the same DAG, the only collective is the max of the
ranks' times, and the whole-job throughput counts every rank's units."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        p, B, mu, sg = bench.workload(rank)
        ms = 10.0 + 5.0 * rank                      # a rank-dependent step time
        ms_max = bench.max_over_ranks(ms, world, dist, "cpu")
        value = bench.job_throughput(3, 100, B, world, ms_max)
        out[rank] = (p.V, p.E, B, float(mu[:, 0].sum()), float(sg.sum()), ms_max, value)
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    r0, r1 = out[0], out[1]
    # the same DAG on both ranks, independent initial states (different seeds)
    assert r0[:3] == r1[:3]
    assert r0[3] != r1[3]
    # the slowest rank's time on both ranks, and every rank's units counted
    assert r0[5] == r1[5] == 15.0
    assert r0[6] == r1[6] == pytest.approx(3 * 100 * r0[2] * world / 0.015)


def test_single_rank_needs_no_collective():
    import bench
    assert bench.max_over_ranks(12.5, 1) == 12.5
    assert bench.job_throughput(2, 10, 64, 1, 20.0) == pytest.approx(2 * 10 * 64 / 0.02)
