"""Multi-rank host logic of bench.py on CPU (gloo, world size 2).

The path shards by frame: every rank voxelizes its own frames, and the only
exchange is the whole-job reduction after the timed regions (slowest rank's
time, sum of points). These tests run that reduction and the per-rank
workload split as two gloo processes; no GPU is touched.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, _ = bench.dist_env()
        assert (w, r) == (world, rank)
        # each rank's own frames: rank-dependent seeds, same shapes
        wl = bench.workload_for_rank(rank, frames=2)
        digest = float(np.asarray(wl.points[:1000], np.float64).sum())
        ms = [3.0, 5.0][rank]
        e2e = [0.2, 0.1][rank]
        pts = [100, 250][rank]
        ms_max, e2e_max, total = bench.aggregate_ranks(ms, e2e, pts, world, torch.device("cpu"))
        out[rank] = (ms_max, e2e_max, total, digest, wl.num_points)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_max_time_and_sum_points():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
        for p in procs:
            if p.is_alive():
                p.kill()
                pytest.fail("gloo rank did not finish")
            assert p.exitcode == 0
        r0, r1 = out[0], out[1]
    # every rank sees the slowest rank's times and the job's total points
    assert r0[:3] == r1[:3] == (5.0, 0.2, 350.0)
    # weak scaling: same per-rank size, different frames
    assert r0[4] == r1[4]
    assert r0[3] != r1[3]


def test_single_rank_aggregate_is_identity():
    import bench
    assert bench.aggregate_ranks(4.0, 0.5, 123, 1, torch.device("cpu")) == (4.0, 0.5, 123.0)
