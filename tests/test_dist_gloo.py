"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): each rank
owns its own parameter shard (distinct inputs, same push sequence), timings
are reduced with a max over ranks, and the whole-job value counts every
rank's units."""

import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    from paper_1601_04033_gb300 import streams
    w_env, r_env, l_env = bench.dist_env()
    assert (w_env, r_env, l_env) == (world, rank, rank)
    bench.init_dist(world, "gloo")
    w = streams.WORKLOADS["fasgd-25m-k8"]
    wr = bench.shard_workload(w, rank)
    pool = streams.gradient_pool(wr, 64, 2)
    ps = streams.push_stream(w, 32, 8)
    local_ms = 10.0 + 5.0 * rank
    bench.barrier(world)
    m = bench.max_over_ranks(local_ms, world)
    gathered = [None] * world
    dist.all_gather_object(gathered, (pool.tobytes(), ps.j.tobytes(), ps.client.tobytes(), m))
    out[rank] = gathered
    dist.destroy_process_group()


def test_two_ranks_shard_and_max():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, out), nprocs=2, join=True, start_method="spawn")
    g0, g1 = out[0], out[1]
    assert g0 == g1
    (pool0, j0, c0, m0), (pool1, j1, c1, m1) = g0
    assert pool0 != pool1                 # distinct shards of the parameter vector
    assert j0 == j1 and c0 == c1          # the same pushes reach every shard
    assert m0 == m1 == 15.0               # the slowest rank's time


def test_single_rank_helpers_need_no_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    bench.barrier(1)
    from paper_1601_04033_gb300 import streams
    w = streams.WORKLOADS["fasgd-25m-k8"]
    assert bench.shard_workload(w, 0) is w
    assert bench.algorithmic_bytes_dense(25_000_000, 8, True) == 1_600_000_000
    assert bench.algorithmic_bytes_dense(10, 4, False) == 10 * (8 + 16)
