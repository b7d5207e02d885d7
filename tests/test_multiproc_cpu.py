"""Multi-process host logic on CPU: the benchmark's replica aggregation.

Each rank runs an independent replica of the path; the reported value is the
sum of the ranks' decisions over the slowest rank's time.  Two gloo ranks on
127.0.0.1 check that reduction (max of seconds, sum of units) and the
environment parsing the benchmark uses under torchrun.
"""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    env = bench.dist_env()
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        secs, units = bench.aggregate(1.5 + rank, 1000.0 * (rank + 1), dist)
        out[rank] = (env, secs, units)
    finally:
        dist.destroy_process_group()


def test_replica_aggregation_two_gloo_ranks():
    world = 2
    port = _free_port()
    with mp.get_context("spawn").Manager() as m:  # no fork of a threaded process
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        env, secs, units = res[rank]
        assert secs == pytest.approx(2.5)      # slowest rank
        assert units == pytest.approx(3000.0)  # all ranks' decisions
        assert env[0] == world and env[1] == rank


def test_aggregate_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate(0.25, 77.0, None) == (0.25, 77.0)
