"""Host logic of bench.py's multi-GPU mode (independent replicas, one per
rank): the job time is the slowest rank's and the value counts every rank's
units.  Runs as two gloo ranks on the CPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert bench.dist_env() == (rank, world, rank)
        ms_local = 10.0 + 5.0 * rank            # rank 1 is the slow one
        units_local = 1e9 * (rank + 1)
        ms, value = bench.aggregate(ms_local, units_local, dist)
        dist.barrier()
        out[rank] = (ms, value)
    finally:
        dist.destroy_process_group()


def test_replicas_aggregate_two_ranks():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, join=True,
                       start_method="spawn")
    for r in range(world):
        ms, value = out[r]
        assert ms == 15.0                              # max over ranks
        assert value == pytest.approx(3e9 / 0.015)    # all ranks' units / slowest time


def test_aggregate_single_process():
    sys.path.insert(0, ROOT)
    import bench
    ms, v = bench.aggregate(20.0, 4e9)
    assert ms == 20.0 and v == pytest.approx(2e11)
