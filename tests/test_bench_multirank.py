"""Host logic of bench.py's multi-GPU mode, run as gloo ranks on the CPU.

On several GPUs every replica is split by parameter range (one contiguous
range per rank) and the one exchange per round is an all-reduce of the ranks'
consensus-error shares.  Checked here: the ranges partition [0, P); ranks
that each run the oracle on their range, exchanging through bench.ce_exchange,
reproduce the single-process oracle (replicas bit for bit, the summed
consensus error to 1e-12 relative); the job's time is the slowest rank's and
its value counts every rank's units.
"""
import ctypes
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _init(rank, world, port):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    return dist


def _aggregate_main(rank, world, port, out):
    dist = _init(rank, world, port)
    import bench
    try:
        assert bench.dist_env() == (rank, world, rank)
        ms_local = 10.0 + 5.0 * rank            # rank 1 is the slow one
        units_local = 1e9 * (rank + 1)
        ms, value = bench.aggregate(ms_local, units_local, dist)
        dist.barrier()
        out[rank] = (ms, value)
    finally:
        dist.destroy_process_group()


def _spawn(fn, world, *args):
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(fn, args=(world, port, out) + args, nprocs=world, join=True, start_method="spawn")
    return dict(out)


def test_aggregate_two_ranks():
    out = _spawn(_aggregate_main, 2)
    for r in range(2):
        ms, value = out[r]
        assert ms == 15.0                              # max over ranks
        assert value == pytest.approx(3e9 / 0.015)    # all ranks' units / slowest time


def test_aggregate_single_process():
    import bench
    ms, v = bench.aggregate(20.0, 4e9)
    assert ms == 20.0 and v == pytest.approx(2e11)


@pytest.mark.parametrize("P", [124_439_808, 1_048_576, 20_000, 4097])
def test_shard_ranges_partition_the_parameters(P):
    import bench
    for world in range(1, 9):
        if -(-P // world) < 1:
            continue
        try:
            parts = [bench.shard_range(P, world, r) for r in range(world)]
        except ValueError:
            assert -(-P // 4096) < world      # fewer blocks of 4096 than ranks
            continue
        assert parts[0][0] == 0 and parts[-1][1] == P
        for (a, b), (c, d) in zip(parts, parts[1:]):
            assert b == c and a < b
        assert all(a % 4096 == 0 for a, _ in parts)


class _OracleRank:
    """Stands in for a rank's context: the oracle held on the rank's range,
    exposing the one call ce_exchange makes (the share copied to memory)."""

    def __init__(self, st):
        self.st = st

    def consensus_error_async(self, addr):
        ctypes.c_double.from_address(addr).value = self.st.consensus_error()


PB = dict(n_workers=8, n_params=20_000, topology="exp", seed=31, weights="metropolis", edge_prob=0.5,
          per_worker_h=True, lr=2e-3, noise_sigma=0.02)
ROUNDS = 4


def _problem():
    import oracle
    kw = dict(PB)
    return oracle.make_problem(kw.pop("n_workers"), kw.pop("n_params"), kw.pop("topology"), **kw)


def _ranges_main(rank, world, port, out):
    dist = _init(rank, world, port)
    import torch
    import bench
    import oracle
    try:
        orc = oracle.get("f32")
        p0, p1 = bench.shard_range(PB["n_params"], world, rank)
        st = orc.state(_problem(), np.arange(p0, p1, dtype=np.int64))
        Hi = orc.draw_local_steps(PB["seed"], PB["n_workers"], 4)
        ce = torch.zeros(ROUNDS, dtype=torch.float64)
        for k in range(ROUNDS):
            st.local_steps(0, Hi)
            st.gossip_round()
            bench.ce_exchange(dist, _OracleRank(st), ce, k)
        out[rank] = ((p0, p1), st.get_all("x"), ce.numpy().copy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_ranks_on_parameter_ranges_reproduce_one_process(world, orc32):
    out = _spawn(_ranges_main, world)
    st = orc32.state(_problem())
    Hi = orc32.draw_local_steps(PB["seed"], PB["n_workers"], 4)
    ces = []
    for _ in range(ROUNDS):
        st.local_steps(0, Hi)
        st.gossip_round()
        ces.append(st.consensus_error())
    x = st.get_all("x")
    for r in range(world):
        (p0, p1), xr, cer = out[r]
        np.testing.assert_array_equal(xr, x[:, p0:p1])
        np.testing.assert_allclose(cer, ces, rtol=1e-12)
    assert sum(out[r][0][1] - out[r][0][0] for r in range(world)) == PB["n_params"]
