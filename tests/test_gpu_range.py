"""Contexts that hold a range of the parameters (gasloc_set_range).

Every step of Algorithm 1 acts on each parameter index on its own (the
synthetic gradient is diagonal; the gossip mixes the workers' values at one
index), so contexts holding disjoint ranges of one problem must reproduce the
matching parts of the context that holds all of it bit for bit, and their
consensus-error shares must add up to its consensus error (the fp64 sums
across elements are taken in another order: relative 1e-12).  A range context
must also equal the oracle held on the same global indices.  This is the
replica store split over GPUs, one range per GPU, run here on one GPU.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import oracle_problem, assert_ce

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _ctx(N, P, topo, seed, hp, numels=None, p_range=None, draw_hmax=None):
    full = dict(wl.COMMON_HP)
    full.update(hp)
    return g.Context(N, P, topo, seed, hparams=g.make_hparams(**full), numels=numels, p_range=p_range,
                     draw_hmax=draw_hmax)


CASES = [
    # N, P, topology, hp, layout, split points, H (-1: per-worker H_i from 1..4)
    (8, 9000, "exp", dict(weights="metropolis", edge_prob=0.5, per_worker_h=True), None, [4096], -1),
    (6, 7001, "ring", dict(storage="bf16"), None, [3333], 2),                  # odd split: bf16 noise pairs cut
    (4, 6150, "torus:2x2", dict(weights="metropolis"), [1000, 3, 4097, 1050], [999, 1003, 5100], 1),
    (5, 5000, "2peer", dict(weights="lazy", outer="eq2", alpha=0.8, gamma=0.3, eta=0.9), None, [1, 2500], 2),
    (3, 4100, "matching", dict(outer="local_dadam"), None, [4099], 3),
]


@pytest.mark.parametrize("N,P,topo,hp,numels,cuts,H", CASES)
def test_ranges_reproduce_the_whole(N, P, topo, hp, numels, cuts, H):
    seed, R = 4242, 3
    hmax = 4 if H < 0 else None
    bounds = [0] + list(cuts) + [P]
    whole = _ctx(N, P, topo, seed, hp, numels, draw_hmax=hmax)
    parts = [_ctx(N, P, topo, seed, hp, numels, p_range=(a, b), draw_hmax=hmax) for a, b in zip(bounds, bounds[1:])]
    try:
        for part, (a, b) in zip(parts, zip(bounds, bounds[1:])):
            assert g.gasloc_get_range(part.h) == (a, b, P) and part.P == b - a
        for r in range(R):
            for c in [whole] + parts:
                c.local_steps(H)
                c.gossip_round()
            ce_parts = [p.consensus_error() for p in parts]
            assert sum(ce_parts) == pytest.approx(whole.consensus_error(), rel=1e-12), r
        for which in ("x", "y", "m", "v", "b", "c", "h"):
            full = whole.read_all(which)
            cat = np.concatenate([p.read_all(which) for p in parts], axis=1)
            np.testing.assert_array_equal(cat, full, err_msg=which)
        np.testing.assert_array_equal(np.concatenate([p.average_host() for p in parts]), whole.average_host())
        # gather counts from the range's first index
        for p, (a, b) in zip(parts, zip(bounds, bounds[1:])):
            idx = np.array([0, (b - a) // 2, b - a - 1], np.int64)
            np.testing.assert_array_equal(p.gather("x", N - 1, idx), whole.gather("x", N - 1, idx + a))
    finally:
        for c in [whole] + parts:
            c.close()


def test_range_matches_the_oracle_on_its_indices():
    N, P, seed = 8, 20000, 77
    hp = dict(wl.COMMON_HP, weights="metropolis", edge_prob=0.5, per_worker_h=True, lr=2e-3, noise_sigma=0.02)
    a, b = 6144, 13001
    ctx = _ctx(N, P, "exp", seed, hp, p_range=(a, b), draw_hmax=5)
    st = oracle.get("f32").state(oracle_problem(N, P, "exp", seed, hp), np.arange(a, b, dtype=np.int64))
    Hi = oracle.get("f32").draw_local_steps(seed, N, 5)
    with ctx:
        np.testing.assert_array_equal(g.gasloc_get_local_steps(ctx.h, N), Hi)
        for _ in range(3):
            ctx.local_steps(g.PER_WORKER_STEPS)
            st.local_steps(0, Hi)
            ctx.gossip_round()
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        for which in ("x", "b", "m", "v"):
            np.testing.assert_array_equal(ctx.read_all(which), st.get_all(which).astype(np.float32), err_msg=which)


def test_consensus_error_share_to_device_memory():
    # the share a context contributes to an all-reduce, copied on its stream
    N, P = 4, 10000
    with _ctx(N, P, "ring", 3, {}, p_range=(2000, 9000)) as ctx:
        ctx.local_steps(1)
        ctx.gossip_round()
        dev = torch.full((2,), -1.0, dtype=torch.float64, device="cuda")
        ctx.consensus_error_async(dev.data_ptr() + 8)
        torch.cuda.synchronize()
        assert dev[1].item() == ctx.consensus_error() and dev[0].item() == -1.0


def test_range_checkpoint_keeps_its_range(tmp_path):
    N, P = 4, 8000
    path = str(tmp_path / "r.ckpt")
    with _ctx(N, P, "ring", 9, {}, p_range=(1000, 5000)) as a:
        a.local_steps(2)
        a.gossip_round()
        a.save(path)
        with _ctx(N, P, "ring", 9, {}, p_range=(1000, 5001)) as other:
            with pytest.raises(g.GaslocError) as e:
                other.load(path)
            assert e.value.code == g.EINVAL
        with _ctx(N, P, "ring", 9, {}, p_range=(1000, 5000)) as b:
            b.load(path)
            for _ in range(2):
                for c in (a, b):
                    c.local_steps(1)
                    c.gossip_round()
            np.testing.assert_array_equal(a.read_all("x"), b.read_all("x"))


def _rank_main(rank, world, port, out, N, P, topo, seed, rounds):
    import os
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch
    import torch.distributed as dist
    import bench
    import paper_2606_11081_gb300 as g
    from paper_2606_11081_gb300 import workloads as wl
    torch.cuda.set_device(0)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        hp = dict(wl.COMMON_HP, weights="metropolis", edge_prob=0.5, per_worker_h=True)
        ctx = g.Context(N, P, topo, seed, hparams=g.make_hparams(**hp), draw_hmax=4,
                        p_range=bench.shard_range(P, world, rank))
        ce = torch.zeros(rounds, dtype=torch.float64, device="cuda")
        for k in range(rounds):
            ctx.local_steps(g.PER_WORKER_STEPS)
            ctx.gossip_round()
            bench.ce_exchange(dist, ctx, ce, k)     # the one exchange of a round
        torch.cuda.synchronize()
        out[rank] = (ctx.read_all("x"), ce.cpu().numpy())
        ctx.close()
    finally:
        dist.destroy_process_group()


def test_ranks_on_parameter_ranges_with_host_collectives():
    # Two ranks, each holding one range of the parameters, exchange their
    # consensus-error shares through bench.ce_exchange (the all-reduce of the
    # multi-GPU bench).  Run here as two processes on this one GPU with a
    # host (gloo) all-reduce: no kernel waits on another process.  Together
    # they must reproduce one context holding everything.
    import socket
    import torch.multiprocessing as mp
    N, P, topo, seed, rounds = 8, 3 * 4096 + 901, "exp", 61, 3
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_rank_main, args=(2, port, out, N, P, topo, seed, rounds), nprocs=2, join=True,
                       start_method="spawn")
    hp = dict(weights="metropolis", edge_prob=0.5, per_worker_h=True)
    with _ctx(N, P, topo, seed, hp, draw_hmax=4) as whole:
        ces = []
        for _ in range(rounds):
            whole.local_steps(g.PER_WORKER_STEPS)
            whole.gossip_round()
            ces.append(whole.consensus_error())
        x = whole.read_all("x")
    np.testing.assert_array_equal(np.concatenate([out[0][0], out[1][0]], axis=1), x)
    for r in range(2):
        np.testing.assert_allclose(out[r][1], ces, rtol=1e-12)
