"""bf16 replica store vs the oracle's bf16 rule (fp32 arithmetic, every stored
value rounded to bfloat16 with ties to even): bit-exact everywhere."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import make_pair, workload_pair, assert_ce

pytestmark = pytest.mark.gpu
BF = dict(storage="bf16")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def same(ctx, st, which):
    for w in which:
        a = ctx.read_all(w)
        b = st.get_all(w).astype(np.float32)
        assert not (a.view(np.uint32) & 0xFFFF).any(), w
        np.testing.assert_array_equal(a, b, err_msg=w)


def test_bf16_init_and_steps():
    ctx, st = make_pair(5, 4099, "ring", seed=3, hp=dict(BF, per_worker_h=True, lr=2e-3))
    with ctx:
        same(ctx, st, ("x", "y", "c", "h"))
        ctx.local_steps(3)
        st.local_steps(3)
        same(ctx, st, ("y", "m", "v"))


@pytest.mark.parametrize("mode", ["nesterov", "sgd", "eq2", "local_dadam"])
@pytest.mark.parametrize("N,topo,kw", [(8, "exp", {}), (16, "matching", {}),
                                       (32, "exp", {"weights": "metropolis", "edge_prob": 0.5})])
def test_bf16_trajectory(mode, N, topo, kw):
    P, R, H = 2 * 1024 + 5, 4, 2
    hp = dict(kw, **BF, outer=mode, lr=2e-3, eta=0.9, alpha=0.8, gamma=0.3, noise_sigma=0.02)
    ctx, st = make_pair(N, P, topo, seed=500 + N, hp=hp)
    with ctx:
        for _ in range(R):
            ctx.local_steps(H)
            st.local_steps(H)
            ctx.gossip_round()
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        same(ctx, st, ("x", "b", "m", "v"))


@pytest.mark.parametrize("mode", ["sgd", "sgdm", "nesterov", "dadam", "local_dadam"])
@pytest.mark.parametrize("N,topo,kw", [(2, "ring", {}), (3, "complete", {}), (5, "2peer", {}),
                                       (8, "matching", {}), (7, "exp", {"weights": "metropolis", "edge_prob": 0.5}),
                                       (6, "torus:2x3", {"weights": "lazy"})])
def test_bf16_dense_mixing(mode, N, topo, kw):
    """Up to 8 workers a bf16 column is mixed densely (zero weight off the
    graph): bit-exact against the neighbour-list sums for every outer mode,
    and on graphs drawn afresh each round (1-Peer, 2-Peer, dropped edges)."""
    P, R, H = 3 * 1024 + 7, 4, 1
    hp = dict(kw, **BF, outer=mode, lr=2e-3, eta=0.9, alpha=0.8, gamma=0.3, noise_sigma=0.02)
    ctx, st = make_pair(N, P, topo, seed=900 + N, hp=hp)
    with ctx:
        for _ in range(R):
            ctx.local_steps(H)
            st.local_steps(H)
            ctx.gossip_round()
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        same(ctx, st, ("x", "b", "m", "v", "y"))


def test_bf16_heterogeneous_and_graph_rounds():
    Hi = np.array([0, 2, 1, 3], np.int32)
    ctx, st = make_pair(4, 3001, "complete", seed=8, hp=dict(BF, lr=1e-3), Hi=Hi)
    with ctx:
        ctx.run(3, g.PER_WORKER_STEPS)
        for _ in range(3):
            st.local_steps(0, Hi)
            st.gossip_round()
        same(ctx, st, ("x", "b", "y"))


def test_bf16_layout_and_host_conversion():
    numels = [1000, 3, 4097, 64, 1, 2048, 5]
    P = sum(numels)
    a, _ = make_pair(8, P, "torus:2x4", seed=11, hp=dict(BF, weights="metropolis"))
    b, _ = make_pair(8, P, "torus:2x4", seed=11, hp=dict(BF, weights="metropolis"), numels=numels)
    with a, b:
        for c in (a, b):
            c.local_steps(2)
            c.gossip_round()
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        # fp32 written from the host is rounded to nearest even bf16
        vals = np.random.default_rng(0).normal(size=P).astype(np.float32)
        a.write("x", 3, vals)
        ref = torch.tensor(vals).to(torch.bfloat16).to(torch.float32).numpy()
        np.testing.assert_array_equal(a.read("x", 3), ref)
        v = b.view("x", 2, numels[2])
        assert v.dtype == torch.bfloat16 and tuple(v.shape) == (8, numels[2])
        np.testing.assert_array_equal(v.float().cpu().numpy(), b.read_all("x")[:, 1003:1003 + 4097])


def test_bf16_bench_workload_full_size_sampled():
    w = wl.ALL_WORKLOADS["exp_n8_gpt2s_bf16"]
    rng = np.random.default_rng(1)
    kidx = np.unique(np.concatenate([[0, 1, 1023, 1024, w.n_params - 1, w.n_params - 4],
                                     rng.integers(0, w.n_params, 1500)])).astype(np.int64)
    ctx, st = make_pair(w.n_workers, w.n_params, w.topology, w.seed, wl.hparams_of(w), kidx=kidx)
    try:
        for _ in range(w.rounds):
            ctx.local_steps(w.H)
            ctx.gossip_round()
            st.local_steps(w.H)
            st.gossip_round()
        for which in ("x", "b", "m", "v"):
            for i in range(w.n_workers):
                np.testing.assert_array_equal(ctx.gather(which, i, kidx), st.get(which, i).astype(np.float32))
        assert ctx.consensus_error() == pytest.approx(ctx.consensus_error_now(), rel=1e-12)
    finally:
        ctx.close()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()


def test_bf16_host_transfer_over_staging_chunks():
    # one tensor longer than the 32 Mi-element staging buffer: two chunks
    P = (1 << 25) + 4099
    bits = np.array([0x3F808000, 0x3F818000, 0xBF808000, 0x7F7FFFFF, 0xFF7FFFFF, 0x7F800000,
                     0xFF800000, 0x00000001, 0x80000001, 0x007FFFFF, 0x3F80FFFF, 0x00000000,
                     0x80000000], np.uint32)
    vals = np.random.default_rng(5).normal(size=P).astype(np.float32)
    vals[:bits.size] = bits.view(np.float32)
    vals[(1 << 25) - 2:(1 << 25) + 2] = bits[:4].view(np.float32)   # across the chunk seam
    ref = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float32).numpy()
    with g.Context(2, P, "ring", 1, hparams=g.make_hparams(storage="bf16")) as ctx:
        ctx.write("c", -1, vals)
        for i in range(2):
            got = ctx.read("c", i)
            np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("storage", ["f32", "bf16"])
@pytest.mark.parametrize("N,topo,kw", [(8, "ring", {}), (8, "exp", {"weights": "metropolis", "edge_prob": 0.5}),
                                       (6, "2peer", {"weights": "lazy"}), (4, "ring", {}),
                                       (4, "exp", {"weights": "metropolis", "edge_prob": 0.5}),
                                       (4, "2peer", {"weights": "lazy"})])
def test_nonfinite_replica_reaches_neighbours_only(storage, N, topo, kw):
    # A diverged replica (inf in some elements of worker j) is mixed only by
    # the workers whose neighbourhood holds j, as in the oracle's neighbour
    # lists; the dense mixing forms (bf16 at n <= 8, and the fp32 kernel that
    # holds a column of every worker in registers at n <= 4) must not carry
    # it elsewhere.
    P = 2 * 1024 + 5
    hp = dict(kw, storage=storage, outer="nesterov")
    ctx, st = make_pair(N, P, topo, seed=900 + N, hp=hp)
    with ctx:
        j = 3
        bad = ctx.read("x", j)
        cols = np.array([0, 1, 700, 1031, P - 1])
        bad[cols[:3]] = np.inf
        bad[cols[3:]] = -np.inf
        ctx.write("x", j, bad)
        st.set("x", j, bad.astype(np.float64))
        # round 0: no local step, every worker sends x
        nbr, w, deg = ctx.topology(0)
        ctx.gossip_round()
        st.gossip_round()
        x = ctx.read_all("x")
        np.testing.assert_array_equal(x, st.get_all("x").astype(np.float32))
        np.testing.assert_array_equal(ctx.read_all("b"), st.get_all("b").astype(np.float32))
        mixes_j = [i for i in range(N) if j in nbr[i, :deg[i] + 1]]
        assert j in mixes_j
        for i in range(N):
            if i in mixes_j:
                assert not np.isfinite(x[i, cols]).any(), i
            else:
                assert np.isfinite(x[i]).all(), i
        # then ordinary rounds: the non-finite values spread along the graph
        # exactly as in the oracle
        for _ in range(2):
            ctx.local_steps(1)
            st.local_steps(1)
            ctx.gossip_round()
            st.gossip_round()
        np.testing.assert_array_equal(ctx.read_all("x"), st.get_all("x").astype(np.float32))
        np.testing.assert_array_equal(ctx.read_all("b"), st.get_all("b").astype(np.float32))
