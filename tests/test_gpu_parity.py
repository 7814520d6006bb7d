"""GPU path vs the oracle, element by element, through the C ABI.

Integer work (neighbour tables, degrees, step counts) must be bit-exact.
fp32 state must lie within |gpu - oracle| <= 1e-5 (1 + |oracle|) (the parity
bound); because both sides follow the same one-rounding-per-operation
sequence in fp32, the runs here are also expected to agree bit for bit, and
that is asserted too so that any drift in the operation order shows up.
The consensus error is a reduction whose summation order differs between the
two sides: relative 1e-5.
"""
import os

import numpy as np
import pytest

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import TOL, assert_ce, ce_bound, make_pair, oracle_problem, within_tol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def assert_state_equal(ctx, st, which=("x", "y", "m", "v", "b"), exact=True):
    for w in which:
        a = ctx.read_all(w)
        b = st.get_all(w)
        ok = within_tol(a, b)
        assert ok.all(), "%s: %d mismatches, max |d| = %g" % (w, (~ok).sum(), np.abs(a - b).max())
        if exact:
            assert np.array_equal(a, b.astype(np.float32)), \
                "%s: not bit-identical (%d differ, max |d| %g)" % (w, (a != b.astype(np.float32)).sum(),
                                                                   np.abs(a - b).max())


# ---------------------------------------------------------------- init ----

@pytest.mark.parametrize("N,P,per_h", [(4, 4099, False), (3, 1, False), (5, 2050, True), (1, 7, False)])
def test_init_bit_exact(N, P, per_h):
    ctx, st = make_pair(N, P, "ring" if N > 1 else "none", seed=12345, hp=dict(per_worker_h=per_h))
    with ctx:
        for w in ("x", "y", "c", "h"):
            np.testing.assert_array_equal(ctx.read_all(w), st.get_all(w).astype(np.float32), err_msg=w)
        for w in ("m", "v", "b"):
            assert not ctx.read_all(w).any()
        # identical initial replicas: zero consensus error
        assert ctx.consensus_error() == 0.0


# ------------------------------------------------------------ topology ----

TOPO_CASES = [
    (4, "ring", {}), (8, "exp", {}), (32, "exp", {}), (8, "torus:2x4", {"weights": "metropolis"}),
    (6, "complete", {}), (3, "none", {}), (16, "matching", {}), (5, "matching", {}),
    (8, "2peer", {"weights": "lazy"}), (7, "2peer", {"weights": "uniform"}),
    (32, "exp", {"weights": "metropolis", "edge_prob": 0.5}),
    (12, "exp", {"weights": "uniform", "edge_prob": 0.3}),
    (9, "ring", {"weights": "lazy", "edge_prob": 0.8}),
    (8, "exp", {"weights": "metropolis", "edge_prob": 0.0}),    # every edge dropped: W = I
    (8, "matching", {"weights": "uniform", "edge_prob": 0.0}),
]


@pytest.mark.parametrize("N,topo,kw", TOPO_CASES)
def test_topology_bit_exact(N, topo, kw):
    ctx, st = make_pair(N, 8, topo, seed=99, hp=kw)
    with ctx:
        orc = oracle.get("f64")
        pb = oracle_problem(N, 8, topo, 99, dict(wl.COMMON_HP, **kw))
        for t in list(range(40)) + [1000, 123456789]:
            nbr, w, deg = ctx.topology(t)
            onbr, ow, odeg = orc.topology(pb, t)
            np.testing.assert_array_equal(deg, odeg)
            for i in range(N):
                k = deg[i] + 1
                np.testing.assert_array_equal(nbr[i, :k], onbr[i, :k])
                np.testing.assert_array_equal(w[i, :k], ow[i, :k].astype(np.float32))


# --------------------------------------------------------- local steps ----

def test_local_steps_bit_exact():
    ctx, st = make_pair(4, 4099, "ring", seed=7, hp=dict(lr=1e-3, noise_sigma=0.05))
    with ctx:
        ctx.local_steps(3)
        st.local_steps(3)
        assert_state_equal(ctx, st, ("y", "m", "v"))
        for i in range(4):
            assert ctx.steps_taken(i) == st.steps_taken(i) == 3


def test_heterogeneous_steps_per_worker_h():
    Hi = np.array([0, 1, 3, 2, 5], np.int32)
    ctx, st = make_pair(5, 3001, "exp", seed=8, hp=dict(per_worker_h=True, lr=1e-3), Hi=Hi)
    with ctx:
        for _ in range(3):
            ctx.local_steps(g.PER_WORKER_STEPS)
            st.local_steps(0, Hi)
            ctx.gossip_round()
            st.gossip_round()
        assert_state_equal(ctx, st)
        for i in range(5):
            assert ctx.steps_taken(i) == 3 * Hi[i]


# --------------------------------------------------------- trajectories ---

MODES = ["nesterov", "sgdm", "sgd", "eq2", "dadam", "local_dadam"]
GRAPHS = [(8, "exp", {}), (16, "matching", {}), (8, "torus:2x4", {"weights": "metropolis"}),
          (32, "exp", {"weights": "metropolis", "edge_prob": 0.5}), (6, "2peer", {"weights": "lazy"}),
          (11, "ring", {"per_worker_h": True}),   # own curvature, more than 7 workers: batches of 2 and a tail
          (4, "ring", {}), (3, "matching", {})]   # few workers, small replicas: the direct gossip variant


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("N,topo,kw", GRAPHS)
def test_trajectory_parity(mode, N, topo, kw):
    P, R, H = 2 * 1024 + 3, 5, 2
    hp = dict(kw, outer=mode, lr=2e-3, eta=0.9, alpha=0.8, gamma=0.3, outer_lr=0.7,
              outer_momentum=0.9, noise_sigma=0.02)
    ctx, st = make_pair(N, P, topo, seed=1000 + N, hp=hp)
    with ctx:
        for r in range(R):
            ctx.local_steps(H)
            st.local_steps(H)
            ctx.gossip_round()
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        assert_state_equal(ctx, st, ("x", "b", "m", "v"))


@pytest.mark.parametrize("N,kw,Hi", [
    (8, {}, None),                                           # shared h, batches of 4
    (16, {"lr_total_steps": 6}, None),                       # shared h, batches of 3, lr schedule
    (5, {"per_worker_h": True}, [2, 0, 1, 2, 1]),            # own h, batches of 3, some workers idle
    (12, {"per_worker_h": True, "lr_total_steps": 6}, None),  # own h, batches of 2, lr schedule
])
def test_register_batched_adamw_on_large_stores(N, kw, Hi):
    # fp32 stores of a few MB per replica and more take the register-batched
    # AdamW (small ones the staged kernel, which the other tests here use):
    # 4 Mi + 333 parameters, every element against the oracle
    P, R = (1 << 22) + 333, 2
    hp = dict(kw, lr=2e-3, noise_sigma=0.02)
    Hi_a = None if Hi is None else np.array(Hi, np.int32)
    ctx, st = make_pair(N, P, "exp", seed=29, hp=hp, Hi=Hi_a)
    H = 2 if Hi is None else g.PER_WORKER_STEPS
    with ctx:
        for _ in range(R):
            ctx.local_steps(H)
            st.local_steps(2 if Hi is None else 0, Hi_a)
            ctx.gossip_round()
            st.gossip_round()
        assert_state_equal(ctx, st, ("x", "y", "m", "v", "b"))


@pytest.mark.parametrize("mode", MODES)
def test_direct_gossip_with_workers_that_took_no_step(mode):
    # Few workers and a small replica store take the direct gossip variant;
    # workers without a local step this round send x, the others y.
    Hi = np.array([0, 2, 1, 0], np.int32)
    hp = dict(per_worker_h=True, lr=2e-3, outer=mode, eta=0.9, alpha=0.8, gamma=0.3, noise_sigma=0.02)
    ctx, st = make_pair(4, 3 * 1024 + 7, "ring", seed=17, hp=hp, Hi=Hi)
    with ctx:
        for _ in range(3):
            ctx.local_steps(g.PER_WORKER_STEPS)
            st.local_steps(0, Hi)
            ctx.gossip_round()
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        assert_state_equal(ctx, st, ("x", "b", "m", "v"))


@pytest.mark.parametrize("N,P,topo", [(1, 5, "none"), (4, 1, "ring"), (4, 3, "complete"),
                                      (2, 1023, "matching"), (5, 1029, "matching"),
                                      (3, 20000, "complete")])
def test_edge_case_shapes(N, P, topo):
    ctx, st = make_pair(N, P, topo, seed=5, hp=dict(lr=5e-3))
    with ctx:
        for _ in range(4):
            ctx.local_steps(2)
            st.local_steps(2)
            ctx.gossip_round()
            st.gossip_round()
        assert_state_equal(ctx, st, ("x", "b"))
        assert_ce(ctx.consensus_error(), st)


def test_ring_n4_p1m_full_size():
    # The 4-worker ring workload at its full size: 1,048,576 parameters, 50 rounds
    w = wl.WORKLOADS["ring_n4_p1m"]
    ctx, st = make_pair(w.n_workers, w.n_params, w.topology, w.seed, wl.hparams_of(w))
    with ctx:
        for r in range(w.rounds):
            ctx.local_steps(w.H)
            st.local_steps(w.H)
            ctx.gossip_round()
            st.gossip_round()
            if r % 10 == 9:
                assert_ce(ctx.consensus_error(), st)
        assert_state_equal(ctx, st, ("x", "b", "m", "v"))
        np.testing.assert_allclose(ctx.average_host(), st.average(), rtol=2e-6, atol=1e-7)


# --------------------------------------------------------- CE / average ---

def test_consensus_error_closed_form_and_paths():
    N, P = 7, 5003
    ctx, _ = make_pair(N, P, "ring", seed=3)
    with ctx:
        for i in range(N):
            ctx.write("x", i, np.full(P, float(i), np.float32))
        # per-element fp32 shifted sums, within the bound of the shifted form
        xs = np.repeat(np.arange(N, dtype=np.float64)[:, None], P, axis=1)
        assert ctx.consensus_error() == pytest.approx(P * (N * N - 1) / 12, rel=ce_bound(xs))
        ctx.local_steps(1)
        ctx.gossip_round()
        fused = ctx.consensus_error()
        # the fused and the standalone reductions take the same per-element
        # terms (both shift by worker 0's new x); only the fp64 order differs
        assert ctx.consensus_error_now() == pytest.approx(fused, rel=1e-12)


@pytest.mark.parametrize("N", [4, 8, 32])
def test_consensus_error_near_consensus_far_from_zero(N):
    # Replicas a thousand times further from zero than from each other:
    # x_ik = a_k + 1e-3 (i - (N-1)/2) with a_k in [1000, 2000).  A one-pass
    # fp32 form without a shift would lose every digit here; the shifted form
    # subtracts worker 0's value exactly (the values are within a factor of 2
    # of each other), so only the sums round.  Compared with the exact
    # consensus error of the stored fp32 values (fp64, two passes), with the
    # oracle, and with the closed form P 1e-6 (N^2 - 1) / 12 of the unrounded
    # values (the fp32 rounding of the values moves it by about 1%).
    P = 3 * 4096 + 77
    hp = dict(outer="sgd", outer_lr=0.0)        # the gossip round leaves x as it is
    ctx, st = make_pair(N, P, "exp", seed=21, hp=hp)
    rng = np.random.default_rng(N)
    a = 1000.0 + 1000.0 * rng.random(P)
    x = np.stack([(a + 1e-3 * (i - (N - 1) / 2)).astype(np.float32) for i in range(N)])
    xd = x.astype(np.float64)
    exact = ((xd - xd.mean(0)) ** 2).sum() / N
    # the shifted form's bound for these values (ce_bound: worker 0's shift
    # makes kappa = sum (x_i - x_0)^2 / sum (x_i - xbar)^2 about 4 here)
    tol = ce_bound(xd)
    with ctx:
        for i in range(N):
            ctx.write("x", i, x[i])
            st.set("x", i, xd[i])
        now = ctx.consensus_error_now()                 # standalone reduction
        ctx.gossip_round()                              # fused reduction of the unchanged x
        np.testing.assert_array_equal(ctx.read_all("x"), x)
        fused = ctx.consensus_error()
        st.gossip_round()
        ref = st.consensus_error()
        assert ref == pytest.approx(exact, rel=1e-12)
        assert ref == pytest.approx(P * 1e-6 * (N * N - 1) / 12, rel=0.05)
        for got in (now, fused):
            assert got == pytest.approx(exact, rel=tol), (got, exact, tol)


@pytest.mark.parametrize("N", [3, 4])
def test_consensus_error_column_sums_over_wide_magnitudes(N):
    # The kernel that holds a column of every worker in registers (at most 4
    # workers, fp32) adds a column's four terms as their exact sum when they
    # lie within 2^26 of the column's largest, and adds the others (smaller,
    # subnormal or zero) one at a time.  Element scales spread over 10^-25 ..
    # 10^10 put every case into most columns: the largest terms near 10^20,
    # terms many binades below them, subnormal terms and exact zeros.  The
    # standalone reduction adds every term on its own, so the two differ only
    # in the order of their fp64 additions; both are within the shifted
    # form's bound of the exact value.
    P = 5 * 1024 + 7
    hp = dict(outer="sgd", outer_lr=0.0)        # the gossip round leaves x as it is
    ctx, st = make_pair(N, P, "ring", seed=40 + N, hp=hp)
    rng = np.random.default_rng(N)
    scale = 10.0 ** rng.uniform(-25.0, 10.0, P)
    scale[rng.random(P) < 0.1] = 0.0            # some columns hold equal replicas: terms of exactly 0
    x = np.stack([(scale * ((i - (N - 1) / 2) + 0.3 * rng.standard_normal(P))).astype(np.float32)
                  for i in range(N)])
    xd = x.astype(np.float64)
    exact = ((xd - xd.mean(0)) ** 2).sum() / N
    with ctx:
        for i in range(N):
            ctx.write("x", i, x[i])
            st.set("x", i, xd[i])
        now = ctx.consensus_error_now()                 # every term added on its own
        ctx.gossip_round()                              # column sums, in the register-column kernel
        np.testing.assert_array_equal(ctx.read_all("x"), x)
        fused = ctx.consensus_error()
        st.gossip_round()
        assert st.consensus_error() == pytest.approx(exact, rel=1e-12)
        assert fused == pytest.approx(now, rel=1e-12)
        tol = ce_bound(xd)
        for got in (now, fused):
            assert got == pytest.approx(exact, rel=tol), (got, exact, tol)
        # a non-finite replica value makes the round's value non-finite in
        # both reductions (the whole column is then added term by term)
        bad = ctx.read("x", 1)
        bad[1030] = np.inf
        ctx.write("x", 1, bad)
        ctx.gossip_round()
        fused = ctx.consensus_error()
        assert not np.isfinite(fused)
        assert not np.isfinite(ctx.consensus_error_now())


@pytest.mark.parametrize("storage", ["f32", "bf16"])
@pytest.mark.parametrize("numels", [None, [1000, 3, 4097, 64, 1, 2048, 5]])
def test_average_is_the_fp32_mean_of_the_replicas(storage, numels):
    # Per element: fp32 sum over ascending workers, then times fl32(1/n).  The
    # tensor list puts tensors at odd offsets of the output (element stores)
    # next to 16-byte-aligned ones (vector stores).
    N, P = 6, 7218
    ctx, _ = make_pair(N, P, "ring", seed=5, hp=dict(lr=2e-3, storage=storage), numels=numels)
    with ctx:
        ctx.local_steps(2)
        ctx.gossip_round()
        X = ctx.read_all("x")
        s = np.zeros(P, np.float32)
        for i in range(N):
            s = (s + X[i]).astype(np.float32)
        ref = (s * np.float32(1.0 / N)).astype(np.float32)
        np.testing.assert_array_equal(ctx.average_host(), ref)


# ------------------------------------------------------ layout / resume ---

def test_tensor_list_equals_flat():
    numels = [1000, 3, 4097, 64, 1, 2048, 5]
    P = sum(numels)
    hp = dict(weights="metropolis", lr=2e-3)
    a, _ = make_pair(8, P, "torus:2x4", seed=11, hp=hp)
    b, _ = make_pair(8, P, "torus:2x4", seed=11, hp=hp, numels=numels)
    with a, b:
        for _ in range(4):
            for c in (a, b):
                c.local_steps(3)
                c.gossip_round()
        # per-element terms are identical and each enters the fp64 sum on its
        # own: only the order of the fp64 sums differs
        assert a.consensus_error() == pytest.approx(b.consensus_error(), rel=1e-12)
        for w in ("x", "y", "m", "v", "b", "c", "h"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        # the per-tensor buffers are separate allocations with the real sizes
        v = b.view("x", 2, numels[2])
        assert tuple(v.shape) == (8, numels[2])
        np.testing.assert_array_equal(v.cpu().numpy(), b.read_all("x")[:, 1003:1003 + 4097])


@pytest.mark.parametrize("sched,storage", [(0, "f32"), (8, "f32"), (8, "bf16")])
def test_resume_is_exact(tmp_path, sched, storage):
    # the resumed context starts with other hyperparameters (no lr schedule):
    # the checkpoint's, schedule included, take over
    hp = dict(weights="metropolis", edge_prob=0.5, per_worker_h=True, lr_total_steps=sched, storage=storage)
    a, _ = make_pair(6, 3000, "exp", seed=21, hp=hp, Hi=[1, 2, 3, 1, 2, 3])
    with a:
        for _ in range(3):
            a.local_steps(g.PER_WORKER_STEPS)
            a.gossip_round()
        path = str(tmp_path / "ckpt.bin")
        a.save(path)
        for _ in range(3):
            a.local_steps(g.PER_WORKER_STEPS)
            a.gossip_round()
        xa = a.read_all("x")
        ce_a = a.consensus_error()
    b, _ = make_pair(6, 3000, "exp", seed=21, hp=dict(hp, lr_total_steps=0), Hi=[1, 1, 1, 1, 1, 1])
    with b:
        b.load(path)
        assert b.round == 3
        for _ in range(3):
            b.local_steps(g.PER_WORKER_STEPS)
            b.gossip_round()
        np.testing.assert_array_equal(b.read_all("x"), xa)
        assert b.consensus_error() == ce_a


def test_gather_rejects_bad_index():
    ctx, _ = make_pair(2, 100, "ring", seed=1)
    with ctx:
        with pytest.raises(g.GaslocError) as e:
            ctx.gather("x", 0, np.array([5, 100]))
        assert e.value.code == g.EINVAL
        np.testing.assert_array_equal(ctx.gather("x", 1, np.array([0, 99, 42])),
                                      ctx.read("x", 1)[[0, 99, 42]])


@pytest.mark.parametrize("storage,per_h", [("f32", False), ("bf16", False), ("bf16", True)])
def test_lr_schedule_matches_oracle(storage, per_h):
    # App. B's warm-up + cosine schedule runs over each worker's own local
    # steps: with different H_i the workers sit at different points of it, and
    # the busiest one passes the warm-up, the decay and the held final rate.
    N, P, R = 6, 2 * 1024 + 9, 5
    Hi = np.array([1, 3, 2, 4, 1, 2], np.int32)
    hp = dict(lr=4e-3, storage=storage, lr_total_steps=9, lr_warmup_frac=0.25, lr_final_frac=0.1,
              per_worker_h=per_h)
    ctx, st = make_pair(N, P, "ring", seed=31, hp=hp, Hi=Hi)
    with ctx:
        for _ in range(R):
            ctx.local_steps(g.PER_WORKER_STEPS)
            ctx.gossip_round()
            st.local_steps(0, Hi)
            st.gossip_round()
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(ctx.read_all(w), st.get_all(w).astype(np.float32), err_msg=w)
