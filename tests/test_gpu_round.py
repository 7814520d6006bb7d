"""gasloc_fused_round: one whole round of Algorithm 1 (H local steps, then the
gossip round) with the round's last local step fused into the gossip kernel,
an opt-in variant outside the one-pass-per-local-step byte model.  It serves
at most 4 workers with fp32 storage and a small store, where every worker
takes the round's last step from the same iterate.  Every step acts on each
parameter index on its own, so the fused round must reproduce the two calls
bit for bit: every array and the step counters.  The consensus error is the
same sum of the same per-element terms, whose fp64 partial sums the fused
kernel takes over other tiles (512 elements, its own grid), so it agrees to
the rounding of the sum order (relative 1e-12).  Where the fused kernel
runs, a round makes exactly one launch fewer than the two calls; elsewhere
(more workers, bf16, workers with different step counts, H = 0) the same
launches.  The oracle checks the fused path directly on every outer mode and
at the 4-worker 1 Mi-parameter size."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import make_pair, assert_ce, oracle_problem

pytestmark = pytest.mark.gpu

MODES = ["sgd", "sgdm", "nesterov", "eq2", "dadam", "local_dadam"]
ARRAYS = ("x", "y", "m", "v", "b", "c", "h")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _ctx(N, P, topo, seed, hp, numels=None, Hi=None, p_range=None):
    full = dict(wl.COMMON_HP)
    full.update(hp)
    return g.Context(N, P, topo, seed, hparams=g.make_hparams(**full), numels=numels, local_steps=Hi,
                     p_range=p_range)


def _outer(mode):
    return dict(outer=mode, lr=2e-3, eta=0.9, alpha=0.8, gamma=0.3, outer_lr=0.7, outer_momentum=0.9,
                noise_sigma=0.02)


CASES = [
    # id, N, P, topology, extra hp, layout, H, H_i, fused
    ("ring_h1", 4, 3 * 512 + 7, "ring", {}, None, 1, None, True),
    ("matching_h3", 3, 5000, "matching", {}, None, 3, None, True),
    ("exp_drop_own_h_sched", 4, 4099, "exp", dict(weights="metropolis", edge_prob=0.5, per_worker_h=True,
                                                  lr_total_steps=5), None, 2, None, True),
    ("tensor_list", 2, 0, "complete", {}, [700, 3, 1029, 515, 1], 1, None, True),
    ("one_worker", 1, 777, "none", {}, None, 2, None, True),
    ("equal_hi", 4, 2048, "2peer", dict(weights="lazy"), None, g.PER_WORKER_STEPS, [2, 2, 2, 2], True),
    ("unequal_hi", 4, 2048, "ring", {}, None, g.PER_WORKER_STEPS, [1, 3, 2, 1], False),
    ("no_steps", 4, 2048, "ring", {}, None, 0, None, False),
    ("five_workers", 5, 2048, "ring", {}, None, 1, None, False),
    ("bf16", 4, 2048, "ring", dict(storage="bf16"), None, 1, None, False),
]


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_fused_round_equals_the_two_calls(case, mode):
    _, N, P, topo, extra, numels, H, Hi, fused = case
    if numels is not None:
        P = sum(numels)
    hp = dict(_outer(mode), **extra)
    Hi_a = None if Hi is None else np.array(Hi, np.int32)
    R = 4
    with _ctx(N, P, topo, 31, hp, numels, Hi_a) as a, _ctx(N, P, topo, 31, hp, numels, Hi_a) as b:
        for r in range(R):
            a.fused_round(H)
            b.local_steps(H)
            b.gossip_round()
            assert a.consensus_error() == pytest.approx(b.consensus_error(), rel=1e-12, abs=1e-300), r
        assert a.round == b.round == R
        for i in range(N):
            assert a.steps_taken(i) == b.steps_taken(i)
        for w in ARRAYS:
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        assert b.launches - a.launches == (R if fused else 0)
        # the rounds go on from the fused state exactly as from the other
        a.local_steps(1)
        a.gossip_round()
        b.fused_round(1)
        np.testing.assert_array_equal(a.read_all("x"), b.read_all("x"))


@pytest.mark.parametrize("mode", MODES)
def test_fused_round_matches_the_oracle(mode):
    N, P, R = 4, 3 * 512 + 5, 3
    ctx, st = make_pair(N, P, "matching", seed=44, hp=_outer(mode))
    with ctx:
        for _ in range(R):
            ctx.fused_round(2)
            st.local_steps(2)
            st.gossip_round()
            assert_ce(ctx.consensus_error(), st)
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(ctx.read_all(w), st.get_all(w).astype(np.float32), err_msg=w)


def test_fused_round_in_the_middle_of_a_round():
    # every worker already took a step this round: the fused step starts from y
    hp = _outer("nesterov")
    with _ctx(4, 3000, "ring", 5, hp) as a, _ctx(4, 3000, "ring", 5, hp) as b:
        for _ in range(2):
            a.local_steps(1)
            a.fused_round(1)
            b.local_steps(2)
            b.gossip_round()
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        assert a.consensus_error() == pytest.approx(b.consensus_error(), rel=1e-12)


def test_fused_round_on_parameter_ranges():
    # range contexts (odd cuts: the noise keys follow the global index) add up
    # to the whole context, all of them running fused rounds
    N, P, cuts = 4, 6001, [1, 2501, 4097]
    hp = dict(_outer("nesterov"), weights="metropolis", edge_prob=0.5)
    bounds = [0] + cuts + [P]
    whole = _ctx(N, P, "exp", 12, hp)
    parts = [_ctx(N, P, "exp", 12, hp, p_range=(lo, hi)) for lo, hi in zip(bounds, bounds[1:])]
    try:
        for r in range(3):
            for c in [whole] + parts:
                c.fused_round(2)
            assert sum(p.consensus_error() for p in parts) == pytest.approx(whole.consensus_error(), rel=1e-12)
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(np.concatenate([p.read_all(w) for p in parts], axis=1), whole.read_all(w))
    finally:
        for c in [whole] + parts:
            c.close()


def test_fused_round_ring_full_size():
    """The 4-worker ring on 1 Mi parameters, one local step per round, in the
    launch configuration the benchmark times: fused rounds equal the two calls
    on every element, and the oracle on sampled elements (the tiles' edges and
    random ones)."""
    w = wl.WORKLOADS["ring_n4_p1m"]
    hp = wl.hparams_of(w)
    P = w.n_params
    rng = np.random.default_rng(3)
    kidx = np.unique(np.concatenate([np.arange(0, P, 512), np.arange(511, P, 512), rng.integers(0, P, 4000)]))
    full = dict(wl.COMMON_HP)
    full.update(hp)
    st = oracle.get("f32").state(oracle_problem(w.n_workers, P, w.topology, w.seed, full), kidx.astype(np.int64))
    with _ctx(w.n_workers, P, w.topology, w.seed, hp) as a, _ctx(w.n_workers, P, w.topology, w.seed, hp) as b:
        for _ in range(3):
            a.fused_round(w.H)
            b.local_steps(w.H)
            b.gossip_round()
            st.local_steps(w.H)
            st.gossip_round()
        assert b.launches - a.launches == 3
        assert a.consensus_error() == pytest.approx(b.consensus_error(), rel=1e-12)
        for arr in ("x", "y", "m", "v", "b"):
            xa = a.read_all(arr)
            np.testing.assert_array_equal(xa, b.read_all(arr), err_msg=arr)
            np.testing.assert_array_equal(xa[:, kidx], st.get_all(arr).astype(np.float32), err_msg=arr)
