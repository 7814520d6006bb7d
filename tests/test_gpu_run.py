"""gasloc_run: rounds replayed from CUDA graphs (one of 8 consecutive rounds
while that many are left, one of a single round for the rest) must be
exactly the rounds the call-by-call API produces (and the oracle's),
including random per-round graphs (the round number is read on the device),
per-worker step counts, a hyperparameter change (new graphs are captured)
and the consensus-error trace."""
import numpy as np
import pytest

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import make_pair, assert_ce

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()


CASES = [
    (8, "matching", dict(), 2, None),
    (6, "exp", dict(weights="metropolis", edge_prob=0.5, per_worker_h=True), -1, [1, 3, 2, 1, 2, 3]),
    (4, "ring", dict(outer="eq2", alpha=0.8, gamma=0.3, eta=0.9), 1, None),
    (8, "2peer", dict(weights="lazy", outer="local_dadam"), 3, None),
]


@pytest.mark.parametrize("N,topo,kw,H,Hi", CASES)
def test_run_matches_stepwise_and_oracle(N, topo, kw, H, Hi):
    # 19 rounds: two replays of the 8-round graph, then three single rounds
    P, R = 3 * 1024 + 7, 19
    hp = dict(kw, lr=2e-3)
    a, st = make_pair(N, P, topo, seed=42, hp=hp, Hi=Hi)
    b, _ = make_pair(N, P, topo, seed=42, hp=hp, Hi=Hi)
    Hc = H if H > 0 else g.PER_WORKER_STEPS
    with a, b:
        trace = a.run(R, Hc, trace=True)
        ces = []
        for _ in range(R):
            b.local_steps(Hc)
            b.gossip_round()
            ces.append(b.consensus_error())
            st.local_steps(H if H > 0 else 0, None if Hi is None else np.array(Hi, np.int32))
            st.gossip_round()
        np.testing.assert_array_equal(trace, np.array(ces))
        assert a.round == b.round == R
        for i in range(N):
            assert a.steps_taken(i) == b.steps_taken(i) == st.steps_taken(i)
        for w in ("x", "b", "m", "v", "y"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        np.testing.assert_array_equal(a.read_all("x"), st.get_all("x").astype(np.float32))
        # continue call by call after graph rounds, and with graph rounds again
        a.local_steps(Hc)
        a.gossip_round()
        b.run(1, Hc)
        np.testing.assert_array_equal(a.read_all("x"), b.read_all("x"))


def test_long_run_matches_stepwise_and_oracle():
    # 75 rounds: nine replays of the 8-round graph, then three single rounds;
    # random per-round graphs and per-worker step counts make every round
    # differ, and the trace holds every round's value
    N, P, R, Hi = 6, 2 * 1024 + 9, 75, [1, 3, 2, 1, 2, 3]
    hp = dict(weights="metropolis", edge_prob=0.5, per_worker_h=True, lr=2e-3)
    a, st = make_pair(N, P, "exp", seed=17, hp=hp, Hi=Hi)
    b, _ = make_pair(N, P, "exp", seed=17, hp=hp, Hi=Hi)
    with a, b:
        trace = a.run(R, g.PER_WORKER_STEPS, trace=True)
        ces = []
        for _ in range(R):
            b.local_steps(g.PER_WORKER_STEPS)
            b.gossip_round()
            ces.append(b.consensus_error())
            st.local_steps(0, np.array(Hi, np.int32))
            st.gossip_round()
        np.testing.assert_array_equal(trace, np.array(ces))
        assert a.round == b.round == R
        for i in range(N):
            assert a.steps_taken(i) == b.steps_taken(i) == st.steps_taken(i)
        for w in ("x", "b", "m", "v", "y"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
        np.testing.assert_array_equal(a.read_all("x"), st.get_all("x").astype(np.float32))


def test_hparam_change_recaptures():
    P = 5000
    a, _ = make_pair(8, P, "exp", seed=7, hp=dict(lr=1e-3))
    b, _ = make_pair(8, P, "exp", seed=7, hp=dict(lr=1e-3))
    with a, b:
        a.run(10, 1)          # both graphs captured: 8 rounds, then 1 + 1
        for _ in range(10):
            b.local_steps(1)
            b.gossip_round()
        hp2 = g.make_hparams(**dict(wl.COMMON_HP, lr=4e-3, outer="sgdm", outer_momentum=0.5))
        a.set_hparams(hp2)
        b.set_hparams(hp2)
        a.run(12, 2)          # both captured again for the new settings and H
        for _ in range(12):
            b.local_steps(2)
            b.gossip_round()
        np.testing.assert_array_equal(a.read_all("x"), b.read_all("x"))
        np.testing.assert_array_equal(a.read_all("b"), b.read_all("b"))
        assert a.consensus_error() == b.consensus_error()
        # not at a round boundary: refused
        a.local_steps(1)
        with pytest.raises(g.GaslocError) as e:
            a.run(1, 1)
        assert e.value.code == g.ESTATE


def test_async_consensus_error_reads():
    """Per-round values copied without waiting equal the blocking reads of
    the same rounds on an identical context (and the oracle's), including a
    read before any round (standalone reduction) and one after a write of x."""
    import torch
    N, P, R = 8, 5 * 1024 + 3, 7
    hp = dict(lr=2e-3, weights="metropolis", edge_prob=0.5)
    a, st = make_pair(N, P, "exp", seed=9, hp=hp)
    b, _ = make_pair(N, P, "exp", seed=9, hp=hp)
    host = torch.full((R + 2,), -1.0, dtype=torch.float64, pin_memory=True)
    base = host.data_ptr()
    with a, b:
        a.consensus_error_async(base)
        want = [b.consensus_error()]
        for r in range(R):
            a.local_steps(2)
            a.gossip_round()
            a.consensus_error_async(base + 8 * (r + 1))
            b.local_steps(2)
            b.gossip_round()
            want.append(b.consensus_error())
            st.local_steps(2)
            st.gossip_round()
        x3 = b.read("x", 3) * np.float32(1.5)
        a.write("x", 3, x3)
        b.write("x", 3, x3)
        a.consensus_error_async(base + 8 * (R + 1))
        want.append(b.consensus_error())
        a.synchronize()
        got = host.numpy().tolist()
    assert got == want
    assert_ce(want[R], st)


def test_hparam_change_matches_oracle():
    """lr, both betas and the outer optimizer changed between rounds: the
    device's step scalars (the refreshed step table, the re-formed beta^n)
    and outer update follow the oracle's bit for bit."""
    from _pairs import oracle_problem
    N, P = 8, 3001
    ctx, st = make_pair(N, P, "exp", seed=17, hp=dict(lr=1e-3))
    with ctx:
        for _ in range(2):
            ctx.local_steps(2)
            ctx.gossip_round()
            st.local_steps(2)
            st.gossip_round()
        full2 = dict(wl.COMMON_HP, lr=4e-3, beta1=0.8, beta2=0.99, outer="sgdm", outer_momentum=0.5)
        ctx.set_hparams(g.make_hparams(**full2))
        st.set_hparams(oracle_problem(N, P, "exp", 17, full2))
        for _ in range(3):
            ctx.local_steps(3)
            ctx.gossip_round()
            st.local_steps(3)
            st.gossip_round()
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(ctx.read_all(w), st.get_all(w).astype(np.float32), err_msg=w)
        assert_ce(ctx.consensus_error(), st)


def test_run_with_lr_schedule_matches_stepwise():
    hp = dict(lr=3e-3, lr_total_steps=12, lr_final_frac=0.05)
    a, _ = make_pair(8, 4099, "matching", seed=23, hp=hp)
    b, _ = make_pair(8, 4099, "matching", seed=23, hp=hp)
    with a, b:
        a.run(6, 3)
        for _ in range(6):
            b.local_steps(3)
            b.gossip_round()
        for w in ("x", "y", "m", "v", "b"):
            np.testing.assert_array_equal(a.read_all(w), b.read_all(w), err_msg=w)
