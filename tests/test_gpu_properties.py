"""Properties of the GPU path that the paper fixes and that hold at any size,
checked on the device path itself (not only through the oracle):

* 1-Peer expected contraction: with no local progress (pure consensus) and
  an SGD outer step of rate alpha on the random matching, the mean one-round
  ratio of consensus errors is 1 - alpha n/(n-1) + alpha^2 n/(2(n-1)), from
  E[Lambda] = E[Lambda^2] = n/(2(n-1)) pi (Prop. 1);
* ring eigenmodes: on the uniform ring a cosine mode decays by exactly
  1/3 + 2/3 cos(2 pi q / n) per round (SGD outer step of rate 1);
* mean preservation (1^T Lambda = 0): the replica mean never moves under pure
  consensus on a doubly stochastic graph."""
import math

import numpy as np
import pytest
import torch

import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

PURE = dict(lr=0.0, noise_sigma=0.0, weight_decay=0.0)


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()


def ctx_of(N, P, topo, **kw):
    hp = g.make_hparams(**dict(wl.COMMON_HP, **kw))
    return g.Context(N, P, topo, 77, hparams=hp)


def test_one_peer_expected_contraction_on_gpu():
    N, P, alpha, T = 16, 1 << 16, 1.0, 600
    pred = 1 - alpha * N / (N - 1) + alpha ** 2 * N / (2 * (N - 1))      # 7/15
    rng = np.random.default_rng(3)
    with ctx_of(N, P, "matching", outer="sgd", outer_lr=alpha, **PURE) as c:
        ratios = []
        for t in range(T):
            if t % 20 == 0:     # fresh random disagreement every 20 rounds
                for i in range(N):
                    c.write("x", i, rng.normal(size=P).astype(np.float32))
            c0 = c.consensus_error()
            c.local_steps(1)
            c.gossip_round()
            ratios.append(c.consensus_error() / c0)
    ratios = np.array(ratios)
    se = ratios.std() / math.sqrt(T)
    assert abs(ratios.mean() - pred) < 4 * se + 1e-3, (ratios.mean(), pred, se)


@pytest.mark.parametrize("N,q", [(8, 1), (16, 3)])
def test_ring_eigenmode_decay_on_gpu(N, q):
    P, R = 3 * 4096 + 11, 6
    phase = np.random.default_rng(0).uniform(0, 2 * math.pi, P)
    lam = 1 / 3 + 2 / 3 * math.cos(2 * math.pi * q / N)
    with ctx_of(N, P, "ring", outer="sgd", outer_lr=1.0, **PURE) as c:
        x0 = np.stack([np.cos(2 * math.pi * q * i / N + phase) for i in range(N)]).astype(np.float32)
        for i in range(N):
            c.write("x", i, x0[i])
        for r in range(1, R + 1):
            c.local_steps(1)
            c.gossip_round()
            np.testing.assert_allclose(c.read_all("x"), lam ** r * x0.astype(np.float64), atol=2e-6)


@pytest.mark.parametrize("topo,kw", [("exp", {}), ("matching", {}), ("torus:2x4", {"weights": "metropolis"}),
                                     ("exp", {"weights": "metropolis", "edge_prob": 0.5})])
def test_mean_preserved_on_gpu(topo, kw):
    N, P = 8, 50_000
    rng = np.random.default_rng(1)
    with ctx_of(N, P, topo, outer="nesterov", **PURE, **kw) as c:
        x0 = rng.normal(size=(N, P)).astype(np.float32)
        for i in range(N):
            c.write("x", i, x0[i])
        m0 = x0.astype(np.float64).mean(0)
        for _ in range(8):
            c.local_steps(1)
            c.gossip_round()
        np.testing.assert_allclose(c.read_all("x").astype(np.float64).mean(0), m0, atol=2e-6)
