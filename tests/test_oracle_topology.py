"""Pins for the oracle's communication graphs and mixing weights.

Fixed graphs are pinned to the closed-form spectra of circulant and Cartesian
product graphs; the randomized 1-Peer / 2-Peer schemes to Prop. 1 of the paper
(E[Lambda^(1)] = E[(Lambda^(1))^2] = n/(2(n-1)) pi, E[(Lambda^(2))^2] =
3n/(8(n-1)) pi) and to its proof (pair probability 1/(n-1), Lambda^(1)
idempotent).
"""
import math

import numpy as np
import pytest

import oracle


def W_of(o, pb, t=0):
    return o.dense_w(pb, t)


def test_ring_uniform_thirds(orc64):
    pb = oracle.make_problem(4, 1, "ring", weights="uniform")
    nbr, w, deg = orc64.topology(pb, 0)
    assert deg.tolist() == [2, 2, 2, 2]
    assert nbr[0, :3].tolist() == [0, 1, 3]
    assert nbr[2, :3].tolist() == [1, 2, 3]
    assert np.all(w[:, :3] == 1.0 / 3.0)


@pytest.mark.parametrize("n", [3, 4, 5, 8, 16])
def test_ring_spectrum(orc64, n):
    # circulant with taps 1/3 at -1, 0, +1: eigenvalues 1/3 + 2/3 cos(2 pi q/n)
    W = W_of(orc64, oracle.make_problem(n, 1, "ring", weights="uniform"))
    ev = np.sort(np.linalg.eigvalsh(W))
    ref = np.sort([1 / 3 + 2 / 3 * math.cos(2 * math.pi * q / n) for q in range(n)])
    np.testing.assert_allclose(ev, ref, atol=1e-12)


@pytest.mark.parametrize("n,deg", [(8, 5), (16, 7), (32, 9)])
def test_exponential_graph(orc64, n, deg):
    pb = oracle.make_problem(n, 1, "exp", weights="metropolis")
    nbr, w, d = orc64.topology(pb, 0)
    assert d.tolist() == [deg] * n
    W = W_of(orc64, pb)
    # circulant with offsets {+-2^q}: eigenvalue_q = sum over the offset set
    offs = sorted({(s * sg) % n for s in [2 ** q for q in range(6) if 2 ** q < n] for sg in (1, -1)})
    assert len(offs) == deg
    ref = np.sort([(1 + sum(math.cos(2 * math.pi * q * o / n) for o in offs)) / (deg + 1)
                   for q in range(n)])
    np.testing.assert_allclose(np.sort(np.linalg.eigvalsh(W)), ref, atol=1e-12)
    # regular graph: uniform == Metropolis (the Metropolis self weight is
    # 1 - sum of the others in double, equal once rounded to fp32)
    W2 = W_of(orc64, oracle.make_problem(n, 1, "exp", weights="uniform"))
    np.testing.assert_allclose(W, W2, atol=1e-15)
    np.testing.assert_array_equal(W.astype(np.float32), W2.astype(np.float32))


def test_torus_2x4_metropolis(orc64):
    pb = oracle.make_problem(8, 1, "torus", torus=(2, 4), weights="metropolis")
    nbr, w, deg = orc64.topology(pb, 0)
    assert deg.tolist() == [3] * 8
    assert np.all(w[:, :4] == 0.25)
    # node (r, c) = r*4 + c: neighbours (1-r, c), (r, c+-1)
    assert nbr[0, :4].tolist() == [0, 1, 3, 4]
    assert nbr[5, :4].tolist() == [1, 4, 5, 6]
    # Cartesian product K2 x C4: Laplacian eigenvalues a + b, a in {0,2},
    # b in {2 - 2cos(2 pi k/4)}; W = I - L/4
    lam = [a + 2 - 2 * math.cos(2 * math.pi * k / 4) for a in (0, 2) for k in range(4)]
    ref = np.sort([1 - l / 4 for l in lam])
    np.testing.assert_allclose(np.sort(np.linalg.eigvalsh(W_of(orc64, pb))), ref, atol=1e-12)


def test_complete_uniform(orc64):
    W = W_of(orc64, oracle.make_problem(6, 1, "complete"))
    np.testing.assert_allclose(W, np.full((6, 6), 1 / 6), atol=0)


def test_none_is_identity(orc64):
    W = W_of(orc64, oracle.make_problem(5, 1, "none"))
    np.testing.assert_array_equal(W, np.eye(5))


@pytest.mark.parametrize("n", [2, 4, 16])
def test_matching_every_round_perfect(orc64, n):
    pb = oracle.make_problem(n, 1, "matching", seed=17)
    for t in range(200):
        nbr, w, deg = orc64.topology(pb, t)
        assert deg.tolist() == [1] * n
        W = W_of(orc64, pb, t)
        assert np.all(np.isin(W, [0.0, 0.5]))
        np.testing.assert_array_equal(W, W.T)
        # Lambda^(1) = I - W is idempotent (proof of Prop. 1)
        L = np.eye(n) - W
        np.testing.assert_allclose(L @ L, L, atol=0)


def test_matching_odd_worker_alone(orc64):
    pb = oracle.make_problem(5, 1, "matching", seed=3)
    for t in range(20):
        nbr, w, deg = orc64.topology(pb, t)
        assert sorted(deg.tolist()) == [0, 1, 1, 1, 1]
        i = int(np.argmin(deg))
        assert nbr[i, 0] == i and w[i, 0] == 1.0


def test_matching_pair_frequency_and_expectation(orc64):
    # P({a,b} matched) = 1/(n-1); E[Lambda^(1)] = n/(2(n-1)) pi  (Prop. 1)
    n, T = 8, 20000
    pb = oracle.make_problem(n, 1, "matching", seed=123)
    cnt = np.zeros((n, n))
    EL = np.zeros((n, n))
    for t in range(T):
        W = W_of(orc64, pb, t)
        cnt += (W > 0) & ~np.eye(n, dtype=bool)
        EL += np.eye(n) - W
    EL /= T
    freq = cnt[np.triu_indices(n, 1)] / T
    p = 1 / (n - 1)
    assert np.all(np.abs(freq - p) < 5 * math.sqrt(p * (1 - p) / T))
    pi = np.eye(n) - np.ones((n, n)) / n
    np.testing.assert_allclose(EL, n / (2 * (n - 1)) * pi, atol=0.015)


def test_twopeer_prop1(orc64):
    # W = I - Lambda^(2) with lazy weights (self 1/2, the two cycle neighbours 1/4)
    n, T = 8, 20000
    pb = oracle.make_problem(n, 1, "2peer", weights="lazy", seed=77)
    E1 = np.zeros((n, n))
    E2 = np.zeros((n, n))
    for t in range(T):
        W = W_of(orc64, pb, t)
        L = np.eye(n) - W
        if t < 50:
            # one Hamiltonian cycle: every node has two neighbours, spectrum of
            # a quarter of the cycle Laplacian (eigenvalues (1 - cos(2 pi k/n))/2)
            assert np.all((W > 0).sum(1) == 3)
            ref = np.sort([(1 - math.cos(2 * math.pi * k / n)) / 2 for k in range(n)])
            np.testing.assert_allclose(np.sort(np.linalg.eigvalsh(L)), ref, atol=1e-12)
        E1 += L
        E2 += L @ L
    pi = np.eye(n) - np.ones((n, n)) / n
    np.testing.assert_allclose(E1 / T, n / (2 * (n - 1)) * pi, atol=0.01)
    np.testing.assert_allclose(E2 / T, 3 * n / (8 * (n - 1)) * pi, atol=0.01)


def test_edge_activation_frequency_and_metropolis(orc64):
    n, T, p = 32, 400, 0.5
    pb = oracle.make_problem(n, 1, "exp", weights="metropolis", edge_prob=p, seed=5)
    base = W_of(orc64, oracle.make_problem(n, 1, "exp"), 0) > 0
    n_edges = (base.sum() - n) // 2
    on = 0
    for t in range(T):
        W = W_of(orc64, pb, t)
        assert np.all((W > 0) <= base)
        np.testing.assert_allclose(W.sum(1), 1.0, atol=1e-15)
        np.testing.assert_array_equal(W, W.T)          # Metropolis: symmetric
        assert np.all(np.diag(W) > 0)
        on += ((W > 0).sum() - n) // 2
    frac = on / (T * n_edges)
    assert abs(frac - p) < 5 * math.sqrt(p * (1 - p) / (T * n_edges))


def test_uniform_rows_stochastic_irregular(orc64):
    pb = oracle.make_problem(12, 1, "exp", weights="uniform", edge_prob=0.5, seed=9)
    for t in range(30):
        nbr, w, deg = orc64.topology(pb, t)
        W = W_of(orc64, pb, t)
        np.testing.assert_allclose(W.sum(1), 1.0, atol=1e-15)
        for i in range(12):
            row = nbr[i, :deg[i] + 1]
            assert list(row) == sorted(row) and i in row
            assert np.all(w[i, :deg[i] + 1] == 1.0 / (deg[i] + 1))
