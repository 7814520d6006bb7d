"""Pins for the oracle's inner and outer updates.

Each test checks the oracle against something other than itself: a library
routine (torch.optim.AdamW / torch.optim.SGD on CPU), a closed form that the
paper's statements fix (exact averaging on the complete graph, mean
preservation, eigenmode decay, the accelerated-gossip recurrence's roots, the
1-Peer one-round contraction from Prop. 1), or a brute-force dense-matrix
iteration on tiny sizes.
"""
import math

import numpy as np
import pytest
import torch

import oracle

SEED = 0x6A510C


def pure_consensus(**kw):
    """lr = 0 and sigma = 0: the local step leaves y = x exactly."""
    kw.setdefault("lr", 0.0)
    kw.setdefault("noise_sigma", 0.0)
    kw.setdefault("weight_decay", 0.0)
    return kw


# --------------------------------------------------------------------------
# Inner optimizer
# --------------------------------------------------------------------------

def _torch_adamw_trajectory(o, pb, worker, nk, steps, x0, c, h):
    p = torch.tensor(x0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([p], lr=pb.lr, betas=(pb.beta1, pb.beta2), eps=pb.eps,
                            weight_decay=pb.weight_decay)
    ct = torch.tensor(c, dtype=torch.float64)
    ht = torch.tensor(h, dtype=torch.float64)
    for n in range(1, steps + 1):
        xi = torch.tensor([o.noise(pb.seed, worker, n, k) for k in range(nk)], dtype=torch.float64)
        with torch.no_grad():
            p.grad = ht * (p - ct) + pb.noise_sigma * xi
        opt.step()
    return p.detach().numpy()


def test_adamw_matches_torch_one_round(orc64):
    N, P, H = 3, 40, 7
    pb = oracle.make_problem(N, P, "none", seed=SEED, lr=3e-3, noise_sigma=0.05,
                             outer="sgd", outer_lr=1.0, outer_momentum=0.0)
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    st.local_steps(H)
    for i in range(N):
        ref = _torch_adamw_trajectory(orc64, pb, i, P, H, x0, c[i], h)
        np.testing.assert_allclose(st.get("y", i), ref, rtol=1e-12, atol=1e-15)


def test_adamw_state_persists_across_rounds(orc64):
    # No edges, SGD outer step with eta_out = 1: x <- x - (x - y) = y (up to one
    # rounding), so R rounds of H steps equal R*H uninterrupted AdamW steps
    # with the moments kept across rounds.
    N, P, H, R = 2, 24, 3, 4
    pb = oracle.make_problem(N, P, "none", seed=SEED + 1, lr=2e-3, noise_sigma=0.02,
                             outer="sgd", outer_lr=1.0, outer_momentum=0.0)
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    for _ in range(R):
        st.local_steps(H)
        st.gossip_round()
    for i in range(N):
        ref = _torch_adamw_trajectory(orc64, pb, i, P, R * H, x0, c[i], h)
        np.testing.assert_allclose(st.get("x", i), ref, rtol=1e-10, atol=1e-14)


def test_hparam_change_follows_torch_adamw(orc64):
    # No edges and an SGD outer step of 1 (x <- y each round): R rounds of H
    # steps are R*H AdamW steps.  Changing lr and both betas after the first
    # rounds matches torch.optim.AdamW with its parameter group changed at the
    # same step (bias corrections 1 - beta^n from the current betas).
    N, P, H, R1, R2 = 2, 16, 2, 2, 3
    kw = dict(seed=SEED + 5, lr=2e-3, noise_sigma=0.02, outer="sgd", outer_lr=1.0, outer_momentum=0.0)
    pb = oracle.make_problem(N, P, "none", **kw)
    pb2 = oracle.make_problem(N, P, "none", **dict(kw, lr=5e-3, beta1=0.8, beta2=0.99))
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    for _ in range(R1):
        st.local_steps(H)
        st.gossip_round()
    st.set_hparams(pb2)
    for _ in range(R2):
        st.local_steps(H)
        st.gossip_round()
    for i in range(N):
        p = torch.tensor(x0, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.AdamW([p], lr=pb.lr, betas=(pb.beta1, pb.beta2), eps=pb.eps,
                                weight_decay=pb.weight_decay)
        ct = torch.tensor(c[i], dtype=torch.float64)
        ht = torch.tensor(h, dtype=torch.float64)
        for n in range(1, (R1 + R2) * H + 1):
            if n == R1 * H + 1:
                opt.param_groups[0]["lr"] = pb2.lr
                opt.param_groups[0]["betas"] = (pb2.beta1, pb2.beta2)
            xi = torch.tensor([orc64.noise(pb.seed, i, n, k) for k in range(P)], dtype=torch.float64)
            with torch.no_grad():
                p.grad = ht * (p - ct) + pb.noise_sigma * xi
            opt.step()
        np.testing.assert_allclose(st.get("x", i), p.detach().numpy(), rtol=1e-10, atol=1e-14)


@pytest.mark.parametrize("T,frac,s0,f", [(100, 0.1, 0.01, 0.0), (37, 0.1, 0.01, 0.1), (20, 0.25, 0.05, 0.2)])
def test_lr_schedule_shape(orc64, T, frac, s0, f):
    # App. B: warm-up over the first 10% of the schedule starting at 1% of
    # the peak, then cosine decay.  Values the statement fixes: the first
    # step's rate, the peak after the warm-up, the final rate, the cosine's
    # midpoint, monotone warm-up and decay.
    lr = 3e-3
    pb = oracle.make_problem(2, 8, "none", lr=lr, lr_total_steps=T, lr_warmup_frac=frac,
                             lr_warmup_start=s0, lr_final_frac=f)
    W = int(round(frac * T))
    r = [orc64.sched_lr(pb, n) for n in range(1, T + 6)]
    assert r[0] == pytest.approx(s0 * lr, rel=1e-15)
    assert r[W] == pytest.approx(lr, rel=1e-15)                  # step W + 1
    assert all(b > a for a, b in zip(r[:W], r[1:W + 1]))       # warm-up rises
    assert all(b <= a for a, b in zip(r[W:], r[W + 1:]))       # then never rises
    for n in range(T, T + 6):
        assert r[n - 1] == pytest.approx(f * lr, rel=1e-12, abs=1e-18)
    if (T - W - 1) % 2 == 0:                                    # cosine midpoint
        n_mid = W + 1 + (T - W - 1) // 2
        assert r[n_mid - 1] == pytest.approx(lr * (1 + f) / 2, rel=1e-14)
    off = oracle.make_problem(2, 8, "none", lr=lr)              # T = 0: constant
    assert [orc64.sched_lr(off, n) for n in (1, 5, 1000)] == [lr, lr, lr]


def test_lr_schedule_enters_adamw_like_torch(orc64):
    # No edges and an SGD outer step of 1: the rounds are one AdamW trajectory.
    # torch.optim.AdamW with its group's lr set to each step's scheduled rate
    # (step size and decoupled weight decay both scale with it) must match.
    N, P, H, R, T = 2, 12, 3, 6, 14
    kw = dict(seed=SEED + 9, lr=4e-3, noise_sigma=0.02, outer="sgd", outer_lr=1.0, outer_momentum=0.0,
              lr_total_steps=T, lr_warmup_frac=0.2, lr_final_frac=0.1)
    pb = oracle.make_problem(N, P, "none", **kw)
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    for _ in range(R):
        st.local_steps(H)
        st.gossip_round()
    for i in range(N):
        p = torch.tensor(x0, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.AdamW([p], lr=pb.lr, betas=(pb.beta1, pb.beta2), eps=pb.eps,
                                weight_decay=pb.weight_decay)
        ct = torch.tensor(c[i], dtype=torch.float64)
        ht = torch.tensor(h, dtype=torch.float64)
        for n in range(1, R * H + 1):
            opt.param_groups[0]["lr"] = orc64.sched_lr(pb, n)
            xi = torch.tensor([orc64.noise(pb.seed, i, n, k) for k in range(P)], dtype=torch.float64)
            with torch.no_grad():
                p.grad = ht * (p - ct) + pb.noise_sigma * xi
            opt.step()
        np.testing.assert_allclose(st.get("x", i), p.detach().numpy(), rtol=1e-10, atol=1e-14)


def test_adamw_first_step_closed_form(orc64):
    # n = 1: m_hat = g, v_hat = g^2, so y1 = y0 (1 - lr wd) - lr g / (|g| + eps)
    N, P = 2, 64
    pb = oracle.make_problem(N, P, "none", seed=SEED + 2, lr=1e-3, noise_sigma=0.01)
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    st.local_steps(1)
    for i in range(N):
        xi = np.array([orc64.noise(pb.seed, i, 1, k) for k in range(P)])
        g = h * (x0 - c[i]) + pb.noise_sigma * xi
        # eps enters as sqrt(v_hat) + eps with v_hat = g^2 (bias-corrected)
        ref = x0 * (1 - pb.lr * pb.weight_decay) - pb.lr * g / (np.abs(g) + pb.eps)
        np.testing.assert_allclose(st.get("y", i), ref, rtol=1e-12, atol=1e-16)
        assert st.steps_taken(i) == 1


def test_per_worker_curvature_and_heterogeneous_steps(orc64):
    N, P = 4, 16
    pb = oracle.make_problem(N, P, "none", seed=SEED, per_worker_h=True, lr=1e-3)
    st = orc64.state(pb)
    h = st.get_all("h")
    assert h.shape == (N, P) and not np.allclose(h[0], h[1])
    x0 = st.get("x", 0)
    Hi = np.array([0, 1, 3, 2], np.int32)
    st.local_steps(0, Hi)
    for i in range(N):
        assert st.steps_taken(i) == Hi[i]
        ref = _torch_adamw_trajectory(orc64, pb, i, P, int(Hi[i]), x0, st.get("c", i), h[i])
        if Hi[i] == 0:
            np.testing.assert_array_equal(st.get("y", i), x0)   # untouched
        else:
            np.testing.assert_allclose(st.get("y", i), ref, rtol=1e-12, atol=1e-15)


def test_zero_step_worker_sends_x(orc64):
    # y_i^{(t)} = x_i^{(t, H_i)} = x_i^{(t)} when H_i = 0 (Algorithm 1)
    N, P = 4, 8
    pb = oracle.make_problem(N, P, "complete", seed=1, outer="sgd", outer_lr=1.0, lr=1e-2)
    st = orc64.state(pb)
    st.local_steps(1)
    st.gossip_round()                 # round 0: everyone fresh
    x = st.get_all("x")
    st.local_steps(0, np.array([1, 0, 1, 1], np.int32))
    y = st.get_all("y")
    y[1] = x[1]
    st.gossip_round()
    np.testing.assert_allclose(st.get_all("x"), np.tile(y.mean(0), (N, 1)), rtol=1e-14)


# --------------------------------------------------------------------------
# Outer optimizer and gossip
# --------------------------------------------------------------------------

def test_complete_graph_exact_averaging(orc64):
    # Lambda = pi recovers DiLoCo; with SGD(eta_out = 1) one round averages exactly
    N, P = 6, 50
    pb = oracle.make_problem(N, P, "complete", seed=3, outer="sgd", outer_lr=1.0, lr=5e-3)
    st = orc64.state(pb)
    st.local_steps(2)
    y = st.get_all("y")
    st.gossip_round()
    np.testing.assert_allclose(st.get_all("x"), np.tile(y.mean(0), (N, 1)), rtol=1e-14, atol=1e-17)
    assert st.consensus_error() < 1e-28


@pytest.mark.parametrize("outer,nesterov,mom", [("nesterov", True, 0.9), ("sgdm", False, 0.7),
                                                ("sgd", False, 0.0)])
def test_complete_graph_is_diloco(orc64, outer, nesterov, mom):
    # On the complete graph every x_i stays equal to one DiLoCo replica whose
    # outer gradient is x - mean_j(y_j), stepped by torch.optim.SGD.
    N, P, H, R, lr_out = 4, 30, 3, 5, 0.7
    pb = oracle.make_problem(N, P, "complete", seed=4, outer=outer, outer_lr=lr_out,
                             outer_momentum=mom, lr=3e-3)
    st = orc64.state(pb)
    xr = torch.tensor(st.get("x", 0), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([xr], lr=lr_out, momentum=mom, nesterov=nesterov)
    for _ in range(R):
        st.local_steps(H)
        ybar = st.get_all("y").mean(0)
        st.gossip_round()
        with torch.no_grad():
            xr.grad = xr - torch.tensor(ybar, dtype=torch.float64)
        opt.step()
        for i in range(N):
            np.testing.assert_allclose(st.get("x", i), xr.detach().numpy(), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("topo,kw", [
    ("ring", {}), ("exp", {}), ("torus", {"torus": (2, 4), "weights": "metropolis"}),
    ("matching", {}), ("2peer", {"weights": "lazy"}),
    ("exp", {"weights": "metropolis", "edge_prob": 0.5}),
])
@pytest.mark.parametrize("outer", ["sgd", "nesterov"])
def test_mean_preserved_doubly_stochastic(orc64, topo, kw, outer):
    # 1^T Lambda = 0 => xbar_{t+1} = xbar_t + eta gbar_t; with no local progress
    # (pure consensus) the replica mean never moves.
    N, P = 8, 40
    pb = oracle.make_problem(N, P, topo, seed=5, outer=outer, outer_lr=0.8, outer_momentum=0.9,
                             **pure_consensus(**kw))
    st = orc64.state(pb)
    rng = np.random.default_rng(0)
    for i in range(N):
        st.set("x", i, rng.normal(size=P))
    m0 = st.get_all("x").mean(0)
    for _ in range(6):
        st.local_steps(1)
        st.gossip_round()
    np.testing.assert_allclose(st.get_all("x").mean(0), m0, atol=1e-13)
    assert st.consensus_error() > 0


@pytest.mark.parametrize("alpha", [1.0, 0.6])
def test_ring_eigenmode_decay(orc64, alpha):
    # x <- (I - alpha Lambda) x with W = I - Lambda the uniform ring:
    # mode q decays by 1 - alpha (1 - (1/3 + 2/3 cos(2 pi q / N))) per round.
    N, P, q = 8, 3, 2
    pb = oracle.make_problem(N, P, "ring", outer="sgd", outer_lr=alpha, **pure_consensus())
    st = orc64.state(pb)
    phase = np.array([0.0, 0.3, 1.1])
    for i in range(N):
        st.set("x", i, np.cos(2 * math.pi * q * i / N + phase))
    lam = 1 / 3 + 2 / 3 * math.cos(2 * math.pi * q / N)
    f = 1 - alpha * (1 - lam)
    for r in range(1, 8):
        st.local_steps(1)
        st.gossip_round()
        for i in range(N):
            np.testing.assert_allclose(st.get("x", i), f ** r * np.cos(2 * math.pi * q * i / N + phase),
                                       atol=1e-14)


@pytest.mark.parametrize("alpha,gamma", [(1.0, 0.5), (0.7, 0.3), (0.9, 0.0)])
def test_eq2_eigenmode_recurrence_roots(orc64, alpha, gamma):
    # Eq. 2 on a fixed graph, pure consensus: mode amplitude a_t solves
    # r^2 - (1 + gamma - alpha lam) r + gamma = 0 (proof of the gossip lemma,
    # part iii) with a_1 = (1 - alpha lam) a_0 (no momentum term at t = 0).
    N, q, T = 8, 1, 25
    pb = oracle.make_problem(N, 1, "ring", outer="eq2", eta=1.0, alpha=alpha, gamma=gamma,
                             **pure_consensus())
    st = orc64.state(pb)
    v = np.cos(2 * math.pi * q * np.arange(N) / N)
    for i in range(N):
        st.set("x", i, v[i:i + 1])
    lam = 1 - (1 / 3 + 2 / 3 * math.cos(2 * math.pi * q / N))   # eigenvalue of I - W
    r = np.roots([1.0, -(1 + gamma - alpha * lam), gamma]).astype(complex)
    a0, a1 = 1.0, 1 - alpha * lam
    if abs(r[0] - r[1]) > 1e-9:
        A = np.linalg.solve(np.array([[1, 1], [r[0], r[1]]]), np.array([a0, a1]))
        amp = [np.real(A[0] * r[0] ** t + A[1] * r[1] ** t) for t in range(T + 1)]
    else:
        rr = r[0]
        B = (a1 - rr) / rr
        amp = [np.real((1 + B * t) * rr ** t) for t in range(T + 1)]
    for t in range(1, T + 1):
        st.local_steps(1)
        st.gossip_round()
        np.testing.assert_allclose(st.get_all("x")[:, 0], amp[t] * v, atol=1e-12)


def test_accelerated_gamma_contracts_at_predicted_rate(orc64):
    # gamma = (1 - sqrt(alpha/chi))^2 gives |r| <= 1 - sqrt(alpha/chi) on every
    # disagreement mode (gossip lemma iii); Eq. 1 (gamma = 0) contracts slower.
    N, alpha = 16, 1.0
    W = orc64.dense_w(oracle.make_problem(N, 1, "ring"), 0)
    ev = np.sort(np.linalg.eigvalsh(np.eye(N) - W))
    chi = 1 / ev[1]
    q = 1 - math.sqrt(alpha / chi)
    gamma = q ** 2
    rng = np.random.default_rng(2)
    x0 = rng.normal(size=(N, 4))
    ce = {}
    for g in (0.0, gamma):
        pb = oracle.make_problem(N, 4, "ring", outer="eq2", eta=1.0, alpha=alpha, gamma=g,
                                 **pure_consensus())
        st = orc64.state(pb)
        for i in range(N):
            st.set("x", i, x0[i])
        hist = []
        for _ in range(120):
            st.local_steps(1)
            st.gossip_round()
            hist.append(st.consensus_error())
        ce[g] = hist
    # sqrt(CE) decays no slower than q^t (times a polynomial factor for the
    # double root) and beats plain gossip
    rate = (ce[gamma][119] / ce[gamma][59]) ** (1 / 120)
    assert rate <= q * 1.02
    assert ce[gamma][119] < ce[0.0][119]


def test_one_peer_expected_contraction(orc64):
    # E ||pi x+||^2 = (1 - alpha n/(n-1) + alpha^2 n/(2(n-1))) ||pi x||^2 for
    # the random matching (from E[Lambda] = E[Lambda^2] = n/(2(n-1)) pi).
    N, P, alpha, T = 16, 8, 1.0, 400
    pred = 1 - alpha * N / (N - 1) + alpha ** 2 * N / (2 * (N - 1))
    pb = oracle.make_problem(N, P, "matching", seed=21, outer="sgd", outer_lr=alpha,
                             **pure_consensus())
    rng = np.random.default_rng(5)
    st = orc64.state(pb)
    ratios = []
    for t in range(T):
        if t % 40 == 0:
            for i in range(N):
                st.set("x", i, rng.normal(size=P))
        c0 = st.consensus_error()
        st.local_steps(1)
        st.gossip_round()
        ratios.append(st.consensus_error() / c0)
    ratios = np.array(ratios)
    se = ratios.std() / math.sqrt(T)
    assert abs(ratios.mean() - pred) < 4 * se + 1e-3


def test_local_dadam_reduces_to_dadam(orc64):
    # App. C: with H = 1 and an SGD outer step of unit rate, Local-DAdam is DAdam
    N, P = 6, 20
    common = dict(seed=8, lr=4e-3, weights="metropolis", edge_prob=0.7)
    a = orc64.state(oracle.make_problem(N, P, "exp", outer="dadam", **common))
    b = orc64.state(oracle.make_problem(N, P, "exp", outer="local_dadam", outer_lr=1.0,
                                        outer_momentum=0.0, **common))
    for _ in range(5):
        for st in (a, b):
            st.local_steps(1)
            st.gossip_round()
        np.testing.assert_allclose(a.get_all("x"), b.get_all("x"), rtol=1e-13, atol=1e-16)


def test_consensus_error_closed_form(orc64):
    # x_ik = i: xbar = (N-1)/2, CE = (1/N) sum_i (i - xbar)^2 * P = P (N^2-1)/12
    N, P = 7, 33
    st = orc64.state(oracle.make_problem(N, P, "ring"))
    for i in range(N):
        st.set("x", i, np.full(P, float(i)))
    assert st.consensus_error() == pytest.approx(P * (N * N - 1) / 12, rel=1e-15)
    st2 = orc64.state(oracle.make_problem(N, P, "ring"))
    assert st2.consensus_error() < 1e-30          # identical initial replicas


def test_average_is_network_mean(orc64):
    N, P = 5, 9
    st = orc64.state(oracle.make_problem(N, P, "ring", seed=2, lr=1e-2))
    st.local_steps(2)
    st.gossip_round()
    np.testing.assert_allclose(st.average(), st.get_all("x").mean(0), rtol=1e-15)


# --------------------------------------------------------------------------
# Brute force: dense N x N matrix iteration on tiny sizes
# --------------------------------------------------------------------------

def _dense_round(W, X, Y, B, mode, eta_out, mu, eta, alpha, gamma, first):
    if mode == "eq2":
        Z = X + eta * (Y - X)
        Zp = Z if first else B
        return (1 - alpha) * Z + alpha * (W @ Z) + gamma * (Z - Zp), Z
    if mode == "dadam":
        return W @ X + (Y - X), B
    if mode == "local_dadam":
        D = X - W @ X
        Bn = mu * B + D
        return Y - eta_out * (D + mu * Bn), Bn
    D = X - W @ Y
    if mode == "sgd":
        return X - eta_out * D, B
    Bn = mu * B + D
    if mode == "sgdm":
        return X - eta_out * Bn, Bn
    return X - eta_out * (D + mu * Bn), Bn


@pytest.mark.parametrize("mode", ["sgd", "sgdm", "nesterov", "eq2", "dadam", "local_dadam"])
@pytest.mark.parametrize("topo,kw", [("ring", {}), ("matching", {}),
                                     ("exp", {"weights": "uniform", "edge_prob": 0.6}),
                                     ("2peer", {"weights": "lazy"})])
def test_bruteforce_dense_matrix(orc64, mode, topo, kw):
    N, P, R = 6, 17, 6
    pb = oracle.make_problem(N, P, topo, seed=31, outer=mode, outer_lr=0.8, outer_momentum=0.6,
                             eta=0.9, alpha=0.8, gamma=0.2, lr=5e-3, **kw)
    st = orc64.state(pb)
    X = st.get_all("x")
    B = np.zeros_like(X)
    for t in range(R):
        st.local_steps(2)
        Y = st.get_all("y")
        W = orc64.dense_w(pb, t)
        X, B = _dense_round(W, X, Y, B, mode, pb.outer_lr, pb.outer_momentum, pb.eta,
                            pb.alpha, pb.gamma, t == 0)
        st.gossip_round()
        np.testing.assert_allclose(st.get_all("x"), X, rtol=1e-12, atol=1e-14)
        if mode not in ("sgd", "dadam"):
            np.testing.assert_allclose(st.get_all("b"), B, rtol=1e-12, atol=1e-14)
        # keep the dense iterate on the oracle's trajectory (y depends on x)
        X = st.get_all("x")
        B = st.get_all("b")


def test_f32_build_tracks_f64(orc32, orc64):
    # The fp32 parity build is the same algorithm with one fp32 rounding per
    # operation: it stays within the parity tolerance 1e-5 (1 + |x|) of the
    # double build over a multi-round run.  Indices whose first gradient is
    # within 1e-6 of 0 are excluded: there the first AdamW step is lr*sign(g)
    # and a last-bit difference flips it.
    N, P, R = 4, 4099, 20
    pb = oracle.make_problem(N, P, "ring", seed=SEED, lr=3e-4, noise_sigma=0.01,
                             outer="nesterov", outer_lr=0.7, outer_momentum=0.9)
    a, b = orc32.state(pb), orc64.state(pb)
    x0, c, h = b.get("x", 0), b.get_all("c"), b.get("h", 0)
    g1 = np.stack([h * (x0 - c[i]) + 0.01 * np.array([orc64.noise(pb.seed, i, 1, k) for k in range(P)])
                   for i in range(N)])
    ok = np.all(np.abs(g1) > 1e-6, axis=0)
    for _ in range(R):
        for st in (a, b):
            st.local_steps(1)
            st.gossip_round()
    xa, xb = a.get_all("x")[:, ok], b.get_all("x")[:, ok]
    assert np.all(np.abs(xa - xb) <= 1e-5 * (1 + np.abs(xb)))
    assert a.consensus_error() == pytest.approx(b.consensus_error(), rel=1e-3)
