"""Pins for the oracle's bfloat16 storage rule: every stored value is the
binary32 result rounded to bfloat16, nearest with ties to even.  The rounding
is checked against torch's float32 -> bfloat16 conversion (a library routine),
including ties, overflow and subnormals; a bf16 run must hold only
bf16-representable values and stay within bf16 resolution of the fp32 run."""
import numpy as np
import pytest
import torch

import oracle


def _torch_bf16(vals):
    return torch.tensor(vals, dtype=torch.float32).to(torch.bfloat16).to(torch.float32).numpy()


def test_bf16_round_matches_torch(orc32):
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        rng.normal(size=4000).astype(np.float32),
        (rng.normal(size=2000) * 1e-30).astype(np.float32),         # tiny / subnormal range
        (rng.normal(size=2000) * 1e30).astype(np.float32),
        np.array([0.0, -0.0, 1.0, -1.0, 3.0e38, -3.39e38, 1e-45, np.finfo(np.float32).max,
                  np.float32(1.0) + np.float32(2.0 ** -8),                  # tie -> even (1.0)
                  np.float32(1.0) + np.float32(3 * 2.0 ** -8),              # tie -> even (up)
                  np.float32(1.0) + np.float32(2.0 ** -8) + np.float32(2.0 ** -20),
                  np.inf, -np.inf], np.float32),
    ]).astype(np.float32)
    ours = np.array([orc32.bf16_round(float(v)) for v in vals], np.float32)
    np.testing.assert_array_equal(ours, _torch_bf16(vals))
    assert np.isnan(orc32.bf16_round(float("nan")))


def test_bf16_run_stores_bf16_values(orc32):
    N, P = 6, 777
    pb = oracle.make_problem(N, P, "exp", seed=5, storage="bf16", weights="metropolis", lr=3e-3)
    st = orc32.state(pb)
    for _ in range(4):
        st.local_steps(2)
        st.gossip_round()
    for w in ("x", "y", "m", "v", "b", "c", "h"):
        a = st.get_all(w).astype(np.float32)
        low = a.view(np.uint32) & 0xFFFF
        assert not low.any(), w


def test_bf16_run_tracks_f32_run(orc32):
    N, P, R = 8, 2000, 5

    def run(storage, sigma):
        s = orc32.state(oracle.make_problem(N, P, "exp", storage=storage, seed=11, lr=3e-4, noise_sigma=sigma))
        for _ in range(R):
            s.local_steps(1)
            s.gossip_round()
        return s

    # Without noise both stores solve the same problem: bf16 keeps 8
    # significant bits, so after R rounds the replicas agree to a few bf16
    # steps of the largest value.
    a, b = run("bf16", 0.0), run("f32", 0.0)
    xa, xb = a.get_all("x"), b.get_all("x")
    assert np.abs(xa - xb).max() <= R * 2 ** -8 * np.abs(xb).max()
    # With noise the stores draw it on different grids (16 and 24 bits), so
    # only the statistics agree: the disagreement between replicas (~1e-4 per
    # element here) is of the order of one bf16 step, and the consensus errors
    # agree roughly.
    a, b = run("bf16", 0.01), run("f32", 0.01)
    assert 0.5 < a.consensus_error() / b.consensus_error() < 2.0


def _bf16_of(t):
    # the oracle's rule for a REAL result: to binary32, then to bfloat16
    return t.float().to(torch.bfloat16).to(torch.float64)


def test_bf16_adamw_matches_torch_with_bf16_rounding(orc64):
    # H AdamW steps with a bf16 store against torch.optim.AdamW in fp64 whose
    # parameter and both moment buffers are rounded to bf16 after every step,
    # with the gradient noise of the bf16 grid.  The two sides order their
    # fp64 operations differently, so a value that lands on a bf16 rounding
    # boundary may round the other way: at most one bf16 step apart, rarely.
    N, P, H = 2, 600, 3
    pb = oracle.make_problem(N, P, "none", seed=77, lr=3e-3, noise_sigma=0.05, outer="sgd",
                             outer_lr=1.0, outer_momentum=0.0, storage="bf16")
    st = orc64.state(pb)
    x0, c, h = st.get("x", 0), st.get_all("c"), st.get("h", 0)
    st.local_steps(H)
    for i in range(N):
        p = torch.tensor(x0, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.AdamW([p], lr=pb.lr, betas=(pb.beta1, pb.beta2), eps=pb.eps,
                                weight_decay=pb.weight_decay)
        ct, ht = torch.tensor(c[i], dtype=torch.float64), torch.tensor(h, dtype=torch.float64)
        for n in range(1, H + 1):
            xi = torch.tensor([orc64.noise(pb.seed, i, n, k, "bf16") for k in range(P)], dtype=torch.float64)
            with torch.no_grad():
                p.grad = ht * (p - ct) + pb.noise_sigma * xi
            opt.step()
            with torch.no_grad():
                p.copy_(_bf16_of(p))
                s = opt.state[p]
                s["exp_avg"].copy_(_bf16_of(s["exp_avg"]))
                s["exp_avg_sq"].copy_(_bf16_of(s["exp_avg_sq"]))
        s = opt.state[p]
        for name, ref in (("y", p.detach()), ("m", s["exp_avg"]), ("v", s["exp_avg_sq"])):
            got, ref = st.get(name, i), ref.numpy()
            diff = got != ref
            ulp = np.abs(ref) * 2.0 ** -7
            assert np.all(np.abs(got - ref)[diff] <= ulp[diff] * 1.0001), name
            assert diff.mean() <= 0.01, (name, diff.mean())
