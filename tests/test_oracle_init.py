"""Pins for the oracle's initial state (oc_create).

The initial state composes the pinned generators into the workload: every
worker starts from the same x_0 (Prop. 2 assumes equal initial replicas) drawn
with standard deviation 0.02 (the workloads' "N(0, 0.02)"), each worker has its
own quadratic centre c_i ~ N(0, 1), the curvature h ~ U(0.1, 1) is shared or
per worker, and the optimizer state starts at zero.  The checks below are the
statistics those statements fix, at a size (about 40 k parameters) where a
wrong scale, tag or worker index in the composition moves a statistic by many
standard errors: x_0 at std 0.2, c_i drawn with worker 0's index (every c_i
equal), x_0 drawn from the centres' stream (x_0 proportional to c_0), h from
the centres' stream (correlated with c_0, out of [0.1, 1)).
"""
import numpy as np
import pytest

import oracle

P = 40_000


def _state(orc, n, per_h, storage="f32", kidx=None, seed=0x5EED):
    pb = oracle.make_problem(n, P, "ring", seed=seed, per_worker_h=per_h, storage=storage)
    return orc.state(pb, kidx)


def _corr(a, b):
    a = a - a.mean()
    b = b - b.mean()
    return float((a * b).sum() / np.sqrt((a * a).sum() * (b * b).sum()))


def _excess_kurtosis(v):
    d = v - v.mean()
    return float((d ** 4).mean() / (d ** 2).mean() ** 2 - 3.0)


@pytest.mark.parametrize("per_h", [False, True])
def test_initial_replicas_identical_with_std_002(orc64, per_h):
    st = _state(orc64, 6, per_h)
    x, y = st.get_all("x"), st.get_all("y")
    # equal initial replicas (Prop. 2), y starts at x
    assert (x == x[0]).all()
    assert np.array_equal(y, x)
    x0 = x[0]
    # "N(0, 0.02)" read as a standard deviation of 0.02: the standard error of
    # the sample std at 40 k draws is 0.35%, so 3% is about 8 standard errors
    assert abs(x0.std() / 0.02 - 1.0) < 0.03
    assert abs(x0.mean()) < 4 * 0.02 / np.sqrt(P)
    # the Irwin-Hall(4) stand-in for the normal: excess kurtosis -0.3
    assert abs(_excess_kurtosis(x0 / 0.02) + 0.3) < 0.1
    # x_0 is drawn from its own stream, not from any worker's centre
    c = st.get_all("c")
    for i in range(c.shape[0]):
        assert abs(_corr(x0, c[i])) < 0.03, i


@pytest.mark.parametrize("per_h", [False, True])
def test_centres_per_worker_unit_normal(orc64, per_h):
    n = 8
    st = _state(orc64, n, per_h)
    c = st.get_all("c")
    assert c.shape == (n, P)
    for i in range(n):
        assert abs(c[i].mean()) < 4.0 / np.sqrt(P), i
        assert abs(c[i].var() - 1.0) < 0.03, i
        assert abs(_excess_kurtosis(c[i]) + 0.3) < 0.1, i
    # each worker has its own centre: pairwise correlations at the noise level
    # (standard error 1/sqrt(P) = 0.005)
    for i in range(n):
        for j in range(i + 1, n):
            assert abs(_corr(c[i], c[j])) < 0.03, (i, j)


@pytest.mark.parametrize("per_h", [False, True])
def test_curvature_uniform_range_and_sharing(orc64, per_h):
    n = 5
    st = _state(orc64, n, per_h)
    h = st.get_all("h")
    assert h.shape == ((n if per_h else 1), P)
    assert h.min() >= 0.1 and h.max() < 1.0
    sd = 0.9 / np.sqrt(12.0)
    for i in range(h.shape[0]):
        assert abs(h[i].mean() - 0.55) < 4 * sd / np.sqrt(P), i
        assert abs(h[i].std() / sd - 1.0) < 0.03, i
    c = st.get_all("c")
    for i in range(h.shape[0]):
        # not drawn from a centre's stream
        for j in range(n):
            assert abs(_corr(h[i], c[j])) < 0.03, (i, j)
    if per_h:
        for i in range(n):
            for j in range(i + 1, n):
                assert abs(_corr(h[i], h[j])) < 0.03, (i, j)


@pytest.mark.parametrize("per_h", [False, True])
def test_streams_share_no_draws(orc64, per_h):
    # Each normal at index k sums the 24-bit draws at counters 4k..4k+3 of its
    # stream, while the curvature at index k takes the single draw at counter
    # k.  If h were drawn from the x_0 or a centre's stream, h at 4k'+j would
    # be one of the four summands of that normal at k' (correlation 1/2).
    n = 5
    st = _state(orc64, n, per_h)
    h, c, x0 = st.get_all("h"), st.get_all("c"), st.get_all("x")[0]
    kq = P // 4
    normals = [x0[:kq]] + [c[i, :kq] for i in range(n)]
    for hi in range(h.shape[0]):
        for j in range(4):
            hs = h[hi, j::4][:kq]
            for q, z in enumerate(normals):
                assert abs(_corr(hs, z)) < 0.06, (hi, j, q)


def test_optimizer_state_starts_at_zero(orc64):
    st = _state(orc64, 4, True)
    for w in ("m", "v", "b"):
        assert not st.get_all(w).any(), w
    assert st.round == 0
    assert all(st.steps_taken(i) == 0 for i in range(4))
    assert st.consensus_error() == 0.0


def test_draws_depend_on_global_index_only(orc64):
    # a state held for a subset of indices (a P-range, or a sample) holds the
    # same values as the full state at those indices
    full = _state(orc64, 3, True)
    kidx = np.concatenate([np.arange(1000, 1500), np.arange(P - 37, P), [5, 17]]).astype(np.int64)
    part = _state(orc64, 3, True, kidx=kidx)
    for w in ("x", "c", "h"):
        np.testing.assert_array_equal(part.get_all(w), full.get_all(w)[:, kidx], err_msg=w)


def test_seed_changes_every_draw(orc64):
    a, b = _state(orc64, 3, True, seed=1), _state(orc64, 3, True, seed=2)
    for w in ("x", "c", "h"):
        va, vb = a.get_all(w), b.get_all(w)
        assert (va != vb).mean() > 0.99, w
        assert abs(_corr(va.ravel(), vb.ravel())) < 0.03, w


def test_bf16_store_rounds_the_same_draws(orc32):
    # with a bf16 store every initial value is the fp32 draw rounded to bf16
    s32 = _state(orc32, 3, True)
    s16 = _state(orc32, 3, True, storage="bf16")
    import torch
    for w in ("x", "c", "h"):
        ref = torch.from_numpy(s32.get_all(w).astype(np.float32)).to(torch.bfloat16).float().numpy()
        np.testing.assert_array_equal(s16.get_all(w).astype(np.float32), ref, err_msg=w)
