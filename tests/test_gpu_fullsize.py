"""Every workload at its full size and round count, checked on sampled
parameter indices.

Each step is element-wise in the parameter index (the synthetic gradient is
diagonal; mixing is across workers at one index), so the oracle can follow the
complete trajectory of any chosen indices on its own.  The GPU runs the whole
replica store in the launch configuration bench.py times; the sampled indices
(tile and tensor boundaries, the ragged ends, random picks) must match the
oracle within the parity bound (and, by the shared fp32 operation order, bit
for bit).  The fused consensus error must equal the standalone reduction.
"""
import numpy as np
import pytest

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

from _pairs import within_tol, workload_pair

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    yield


def sample_indices(w, n_random=1500, seed=0):
    P = w.n_params
    rng = np.random.default_rng(seed)
    pts = {0, 1, 2, 3, 4, 5, P - 1, P - 2, P - 3, P - 4, P // 2}
    for t in (1024, 256, 512):                         # tile edges of both kernels
        for k in (1, 2, 7, 1000):
            pts.update({k * t - 1, k * t})
    if w.numels:                                       # tensor boundaries
        off = 0
        for n in w.numels:
            pts.update({off, off + n - 1})
            off += n
    pts.update(int(v) for v in rng.integers(0, P, n_random))
    return np.array(sorted(p for p in pts if 0 <= p < P), np.int64)


@pytest.mark.parametrize("name", list(wl.WORKLOADS))
def test_workload_full_size_sampled(name):
    import torch
    w = wl.WORKLOADS[name]
    kidx = sample_indices(w)
    _, (ctx, st) = workload_pair(name, kidx)
    try:
        Hi = None
        if w.H < 0:
            Hi = g.gasloc_get_local_steps(ctx.h, w.n_workers)
            np.testing.assert_array_equal(Hi, oracle.get("f32").draw_local_steps(w.seed, w.n_workers,
                                                                                 w.draw_hmax))
        H = w.H if w.H > 0 else g.PER_WORKER_STEPS
        for r in range(w.rounds):
            ctx.local_steps(H)
            ctx.gossip_round()
            st.local_steps(w.H if w.H > 0 else 0, Hi)
            st.gossip_round()
        ce_fused = ctx.consensus_error()
        ce_now = ctx.consensus_error_now()
        assert ce_fused == pytest.approx(ce_now, rel=1e-12) and ce_fused > 0
        for which in ("x", "b", "m", "v"):
            for i in range(w.n_workers):
                a = ctx.gather(which, i, kidx)
                b = st.get(which, i)
                ok = within_tol(a, b)
                assert ok.all(), "%s[%d]: %d of %d outside the bound" % (which, i, (~ok).sum(), ok.size)
                assert np.array_equal(a, b.astype(np.float32)), "%s[%d] not bit-identical" % (which, i)
        for i in range(w.n_workers):
            assert ctx.steps_taken(i) == st.steps_taken(i)
    finally:
        ctx.close()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()


def test_maximum_replica_size():
    # n_params at its limit (2^31 - 1): worker offsets exceed 2^32 floats and
    # element coordinates reach the top of int32; checked on the last tiles.
    import torch
    P, N = 2 ** 31 - 1, 2
    free, _ = torch.cuda.mem_get_info()
    need = (6 * N + 1) * (P + 64) * 4
    if free < need + (8 << 30):
        pytest.skip("not enough device memory for the maximum size")
    kidx = np.array([0, 1, 1023, 1024, 2 ** 30, 2 ** 31 - 1025, 2 ** 31 - 1024, 2 ** 31 - 257,
                     2 ** 31 - 256, 2 ** 31 - 5, 2 ** 31 - 4, 2 ** 31 - 3, 2 ** 31 - 2], np.int64)
    from _pairs import make_pair
    ctx, st = make_pair(N, P, "ring", seed=91, hp=dict(lr=1e-3), kidx=kidx)
    try:
        for _ in range(2):
            ctx.local_steps(2)
            ctx.gossip_round()
            st.local_steps(2)
            st.gossip_round()
        for which in ("x", "b", "m", "v", "y"):
            for i in range(N):
                a = ctx.gather(which, i, kidx)
                b = st.get(which, i).astype(np.float32)
                np.testing.assert_array_equal(a, b, err_msg="%s[%d]" % (which, i))
        # a 2-node ring is the complete graph: both replicas receive the same mix
        # from identical starting points, so they stay equal (exact consensus)
        assert ctx.consensus_error() == 0.0
        assert np.array_equal(ctx.gather("x", 0, kidx), ctx.gather("x", 1, kidx))
    finally:
        ctx.close()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
