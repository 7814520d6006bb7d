"""Failure detection on the GPU without faulting it: a wait that can never be
satisfied expires within its limit, is reported as GASLOC_EDEVICE by the next
synchronising call, and leaves the context usable (the following rounds still
match the oracle)."""
import time

import numpy as np
import pytest

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild

from _pairs import make_pair

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_and_context_survives():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    oracle.build()
    ctx, st = make_pair(8, 5000, "exp", seed=3, hp=dict(lr=2e-3))
    with ctx:
        ctx.local_steps(1)
        ctx.gossip_round()
        st.local_steps(1)
        st.gossip_round()
        t0 = time.perf_counter()
        rc = g.gasloc_selftest_bounded_wait(ctx.h, 20_000_000)      # 20 ms limit
        el = time.perf_counter() - t0
        assert rc == g.EDEVICE, g.gasloc_last_error()
        assert "timed out" in g.gasloc_last_error()
        assert el < 5.0
        # the flag was cleared and the context still works
        for _ in range(2):
            ctx.local_steps(1)
            ctx.gossip_round()
            st.local_steps(1)
            st.gossip_round()
        assert ctx.consensus_error() == pytest.approx(st.consensus_error(), rel=1e-5)
        np.testing.assert_array_equal(ctx.read_all("x"), st.get_all("x").astype(np.float32))
        with pytest.raises(g.GaslocError):
            g._check(g.gasloc_selftest_bounded_wait(ctx.h, 0))      # limit out of range
