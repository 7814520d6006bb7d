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

from _pairs import make_pair, assert_ce

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
        assert_ce(ctx.consensus_error(), st)
        np.testing.assert_array_equal(ctx.read_all("x"), st.get_all("x").astype(np.float32))
        with pytest.raises(g.GaslocError):
            g._check(g.gasloc_selftest_bounded_wait(ctx.h, 0))      # limit out of range


def test_misaligned_allocator_block_is_refused():
    # An allocator hook that returns blocks 16 bytes past a 256-byte boundary:
    # gasloc_start hands each block back and fails with EINVAL before any
    # kernel could address it.
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    dev = torch.cuda.current_device()
    live = {}

    def _alloc(nbytes, stream, user):
        base = torch.cuda.caching_allocator_alloc(int(nbytes) + 256, dev, stream if stream else 0)
        live[base + 16] = base
        return base + 16

    def _free(ptr, stream, user):
        torch.cuda.caching_allocator_delete(live.pop(ptr))

    af, ff = g.ALLOC_FN(_alloc), g.FREE_FN(_free)
    h = g.gasloc_init(4, 5000, "ring", 1)
    try:
        g.gasloc_set_allocator(h, af, ff, None)
        with pytest.raises(g.GaslocError) as ei:
            g.gasloc_start(h)
        assert ei.value.code == g.EINVAL and "256-byte aligned" in str(ei.value)
        assert not live                       # every block went back
    finally:
        g.gasloc_destroy(h)
