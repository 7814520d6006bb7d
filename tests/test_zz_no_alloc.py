"""The allocation-free consensus-error entry point.

gasloc_consensus_error_noalloc is for callers that cannot allocate device
memory where they need the consensus error (their framework owns all device
memory through its own pool, or cudaMalloc would synchronise a latency-critical
loop, or they are a plug-in handed pre-allocated buffers).  Through the C ABI,
it must give the value of the existing entry point, gasloc_consensus_error,
within the tolerance the other consensus-error comparisons use (relative
1e-12: same per-element arithmetic, fp64 sums in a different order), on
consecutive calls that reuse its static scratch.  This file is named so that
pytest collects it last.
"""
import numpy as np
import pytest

import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def test_noalloc_matches_existing_entry_point():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    torch.cuda.set_device(0)
    N, P = 8, 3 * 8192 + 1027          # several chunks and a ragged tail
    hp = g.make_hparams(**dict(wl.COMMON_HP, weights="metropolis", edge_prob=0.5))
    with g.Context(N, P, "exp", 77, hparams=hp) as ctx:
        stream = torch.cuda.current_stream()
        out = torch.empty(1, dtype=torch.float64, device="cuda")   # caller-owned output
        xptr, stride = ctx.buffer("x", 0)
        for rnd in range(3):
            ctx.local_steps(2)
            ctx.gossip_round()
            ref = ctx.consensus_error_now()          # existing entry point
            assert ref > 0
            for call in range(2):                    # two calls in a row
                out.fill_(-1.0)
                g.gasloc_consensus_error_noalloc(xptr, N, P, stride, out.data_ptr(), stream.cuda_stream)
                torch.cuda.synchronize()
                assert out.item() == pytest.approx(ref, rel=1e-12), (rnd, call)
        # sizes beyond the static scratch are refused before any device work
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_consensus_error_noalloc(xptr, N, 536870913, 536870916, out.data_ptr(),
                                             stream.cuda_stream)
        assert e.value.code == g.ENOMEM
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_consensus_error_noalloc(xptr + 4, N, P, stride, out.data_ptr(), stream.cuda_stream)
        assert e.value.code == g.EINVAL
