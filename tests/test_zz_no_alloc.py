"""The allocation-free consensus-error entry point.

gasloc_consensus_error_noalloc is for callers that cannot allocate device
memory where they need the consensus error (their framework owns all device
memory through its own pool, or cudaMalloc would synchronise a latency-critical
loop, or they are a plug-in handed pre-allocated buffers).  Through the C ABI,
it must give the value of the existing entry point, gasloc_consensus_error,
within the tolerance the other consensus-error comparisons use (relative
1e-12: same per-element arithmetic, fp64 sums in a different order), on
consecutive calls that reuse its static scratch; it must leave the device's
free memory unchanged; and its scratch address must follow the CUDA context
it is called in (a reset device, or a driver context of the caller's own).
This file is named so that pytest collects it last.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild
from paper_2606_11081_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    torch.cuda.set_device(0)
    return torch


def _check_calls(torch, ctx, N, P, calls=2):
    stream = torch.cuda.current_stream()
    out = torch.empty(1, dtype=torch.float64, device="cuda")   # caller-owned output
    xptr, stride = ctx.buffer("x", 0)
    ref = ctx.consensus_error_now()          # existing entry point
    assert ref > 0
    for call in range(calls):                # calls in a row share the scratch
        out.fill_(-1.0)
        g.gasloc_consensus_error_noalloc(xptr, N, P, stride, out.data_ptr(), stream.cuda_stream)
        torch.cuda.synchronize()
        assert out.item() == pytest.approx(ref, rel=1e-12), call
    return xptr, stride, out


def test_noalloc_matches_existing_entry_point(torch_cuda):
    torch = torch_cuda
    N, P = 8, 3 * 8192 + 1027          # several chunks and a ragged tail
    hp = g.make_hparams(**dict(wl.COMMON_HP, weights="metropolis", edge_prob=0.5))
    with g.Context(N, P, "exp", 77, hparams=hp) as ctx:
        for rnd in range(3):
            ctx.local_steps(2)
            ctx.gossip_round()
            xptr, stride, out = _check_calls(torch, ctx, N, P)
        stream = torch.cuda.current_stream()
        # sizes beyond the static scratch are refused before any device work
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_consensus_error_noalloc(xptr, N, 536870913, 536870916, out.data_ptr(),
                                             stream.cuda_stream)
        assert e.value.code == g.ENOMEM
        with pytest.raises(g.GaslocError) as e:
            g.gasloc_consensus_error_noalloc(xptr + 4, N, P, stride, out.data_ptr(), stream.cuda_stream)
        assert e.value.code == g.EINVAL


def test_noalloc_more_chunks_than_the_grid(torch_cuda):
    # 3 workers of 16.8 M parameters (no graph: the replicas drift apart):
    # 2,050 chunks of 8192 elements against a launch grid of (SMs x CTAs per
    # SM), so CTAs walk several chunks and reuse their reduction slots; the
    # last chunk is ragged
    torch = torch_cuda
    N, P = 3, 2050 * 8192 - 3001
    with g.Context(N, P, "none", 5) as ctx:
        ctx.local_steps(1)
        ctx.gossip_round()
        _check_calls(torch, ctx, N, P, calls=3)


def test_noalloc_allocates_nothing(torch_cuda):
    torch = torch_cuda
    N, P = 4, 5 * 8192 + 9
    with g.Context(N, P, "ring", 11) as ctx:
        ctx.local_steps(1)
        ctx.gossip_round()
        xptr, stride, out = _check_calls(torch, ctx, N, P, calls=1)   # warm-up call
        stream = torch.cuda.current_stream()
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        for _ in range(5):
            g.gasloc_consensus_error_noalloc(xptr, N, P, stride, out.data_ptr(), stream.cuda_stream)
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        assert free1 == free0


# Runs without torch, on the CUDA runtime the library itself loaded, so that
# the device can be reset and a driver context of the caller's own created.
_CONTEXTS_SCRIPT = r"""
import ctypes, os, sys
import numpy as np
lib = ctypes.CDLL(sys.argv[1])
rt = ctypes.CDLL("libcudart.so.13")      # the runtime the library loaded
cu = ctypes.CDLL("libcuda.so.1")
c_p, c_i32, c_i64, c_dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
lib.gasloc_init.argtypes = [c_i32, c_i64, ctypes.c_char_p, ctypes.c_uint64, ctypes.POINTER(c_p)]
lib.gasloc_start.argtypes = [c_p]
lib.gasloc_write.argtypes = [c_p, c_i32, c_i32, c_p]
lib.gasloc_buffer.argtypes = [c_p, c_i32, c_i32, ctypes.POINTER(c_p), ctypes.POINTER(c_i64)]
lib.gasloc_consensus_error_now.argtypes = [c_p, ctypes.POINTER(c_dbl)]
lib.gasloc_consensus_error_noalloc.argtypes = [c_p, c_i32, c_i64, c_i64, c_p, c_p]
lib.gasloc_destroy.argtypes = [c_p]
lib.gasloc_last_error.restype = ctypes.c_char_p

def ck(rc, what):
    if rc != 0:
        raise SystemExit("%s failed: %d %s" % (what, rc, lib.gasloc_last_error()))

N, P = 6, 4 * 8192 + 333
rng = np.random.default_rng(3)
x = (1.0 + 1e-2 * rng.standard_normal((N, P))).astype(np.float32)

def one_pass(tag):
    ctx = c_p()
    ck(lib.gasloc_init(N, P, b"ring", 9, ctypes.byref(ctx)), "init")
    ck(lib.gasloc_start(ctx), "start")
    for i in range(N):
        row = np.ascontiguousarray(x[i])
        ck(lib.gasloc_write(ctx, 0, i, row.ctypes.data), "write")
    ref = c_dbl()
    ck(lib.gasloc_consensus_error_now(ctx, ctypes.byref(ref)), "existing entry point")
    xp, stride = c_p(), c_i64()
    ck(lib.gasloc_buffer(ctx, 0, 0, ctypes.byref(xp), ctypes.byref(stride)), "buffer")
    out = c_p()
    ck(rt.cudaMalloc(ctypes.byref(out), 8), "cudaMalloc (test output)")
    for call in range(2):
        ck(lib.gasloc_consensus_error_noalloc(xp, N, P, stride.value, out, None), "noalloc")
        ck(rt.cudaDeviceSynchronize(), "synchronize")
        v = c_dbl(-1.0)
        ck(rt.cudaMemcpy(ctypes.byref(v), out, 8, 2), "copy back")
        if not abs(v.value - ref.value) <= 1e-12 * abs(ref.value):
            raise SystemExit("%s call %d: %r != %r" % (tag, call, v.value, ref.value))
    ck(rt.cudaFree(out), "cudaFree (test output)")
    lib.gasloc_destroy(ctx)
    print(tag, "ok", ref.value)

ck(rt.cudaSetDevice(0), "cudaSetDevice")
one_pass("primary")
# a reset device: its primary context is replaced, with a new address space
ck(rt.cudaDeviceReset(), "cudaDeviceReset")
one_pass("after reset")
# a driver context of the caller's own, current on this thread
ck(cu.cuInit(0), "cuInit")
dev = ctypes.c_int()
ck(cu.cuDeviceGet(ctypes.byref(dev), 0), "cuDeviceGet")
own = c_p()
ck(cu.cuCtxCreate_v2(ctypes.byref(own), 0, dev), "cuCtxCreate")
one_pass("own context")
ck(cu.cuCtxDestroy_v2(own), "cuCtxDestroy")
ck(rt.cudaSetDevice(0), "cudaSetDevice")
one_pass("primary again")
"""


def test_noalloc_follows_the_cuda_context(torch_cuda):
    lib = os.environ.get("GASLOC_LIBRARY") or g.LIB_PATH
    r = subprocess.run([sys.executable, "-c", _CONTEXTS_SCRIPT, lib], cwd=ROOT, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    for tag in ("primary", "after reset", "own context", "primary again"):
        assert tag + " ok" in r.stdout, r.stdout
