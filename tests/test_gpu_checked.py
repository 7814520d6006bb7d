"""The index-checked build, this library's stand-in for a memory sanitizer:
the same kernels with every worker row, column range, neighbour index and TMA
offset tested before the access (a failed test skips the access and is
reported as GASLOC_EDEVICE).  Its self-test must see a failing check, and the
GPU parity suites run against it must pass -- no kernel addressed anything
outside its buffers on any of their cases (ragged tails, tensor lists, odd
sizes, random graphs, per-worker steps, bf16, every workload at full size and
the largest replica the ABI accepts)."""
import os
import subprocess
import sys

import pytest
import torch

import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import build as gbuild

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def checked_lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return gbuild.build(checked=True)


def _env(lib):
    env = dict(os.environ)
    env["GASLOC_LIBRARY"] = lib
    env["PYTHONPATH"] = ROOT + os.pathsep + env.get("PYTHONPATH", "")
    return env


def test_normal_build_has_no_checks():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gbuild.build()
    assert not g.gasloc_checked_build()
    with g.Context(4, 5000, "ring", 1) as ctx:
        assert g.gasloc_selftest_index_check(ctx.h) == g.OK


def test_checked_build_reports_a_failing_check(checked_lib):
    code = "\n".join([
        "import paper_2606_11081_gb300 as g",
        "assert g.gasloc_checked_build()",
        "with g.Context(4, 5000, 'ring', 1) as ctx:",
        "    assert g.gasloc_selftest_index_check(ctx.h) == g.EDEVICE",
        "    ctx.local_steps(1)",
        "    ctx.gossip_round()",
        "    assert ctx.consensus_error() > 0.0   # the context stays usable",
        "print('checked ok')",
    ])
    r = subprocess.run([sys.executable, "-c", code], env=_env(checked_lib), cwd=ROOT, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0 and "checked ok" in r.stdout, r.stdout + r.stderr


def test_parity_suites_under_index_checks(checked_lib):
    suites = ["tests/test_gpu_parity.py", "tests/test_gpu_bf16.py", "tests/test_gpu_run.py",
              "tests/test_gpu_failure.py", "tests/test_gpu_properties.py", "tests/test_gpu_fullsize.py",
              "tests/test_gpu_round.py", "tests/test_zz_no_alloc.py"]
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider"] + suites,
                       env=_env(checked_lib), cwd=ROOT, capture_output=True, text=True, timeout=1200)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
