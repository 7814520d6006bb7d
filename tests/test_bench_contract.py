"""bench.py keeps its output contract: one JSON line with the keys the driver
reads.  The reference arm (the CPU oracle) runs here without a GPU; the main
arm runs on a GPU on a reduced workload."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
BASE = ["metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
        "scaling", "vs_baseline", "dtype", "data", "config"]


def _run(args, timeout):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + args, cwd=ROOT,
                       capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.strip().splitlines() if l.startswith("{")]
    assert len(lines) == 1
    return json.loads(lines[0])


def test_reference_arm_line():
    d = _run(["--impl", "reference", "--steps", "2", "--warmup", "1"], 600)
    for k in BASE + ["impl", "cpu_baseline", "e2e"]:
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["config"]["workload"] == "hetero_exp_n32_gpt2s"


@pytest.mark.gpu
def test_main_arm_line():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    d = _run(["--workload", "exp_n32_p4m_hetero", "--steps", "5", "--warmup", "3", "--cpu-seconds", "1",
              "--extras", "ring_n4_p1m,exp_n8_p16m_bf16"], 900)
    for k in BASE + ["roofline", "e2e", "cpu_baseline", "gpu_launches", "clocks"]:
        assert k in d, k
    rf = d["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in rf, k
    assert rf["bound"] == "hbm" and 0 < rf["frac"] < 1.2
    # per round: one AdamW launch per local sub-step (H_i up to 8), the
    # round's random neighbour table, and gossip
    subs = d["kernels"]["adamw"]["substeps"]
    assert d["gpu_launches"] == 5 * (len(subs) + 2)
    assert [s["substep"] for s in subs] == list(range(1, len(subs) + 1))
    assert all(0 < s["frac"] < 1.3 for s in subs)
    assert d["config"]["workload"] == "exp_n32_p4m_hetero"
    for name in ("ring_n4_p1m", "exp_n8_p16m_bf16"):
        x = d["workloads"][name]
        assert x["adamw"]["gbs"] > 0 and x["gossip"]["gbs"] > 0 and x["value"] > 0

    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    assert d["cpu_baseline"]["cores"] >= 1


def test_profile_digest_follows_included_headers(tmp_path, monkeypatch):
    """A profile's traffic counts only while the code it was taken from is
    unchanged: the kernel file and every local header it includes, however
    deep, but nothing else."""
    sys.path.insert(0, ROOT)
    import bench
    (tmp_path / "k.cu").write_text('#include "a.cuh"\n#include <cstdio>\nint k;\n')
    (tmp_path / "a.cuh").write_text('#pragma once\n#include "b.cuh"\n')
    (tmp_path / "b.cuh").write_text('int b = 1;\n')
    (tmp_path / "c.cuh").write_text('int c = 1;\n')
    monkeypatch.setattr(bench, "CSRC", str(tmp_path))
    d0 = bench.source_digest("k.cu")
    (tmp_path / "c.cuh").write_text('int c = 2;\n')     # not included
    assert bench.source_digest("k.cu") == d0
    (tmp_path / "b.cuh").write_text('int b = 2;\n')     # included through a.cuh
    d1 = bench.source_digest("k.cu")
    assert d1 != d0
    (tmp_path / "k.cu").write_text('#include "a.cuh"\n#include <cstdio>\nint k2;\n')
    assert bench.source_digest("k.cu") != d1


def test_every_profiled_kernel_source_exists():
    sys.path.insert(0, ROOT)
    import bench
    for f in bench.KERNEL_SOURCE.values():
        assert os.path.exists(os.path.join(bench.CSRC, f)), f
