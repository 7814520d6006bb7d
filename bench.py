#!/usr/bin/env python3
"""Benchmark of the GASLoC replica-update path on GB300.

One step = one outer round of the whole hot path on the workload's replicas,
already resident in HBM: H local AdamW steps for every worker (K_adamw), the
round's neighbour table where it is random (K_topo), and the gossip round with
the outer optimizer and the fused consensus-error reduction (K_gossip).

Prints ONE JSON line (rank 0).  `value` is replica-element updates per second
over the timed rounds (n_workers * n_params * rounds / time).  On several GPUs
(torchrun) every replica is split by parameter range, one contiguous range per
GPU (the steps are element-wise in the parameter index), and the one exchange
per round is an all-reduce of the ranks' consensus-error shares; the job's
time is the slowest rank's and `value` counts every rank's elements.
`e2e` repeats the measurement through the public C ABI from host buffers:
upload of the initial replicas, centres and curvature from pinned host memory,
every round's consensus error read back to the host, and the network average
read back at the end.  `roofline` is the dominant kernel's algorithmic bytes
per launch over its CUDA-event duration, against the measured HBM copy peak.
`cpu_baseline` is the CPU oracle timed on the host cores on a bounded slice.

--impl reference runs the CPU oracle as the reference arm (there is no
released code for the paper; the oracle written from it is the baseline).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "replica-element updates/sec per gossip round; achieved HBM GB/s vs 8 TB/s"
UNIT = "replica-element updates/s"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0      # the metric's "vs 8 TB/s" (GB300 HBM3e, nominal)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed rounds (default: the workload's round count)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gasloc", choices=["gasloc", "reference"])
    ap.add_argument("--workload", default=None)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--extras", default="all",
                    help="other workloads timed after the main one: 'all', 'none' or a comma list")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    return ap.parse_args()


def peak_hbm():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_SOURCE = {"adamw": "adamw.cu", "gossip": "gossip.cu", "ce": "ce.cu", "average": "setup.cu",
                 "round": "round.cu"}
CSRC = os.path.join(ROOT, "paper_2606_11081_gb300", "csrc")


def source_digest(name: str) -> str:
    """sha256 over a kernel source file and the local headers it includes,
    transitively (each file once, in name order): the code a profile of its
    kernels was taken from."""
    seen, todo = set(), [name]
    while todo:
        f = todo.pop()
        if f in seen or not os.path.exists(os.path.join(CSRC, f)):
            continue
        seen.add(f)
        text = open(os.path.join(CSRC, f)).read()
        todo.extend(re.findall(r'^#include "([^"]+)"', text, re.M))
    h = hashlib.sha256()
    for f in sorted(seen):
        h.update(f.encode() + b"\0" + open(os.path.join(CSRC, f), "rb").read())
    return h.hexdigest()


def kernel_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if the kernel's
    source (its file and the headers it includes) is unchanged since the
    capture (else None)."""
    prof = os.path.join(ROOT, "profiles", "%s_%s.md" % (kernel, workload))
    try:
        text = open(prof).read()
        m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
        h = re.search(r"source_sha256:\s*([0-9a-f]+)", text)
        if m and h and h.group(1) == source_digest(KERNEL_SOURCE[kernel]):
            return float(m.group(1))
    except Exception:
        pass
    return None


class ClockSampler:
    """Samples nvidia-smi during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                smax.append(float(p[2]))
            except ValueError:
                continue
            for nm, v in zip(names, p[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def aggregate(ms_local: float, units_local: float, dist_mod=None, device=None):
    """Whole-job timing over the ranks (one GPU each, each holding a range of
    the parameters): the job's time is the slowest rank's timed region and its
    throughput is the units all ranks processed over that time.  Returns
    (ms_max, units_per_second)."""
    if dist_mod is None:
        return ms_local, units_local / (ms_local / 1e3)
    import torch
    t_max = torch.tensor([ms_local], dtype=torch.float64, device=device)
    t_sum = torch.tensor([units_local], dtype=torch.float64, device=device)
    dist_mod.all_reduce(t_max, op=dist_mod.ReduceOp.MAX)
    dist_mod.all_reduce(t_sum, op=dist_mod.ReduceOp.SUM)
    ms = float(t_max.item())
    return ms, float(t_sum.item()) / (ms / 1e3)


def shard_range(P: int, world: int, rank: int, align: int = 4096):
    """The part [p0, p1) of the P parameters that `rank` holds when every
    replica is split over `world` GPUs: contiguous, in multiples of `align`
    elements (the last part takes the rest)."""
    units = -(-P // align)                       # blocks of `align` elements, the last one ragged
    p0 = min(rank * units // world * align, P)
    p1 = min((rank + 1) * units // world * align, P)
    if p1 <= p0:
        raise ValueError("%d parameters do not split over %d ranks in parts of %d" % (P, world, align))
    return p0, p1


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def cpu_baseline(w, seconds: float):
    """Times the CPU oracle (fp32 build) on a slice of the workload's
    parameter indices: full n_workers, the workload's H, whole rounds."""
    import oracle
    oracle.build()
    orc = oracle.get("f32")
    from paper_2606_11081_gb300 import workloads as wl
    hp = wl.hparams_of(w)
    topo, torus = w.topology, (0, 0)
    if topo.startswith("torus:"):
        r, c = topo[6:].split("x")
        topo, torus = "torus", (int(r), int(c))
    slice_p = 1 << 20
    pb = oracle.make_problem(w.n_workers, w.n_params, topo, seed=w.seed, torus=torus,
                             **{k: (bool(v) if k == "per_worker_h" else v) for k, v in hp.items()})
    import numpy as np
    kidx = np.arange(slice_p, dtype=np.int64)
    st = orc.state(pb, kidx)
    Hi = orc.draw_local_steps(w.seed, w.n_workers, w.draw_hmax) if w.H < 0 else None
    rounds = 0
    t0 = time.perf_counter()
    while True:
        st.local_steps(w.H if w.H > 0 else 0, Hi)
        st.gossip_round()
        st.consensus_error()
        rounds += 1
        el = time.perf_counter() - t0
        if el >= seconds or rounds >= 100000:
            break
    value = w.n_workers * slice_p * rounds / el
    return {"value": value, "unit": UNIT, "cores": orc.lib.oc_num_threads(), "kind": "oracle",
            "sample": "%d rounds of the workload on parameter indices [0, %d) with all %d workers "
                      "(fp32 oracle, OpenMP over elements), %.1f s" % (rounds, slice_p, w.n_workers, el)}


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import numpy as np
    import oracle
    from paper_2606_11081_gb300 import workloads as wl
    oracle.build()
    orc = oracle.get("f32")
    hp = wl.hparams_of(w)
    topo, torus = w.topology, (0, 0)
    if topo.startswith("torus:"):
        r, c = topo[6:].split("x")
        topo, torus = "torus", (int(r), int(c))
    pb = oracle.make_problem(w.n_workers, w.n_params, topo, seed=w.seed, torus=torus,
                             **{k: (bool(v) if k == "per_worker_h" else v) for k, v in hp.items()})
    slice_p = 1 << 20   # the cpu_baseline sample: about 9 ms per round on 16 cores
    st = orc.state(pb, np.arange(slice_p, dtype=np.int64))
    Hi = orc.draw_local_steps(w.seed, w.n_workers, w.draw_hmax) if w.H < 0 else None

    def step():
        st.local_steps(w.H if w.H > 0 else 0, Hi)
        st.gossip_round()
        return st.consensus_error()

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    value = w.n_workers * slice_p * args.steps / el
    sample = ("each step: one round of the workload on parameter indices [0, %d) with all %d "
              "workers (fp32 oracle, OpenMP over elements)" % (slice_p, w.n_workers))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * el / args.steps,
            "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": workload_config(w, args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": orc.lib.oc_num_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def ce_exchange(dist_mod, ctx, ce_dev, k):
    """The one exchange of a round when the replicas are split over GPUs by
    parameter range: this GPU's consensus-error share is copied to device
    memory on the round's stream and summed over the ranks (all-reduce)."""
    ctx.consensus_error_async(ce_dev.data_ptr() + 8 * k)
    dist_mod.all_reduce(ce_dev[k:k + 1], op=dist_mod.ReduceOp.SUM)


def workload_config(w, args, world=1):
    state_gb = w.n_workers * w.n_params * 4 * (6 + (1 if w.hp.get("per_worker_h") else 0)) / 1e9 / world
    return {"workload": w.name, "n_workers": w.n_workers, "n_params": w.n_params,
            "topology": w.topology, "H": w.H if w.H > 0 else "H_i~U{1..%d}" % w.draw_hmax,
            "layout": "tensor-list(%d)" % len(w.numels) if w.numels else "flat",
            "storage": w.hp.get("storage", "f32"),
            "weights": w.hp.get("weights", "uniform"), "outer": "nesterov(0.7, 0.9)",
            "seed": w.seed,
            "parallelism": ("parameter ranges x%d (each GPU holds a contiguous range of every replica; "
                            "one fp64 all-reduce of the consensus-error shares per round)" % world
                            if world > 1 else "one GPU"),
            "l2": "inputs larger than L2 (%.1f GB replica state per GPU, no flush)" % state_gb}


def adamw_bytes_of(w, steps, es, P=None):
    """Algorithmic bytes of every AdamW launch of one round (a launch per
    sub-step; sub-step s steps the workers with H_i > s) over P parameters
    per replica (default: all of them)."""
    P = w.n_params if P is None else P
    per_h = bool(w.hp.get("per_worker_h"))
    out = []
    for s in range(max(steps)):
        act = sum(1 for h in steps if h > s)
        if act:
            out.append(((8 * es * act) if per_h else (7 * es * act + es)) * P)
    return out


def time_rounds(ctx, torch, stream, K, H, after_round=None, split=False):
    """K rounds timed with CUDA events on the launch stream; returns (total ms,
    local-step ms, gossip ms), the last two summed over the rounds when
    `split` (events around the local steps and the gossip round of each
    round; an event between two kernels keeps the second from starting before
    the first ends, so the rounds' total is taken without them).
    after_round(k) runs after round k's gossip (the ranks' exchange)."""
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)] if split else None
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(K):
        if split:
            ev[k][0].record(stream)
        ctx.local_steps(H)
        if split:
            ev[k][1].record(stream)
        ctx.gossip_round()
        if split:
            ev[k][2].record(stream)
        if after_round is not None:
            after_round(k)
    t_end.record(stream)
    torch.cuda.synchronize()
    ms = t_start.elapsed_time(t_end)
    if not split:
        return ms, None, None
    local_ms = sum(ev[k][0].elapsed_time(ev[k][1]) for k in range(K))
    gossip_ms = sum(ev[k][1].elapsed_time(ev[k][2]) for k in range(K))
    return ms, local_ms, gossip_ms


def measure_fused(ctx, torch, stream, K, H, w, steps, es, round_bytes, peak):
    """The same rounds through gasloc_fused_round, where its fused kernel
    serves the store (None elsewhere): the round's last local step runs in
    the gossip kernel, which reads that step's iterate once instead of the
    local-step kernel writing it and the gossip kernel reading it back.  A
    labelled variant outside the one-pass-per-step byte model the targets use;
    its rate is over its own algorithmic bytes (the round's, less the rows the
    gossip no longer reads: the new y, and x too when the step started from
    x)."""
    l0 = ctx.launches
    ctx.local_steps(H)
    ctx.gossip_round()
    l1 = ctx.launches
    ctx.fused_round(H)
    if ctx.launches - l1 != (l1 - l0) - 1:   # fused: one launch fewer per round
        torch.cuda.synchronize()
        return None
    for _ in range(2):
        ctx.fused_round(H)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        ctx.fused_round(H)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / K
    saved = (2 if max(steps) == 1 else 1) * es * w.n_workers * w.n_params
    fb = round_bytes - saved
    return dict(kernel_entry(fb, ms, peak), ms_per_round=ms, bytes=fb,
                value=float(w.n_workers) * w.n_params / (ms / 1e3),
                note="gasloc_fused_round: the last local step fused into the gossip kernel; a variant outside "
                     "the byte model of the targets (one HBM pass per local step), not the measured path")


def kernel_entry(bytes_, time_ms, peak, **extra):
    """Rate of `bytes_` algorithmic bytes moved in `time_ms`, against the peak."""
    gbs = bytes_ / (time_ms / 1e3) / 1e9
    d = {"gbs": gbs, "frac": gbs / peak, "frac_of_nominal_8tbs": gbs / NOMINAL_HBM_GBS}
    d.update(extra)
    return d


def substep_profile(g, ctx, torch, stream, w, Hi, es, peak, reps=3):
    """AdamW launches of the heterogeneous workload one sub-step at a time:
    sub-step s steps the workers with H_i > s (the same launch as inside a
    round); each is timed over `reps` launches with CUDA events."""
    out = []
    for s in range(max(Hi)):
        mask = [1 if h > s else 0 for h in Hi]
        act = sum(mask)
        if act == 0:
            continue
        g.gasloc_set_local_steps(ctx.h, mask)
        ctx.local_steps(g.PER_WORKER_STEPS)   # warm-up launch
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            ctx.local_steps(g.PER_WORKER_STEPS)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        b = adamw_bytes_of(w, mask, es, ctx.P)[0]
        out.append(kernel_entry(b, ms, peak, substep=s + 1, active_workers=act, ms=ms, bytes=b))
    g.gasloc_set_local_steps(ctx.h, Hi)
    ctx.gossip_round()   # back to a round boundary
    torch.cuda.synchronize()
    return out


def measure_workload(g, torch, wl, name, K, warmup, peak):
    """Per-kernel rates of another workload in the same run (its own context,
    created and released here): AdamW, gossip and the round, CUDA events on the
    launch stream, plus the same rounds replayed from a CUDA graph."""
    w = wl.ALL_WORKLOADS[name]
    es = 2 if w.hp.get("storage") == "bf16" else 4
    hp = g.make_hparams(**wl.hparams_of(w))
    ctx = g.Context(w.n_workers, w.n_params, w.topology, w.seed, hparams=hp, numels=w.numels,
                    draw_hmax=w.draw_hmax)
    try:
        H = w.H if w.H > 0 else g.PER_WORKER_STEPS
        Hi = g.gasloc_get_local_steps(ctx.h, w.n_workers).tolist() if w.H < 0 else None
        stream = torch.cuda.current_stream()
        for _ in range(warmup):
            ctx.local_steps(H)
            ctx.gossip_round()
        torch.cuda.synchronize()
        ms, _, _ = time_rounds(ctx, torch, stream, K, H)
        ms_split, local_ms, gossip_ms = time_rounds(ctx, torch, stream, K, H, split=True)
        steps = [H] * w.n_workers if H > 0 else Hi
        ab = adamw_bytes_of(w, steps, es)
        gb = 5 * es * w.n_workers * w.n_params
        graph_ms = measure_graph(ctx, torch, stream, K, H)
        units = float(w.n_workers) * w.n_params
        fused = measure_fused(ctx, torch, stream, K, H, w, steps, es, sum(ab) + gb, peak)
        return {
            "rounds": K, "ms_per_round": ms / K, "value": units * K / (ms / 1e3),
            "ms_per_round_split": ms_split / K,
            "graph_ms_per_round": graph_ms, "graph_value": units / (graph_ms / 1e3),
            "adamw": kernel_entry(sum(ab), local_ms / K, peak, ms_per_round=local_ms / K,
                                  bytes_per_round=sum(ab), launches_per_round=len(ab)),
            "gossip": kernel_entry(gb, gossip_ms / K, peak, ms_per_round=gossip_ms / K, bytes_per_round=gb),
            "round": kernel_entry(sum(ab) + gb, ms / K, peak, bytes=sum(ab) + gb),
            "storage": "bf16" if es == 2 else "f32",
            "fused_round": fused,
        }
    finally:
        ctx.close()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()


# Other workloads timed in the same run, after the main one (name: rounds
# timed).  The 105 MB ring is short enough for launch gaps to count, so it
# takes more rounds.
EXTRA_WORKLOADS = {"ring_n4_p1m": 200, "exp_n8_gpt2s": 20, "exp_n8_gpt2s_bf16": 20,
                   "matching_n16_gpt2s_h8": 5, "torus2x4_n8_gpt2m_h4": 5}


def main():
    args = parse_args()
    from paper_2606_11081_gb300 import workloads as wl
    w = wl.ALL_WORKLOADS[args.workload or wl.BENCH_WORKLOAD]
    if args.steps is None:
        args.steps = w.rounds
    if args.impl == "reference":
        return run_reference(args, w)

    import numpy as np
    import torch
    import paper_2606_11081_gb300 as g
    from paper_2606_11081_gb300 import build as gbuild

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        pg = dist
    if rank == 0 or world == 1:
        gbuild.build()
    if pg:
        pg.barrier()

    hp = g.make_hparams(**wl.hparams_of(w))
    # more than one GPU: each holds a contiguous range of every replica's
    # parameters (every step is element-wise in the parameter index); the one
    # exchange per round is the sum of the ranks' consensus-error shares
    p_range = shard_range(w.n_params, world, rank) if world > 1 else None
    ctx = g.Context(w.n_workers, w.n_params, w.topology, w.seed, hparams=hp, numels=w.numels,
                    draw_hmax=w.draw_hmax, p_range=p_range)
    H = w.H if w.H > 0 else g.PER_WORKER_STEPS
    Hi = g.gasloc_get_local_steps(ctx.h, w.n_workers).tolist() if w.H < 0 else None
    stream = torch.cuda.current_stream()
    K = args.steps
    ce_dev = torch.zeros(max(K, args.warmup, 1), dtype=torch.float64, device="cuda")
    exchange = (lambda k: ce_exchange(pg, ctx, ce_dev, k)) if pg else None

    for k in range(args.warmup):
        ctx.local_steps(H)
        ctx.gossip_round()
        if exchange:
            exchange(k)
    torch.cuda.synchronize()

    clocks = ClockSampler(local)
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    l0 = ctx.launches
    ms, _, _ = time_rounds(ctx, torch, stream, K, H, exchange)
    launches = ctx.launches - l0
    # the same number of rounds again with events around each kernel, for the
    # kernels' own rates
    ms_split, local_ms, gossip_ms = time_rounds(ctx, torch, stream, K, H, exchange, split=True)
    clk = clocks.stop()
    N, P = w.n_workers, ctx.P        # P: the parameters this GPU holds
    units = float(N) * P * K
    ms, value = aggregate(ms, units, pg, torch.device("cuda", local) if pg else None)
    if pg:
        pg.barrier()
        ce = float(ce_dev[K - 1].item())        # the all-reduced sum of the shares
    else:
        ce = ctx.consensus_error()

    # algorithmic bytes (of this GPU's range)
    es = 2 if w.hp.get("storage") == "bf16" else 4      # bytes per stored element
    steps = [H] * N if H > 0 else Hi
    adamw_per_launch = adamw_bytes_of(w, steps, es, P)
    adamw_launches = len(adamw_per_launch)
    adamw_bytes = sum(adamw_per_launch)
    gossip_bytes = 5 * es * N * P
    peak, peak_kind = peak_hbm()
    adamw_gbs = adamw_bytes / (local_ms / K / 1e3) / 1e9
    gossip_gbs = gossip_bytes / (gossip_ms / K / 1e3) / 1e9
    dom = "adamw" if local_ms >= gossip_ms else "gossip"
    dom_gbs = adamw_gbs if dom == "adamw" else gossip_gbs
    dom_bytes_launch = adamw_bytes / adamw_launches if dom == "adamw" else gossip_bytes
    dom_ms_launch = local_ms / K / adamw_launches if dom == "adamw" else gossip_ms / K
    def traffic_of(kernel):
        # a profile is of a launch over all the parameters: this GPU's share
        t = kernel_traffic(kernel, w.name)
        return None if t is None else t * P / w.n_params
    traffic = traffic_of(dom)

    # the same rounds replayed from a CUDA graph (gasloc_run)
    graph_ms = measure_graph(ctx, torch, stream, K, H)
    # the labelled fused-round variant, where its kernel serves the store
    fused = None
    if N <= 4 and es == 4 and world == 1:
        fused = measure_fused(ctx, torch, stream, K, H, w, steps, es, adamw_bytes + gossip_bytes, peak)
    # the network average (Algorithm 1's output), timed on its own
    avg_ms = measure_average(g, ctx, torch, stream, P, 5)
    avg_bytes = es * N * P + 4 * P
    avg_gbs = avg_bytes / (avg_ms / 1e3) / 1e9
    # the standalone consensus-error reduction, timed on its own
    ce_ms = measure_ce(ctx, torch, stream, 10)
    ce_bytes = es * N * P
    ce_gbs = ce_bytes / (ce_ms / 1e3) / 1e9
    # AdamW one sub-step at a time (heterogeneous local steps)
    substeps = substep_profile(g, ctx, torch, stream, w, Hi, es, peak) if Hi is not None else None

    e2e = None
    ctx.close()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if not args.no_e2e:
        e2e = measure_e2e(g, torch, w, hp, H, K, p_range, pg)
        # whole job: every rank's units over the slowest rank's time
        _, e2e["value"] = aggregate(e2e["seconds"] * 1e3, float(N) * P * K, pg,
                                    torch.device("cuda", local) if pg else None)
        torch.cuda.empty_cache()

    extras = None
    names = [] if (args.extras == "none" or world > 1) else (
        list(EXTRA_WORKLOADS) if args.extras == "all" else args.extras.split(","))
    names = [n for n in names if n != w.name]
    if names:
        extras = {}
        eclk = ClockSampler(local)
        eclk.start()
        for name in names:
            extras[name] = measure_workload(g, torch, wl, name, EXTRA_WORKLOADS.get(name, 10), 3, peak)
        extras["clocks"] = eclk.stop()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms / K, "ms_per_step_split": ms_split / K,
            "higher_is_better": True,
            "scaling": "strong", "vs_baseline": None, "dtype": "bf16" if es == 2 else "f32",
            "data": "synthetic", "config": workload_config(w, args, world),
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": dom_gbs, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": dom_gbs / peak,
                         "frac_of_nominal_8tbs": dom_gbs / NOMINAL_HBM_GBS,
                         "traffic": traffic, "algorithmic_bytes_per_launch": dom_bytes_launch,
                         "ms_per_launch": dom_ms_launch,
                         "note": "algorithmic bytes of the kernel's launches over their summed "
                                 "CUDA-event time (AdamW: one launch per local sub-step)"},
            "kernels": {"adamw": {"gbs": adamw_gbs, "frac": adamw_gbs / peak,
                                  "frac_of_nominal_8tbs": adamw_gbs / NOMINAL_HBM_GBS, "ms_per_round": local_ms / K,
                                  "bytes_per_round": adamw_bytes, "launches_per_round": adamw_launches,
                                  "substeps": substeps},
                        "gossip": {"gbs": gossip_gbs, "frac": gossip_gbs / peak,
                                   "frac_of_nominal_8tbs": gossip_gbs / NOMINAL_HBM_GBS,
                                   "ms_per_round": gossip_ms / K, "bytes_per_round": gossip_bytes},
                        "ce": {"gbs": ce_gbs, "frac": ce_gbs / peak, "frac_of_nominal_8tbs": ce_gbs / NOMINAL_HBM_GBS,
                               "ms_per_launch": ce_ms, "bytes_per_launch": ce_bytes,
                               "traffic": traffic_of("ce"),
                               "note": "standalone reduction (after a direct write of x); each round's "
                                       "value comes fused from the gossip kernel"},
                        "average": {"gbs": avg_gbs, "frac": avg_gbs / peak,
                                    "frac_of_nominal_8tbs": avg_gbs / NOMINAL_HBM_GBS,
                                    "ms_per_launch": avg_ms, "bytes_per_launch": avg_bytes,
                                    "traffic": traffic_of("average"),
                                    "note": "network average x-bar (end of a run)"},
                        "round": {"bytes": adamw_bytes + gossip_bytes,
                                  "gbs": (adamw_bytes + gossip_bytes) / (ms / K / 1e3) / 1e9,
                                  "frac": (adamw_bytes + gossip_bytes) / (ms / K / 1e3) / 1e9 / peak,
                                  "frac_of_nominal_8tbs":
                                      (adamw_bytes + gossip_bytes) / (ms / K / 1e3) / 1e9 / NOMINAL_HBM_GBS}},
            "graph": {"ms_per_step": graph_ms, "value": units / (graph_ms * K / 1e3),
                      "note": "the same rounds through gasloc_run (graphs of 8 captured rounds replayed, single "
                              "rounds for the rest), "
                              "timed after the main measurement; this GPU's parameters (its range when "
                              "the replicas are split over GPUs)"},
            "fused_round": fused,
            "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": launches, "clocks": clk,
            "consensus_error": ce,
        }
        if extras is not None:
            line["workloads"] = extras
            if "exp_n8_gpt2s_bf16" in extras:
                xb = extras["exp_n8_gpt2s_bf16"]
                line["kernels_bf16"] = {"workload": "exp_n8_gpt2s_bf16", "adamw": xb["adamw"],
                                        "gossip": xb["gossip"], "round": xb["round"]}
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()
    return 0


def measure_graph(ctx, torch, stream, K, H):
    """Mean round time (ms) of K rounds run by gasloc_run from its CUDA graphs
    (of 8 rounds and of one, both captured before the timed region)."""
    ctx.run(9 if K >= 8 else 1, H)   # captures (and 9 or 1 rounds)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    ctx.run(K, H)
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / K


def measure_average(g, ctx, torch, stream, P, reps):
    """Mean duration (ms) of the network-average kernel into a device buffer."""
    dst = torch.empty(P, dtype=torch.float32, device="cuda")
    g.gasloc_average(ctx.h, dst.data_ptr())   # warm-up
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        g.gasloc_average(ctx.h, dst.data_ptr())
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def measure_ce(ctx, torch, stream, reps):
    """Mean duration (ms) of the standalone consensus-error reduction: once x
    has been written directly, every read runs it.  The reads are enqueued
    without waiting (each copies 8 bytes to pinned memory) between two events."""
    ctx.write("x", 0, ctx.read("x", 0))   # same values; the fused value is no longer current
    host = torch.zeros(reps + 1, dtype=torch.float64, pin_memory=True)
    ctx.consensus_error_async(host.data_ptr())   # warm-up
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for r in range(reps):
        ctx.consensus_error_async(host.data_ptr() + 8 * (r + 1))
    e1.record(stream)
    torch.cuda.synchronize()
    vals = host.numpy()
    if not (vals == vals[0]).all():
        raise RuntimeError("standalone consensus-error reductions disagree")
    return e0.elapsed_time(e1) / reps


def measure_e2e(g, torch, w, hp, H, K, p_range=None, dist_mod=None):
    """Same rounds through the public C ABI from host buffers: upload the
    initial replicas (x_0 broadcast), centres and curvature from pinned memory,
    read the consensus error back every round, read the average back at the
    end.  Split over GPUs, each rank does so for its parameter range, and each
    round's value read back is the all-reduced sum of the ranks' shares."""
    import numpy as np
    N = w.n_workers
    ctx = g.Context(N, w.n_params, w.topology, w.seed, hparams=hp, numels=w.numels, draw_hmax=w.draw_hmax,
                    p_range=p_range)
    P = ctx.P
    per_h = bool(w.hp.get("per_worker_h"))
    nh = N if per_h else 1
    # host inputs (taken from the device initialisation, untimed)
    x0 = torch.empty(P, dtype=torch.float32, pin_memory=True)
    cs = torch.empty((N, P), dtype=torch.float32, pin_memory=True)
    hs = torch.empty((nh, P), dtype=torch.float32, pin_memory=True)
    g.gasloc_read(ctx.h, "x", 0, x0.numpy())
    for i in range(N):
        g.gasloc_read(ctx.h, "c", i, cs[i].numpy())
    for i in range(nh):
        g.gasloc_read(ctx.h, "h", i, hs[i].numpy())
    out = torch.empty(P, dtype=torch.float32, pin_memory=True)
    ces = torch.zeros(K, dtype=torch.float64, pin_memory=True)
    ce_dev = torch.zeros(K, dtype=torch.float64, device="cuda") if dist_mod else None
    # untimed warm-up of the host-to-device path: one upload of every input
    # (the first transfer from freshly written pinned pages runs slower); the
    # timed region below uploads everything again
    g.gasloc_write_ptr(ctx.h, "x", -1, x0.data_ptr())
    for i in range(N):
        g.gasloc_write_ptr(ctx.h, "c", i, cs[i].data_ptr())
    for i in range(nh):
        g.gasloc_write_ptr(ctx.h, "h", i, hs[i].data_ptr())
    torch.cuda.synchronize()
    if dist_mod:
        dist_mod.barrier()
    t0 = time.perf_counter()
    g.gasloc_write_ptr(ctx.h, "x", -1, x0.data_ptr())
    for i in range(N):
        g.gasloc_write_ptr(ctx.h, "c", i, cs[i].data_ptr())
    for i in range(nh):
        g.gasloc_write_ptr(ctx.h, "h", i, hs[i].data_ptr())
    t1 = time.perf_counter()
    # every round's consensus error is copied to pinned host memory as the
    # round completes; the host waits once, after the last round
    base = ces.data_ptr()
    for k in range(K):
        ctx.local_steps(H)
        ctx.gossip_round()
        if dist_mod:
            ce_exchange(dist_mod, ctx, ce_dev, k)
            ces[k:k + 1].copy_(ce_dev[k:k + 1], non_blocking=True)
        else:
            ctx.consensus_error_async(base + 8 * k)
    ctx.synchronize()
    torch.cuda.synchronize()
    t2 = time.perf_counter()
    g.gasloc_average_host(ctx.h, out.numpy())
    el = time.perf_counter() - t0
    t3 = el - (t2 - t0)
    if not (ces.numpy() > 0).all():
        raise RuntimeError("a round's consensus error did not arrive on the host")
    # the same rounds with a blocking read after each one, for comparison
    tb = time.perf_counter()
    for k in range(K):
        ctx.local_steps(H)
        ctx.gossip_round()
        if dist_mod:
            ce_exchange(dist_mod, ctx, ce_dev, k)
            float(ce_dev[k].item())
        else:
            ctx.consensus_error()
    tb = time.perf_counter() - tb
    ctx.close()
    h2d = (P + N * P + nh * P) * 4
    d2h = 8 * K + 4 * P
    return {"value": N * P * K / el, "unit": UNIT, "h2d_bytes_per_step": h2d / K,
            "d2h_bytes_per_step": d2h / K, "seconds": el,
            "upload_s": t1 - t0, "rounds_s": t2 - t1, "download_s": t3,
            "value_blocking_read": N * P * K / tb,
            "note": "initial replicas, centres and curvature uploaded once per run (amortised, after "
                    "one untimed upload of the same buffers); "
                    "every round's consensus error copied to pinned host memory without "
                    "blocking, one wait after the last round; average read at the end; "
                    "value_blocking_read: rounds only, waiting for each round's value"}


if __name__ == "__main__":
    sys.exit(main())
