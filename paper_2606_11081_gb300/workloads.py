"""Synthetic workloads shaped like the paper's LLM runs.

Only shapes, seeds and hyperparameters live here -- no arithmetic of the
method.  The paper trains Llama-style models on FineWeb (App. B); neither the
data nor trained weights are used.  The replica-update path sees a synthetic
diagonal quadratic per worker instead, on parameter vectors with the sizes of
GPT-2 small (124,439,808 parameters in 148 tensors) and GPT-2 medium
(354,823,168 parameters in 292 tensors), computed from the public architecture
constants below.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional

SEED = 0x6A510C
VOCAB, CTX = 50257, 1024


def gpt2_numels(d_model: int, n_layer: int) -> List[int]:
    """Element counts of the GPT-2 parameter tensors in declaration order."""
    d = d_model
    out = [VOCAB * d, CTX * d]                          # wte, wpe
    for _ in range(n_layer):
        out += [d, d,                                   # ln_1 weight, bias
                d * 3 * d, 3 * d,                       # attn c_attn weight, bias
                d * d, d,                               # attn c_proj weight, bias
                d, d,                                   # ln_2 weight, bias
                d * 4 * d, 4 * d,                       # mlp c_fc weight, bias
                4 * d * d, d]                           # mlp c_proj weight, bias
    out += [d, d]                                       # ln_f weight, bias
    return out


GPT2_SMALL = gpt2_numels(768, 12)
GPT2_MEDIUM = gpt2_numels(1024, 24)
GPT2_SMALL_P = sum(GPT2_SMALL)     # 124,439,808
GPT2_MEDIUM_P = sum(GPT2_MEDIUM)   # 354,823,168


@dataclass
class Workload:
    name: str
    n_workers: int
    n_params: int
    topology: str
    H: int                           # local steps per round (-1: per-worker H_i)
    rounds: int
    hp: Dict[str, object] = field(default_factory=dict)
    numels: Optional[List[int]] = None
    draw_hmax: Optional[int] = None  # H_i drawn from {1..draw_hmax}
    seed: int = SEED

    def bytes_per_round(self, H_i: Optional[List[int]] = None) -> int:
        """Algorithmic HBM bytes of one round: every local step reads the
        iterate, m, v, c and writes y, m, v (7 elements per worker-element:
        28 B in fp32, 14 B in bf16) plus the shared curvature (one element per
        element; per worker-element when each worker has its own), and the
        gossip round reads the sent y once and x, b, and writes x, b (5
        elements per worker-element)."""
        N, P = self.n_workers, self.n_params
        per_h = bool(self.hp.get("per_worker_h", False))
        es = 2 if self.hp.get("storage") == "bf16" else 4
        if self.H > 0:
            steps = [self.H] * N
        else:
            assert H_i is not None
            steps = list(H_i)
        local = 0
        for s in range(max(steps)):
            act = sum(1 for h in steps if h > s)
            local += (8 * es * act if per_h else 7 * es * act + es) * P
        return local + 5 * es * N * P


WORKLOADS = {
    "ring_n4_p1m": Workload(
        "ring_n4_p1m", 4, 1_048_576, "ring", 1, 50,
        hp=dict(weights="uniform", noise_sigma=0.01)),
    "exp_n8_gpt2s": Workload(
        "exp_n8_gpt2s", 8, GPT2_SMALL_P, "exp", 1, 200,
        hp=dict(weights="uniform", noise_sigma=0.01)),
    "matching_n16_gpt2s_h8": Workload(
        "matching_n16_gpt2s_h8", 16, GPT2_SMALL_P, "matching", 8, 100,
        hp=dict(weights="uniform", noise_sigma=0.05)),
    "torus2x4_n8_gpt2m_h4": Workload(
        "torus2x4_n8_gpt2m_h4", 8, GPT2_MEDIUM_P, "torus:2x4", 4, 50,
        hp=dict(weights="metropolis", noise_sigma=0.01), numels=GPT2_MEDIUM),
    "hetero_exp_n32_gpt2s": Workload(
        "hetero_exp_n32_gpt2s", 32, GPT2_SMALL_P, "exp", -1, 50,
        hp=dict(weights="metropolis", noise_sigma=0.01, edge_prob=0.5, per_worker_h=True),
        draw_hmax=8),
}

# GPT-2 medium's position table, first layer and final norm: its tensor-list
# layout (ragged 1024-element tensors among large ones) at 13.6 M parameters.
GPT2_MEDIUM_1L = GPT2_MEDIUM[1:14] + GPT2_MEDIUM[-2:]

# Reduced copies of the workloads for profiler captures: a few GB of replica
# state each, well above the 129 MB L2.
PROFILE_WORKLOADS = {
    "exp_n8_p16m": Workload(
        "exp_n8_p16m", 8, 1 << 24, "exp", 1, 10,
        hp=dict(weights="uniform", noise_sigma=0.01)),
    "matching_n16_p8m_h8": Workload(
        "matching_n16_p8m_h8", 16, 1 << 23, "matching", 8, 10,
        hp=dict(weights="uniform", noise_sigma=0.05)),
    "torus2x4_n8_gpt2m1l_h4": Workload(
        "torus2x4_n8_gpt2m1l_h4", 8, sum(GPT2_MEDIUM_1L), "torus:2x4", 4, 10,
        hp=dict(weights="metropolis", noise_sigma=0.01), numels=GPT2_MEDIUM_1L),
    "exp_n32_p4m_hetero": Workload(
        "exp_n32_p4m_hetero", 32, 1 << 22, "exp", -1, 10,
        hp=dict(weights="metropolis", noise_sigma=0.01, edge_prob=0.5, per_worker_h=True),
        draw_hmax=8),
}

# The benchmark workload with a bfloat16 replica store (the paper trains in
# bf16): same arithmetic in fp32, every stored value rounded to bf16.
BF16_WORKLOADS = {
    "exp_n8_gpt2s_bf16": Workload(
        "exp_n8_gpt2s_bf16", 8, GPT2_SMALL_P, "exp", 1, 200,
        hp=dict(weights="uniform", noise_sigma=0.01, storage="bf16")),
    "exp_n8_p16m_bf16": Workload(
        "exp_n8_p16m_bf16", 8, 1 << 24, "exp", 1, 10,
        hp=dict(weights="uniform", noise_sigma=0.01, storage="bf16")),
}

ALL_WORKLOADS = dict(WORKLOADS, **PROFILE_WORKLOADS, **BF16_WORKLOADS)

# AdamW settings shared by every workload (App. B: weight decay 0.1,
# betas (0.9, 0.95)); constant lr 3e-4; Nesterov outer step 0.7 / 0.9.
COMMON_HP = dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1,
                 outer="nesterov", outer_lr=0.7, outer_momentum=0.9)

# The workload bench.py measures by default: the largest one that fits one GPU
# (112 GB of replica state, about 650 GB moved per round).
BENCH_WORKLOAD = "hetero_exp_n32_gpt2s"


def hparams_of(w: Workload) -> Dict[str, object]:
    d = dict(COMMON_HP)
    d.update(w.hp)
    return d
