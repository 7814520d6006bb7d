"""Builds a GPU context and an oracle state for the same problem (test helper)."""
import numpy as np

import oracle
import paper_2606_11081_gb300 as g
from paper_2606_11081_gb300 import workloads as wl

TOL = 1e-5   # parity bound: |x_gpu - x_oracle| <= 1e-5 (1 + |x_oracle|)


def within_tol(gpu, ref, tol=TOL):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    return np.abs(gpu - ref) <= tol * (1.0 + np.abs(ref))


def oracle_problem(N, P, topology, seed, hp):
    torus = (0, 0)
    topo = topology
    if topology.startswith("torus:"):
        r, c = topology[6:].split("x")
        torus = (int(r), int(c))
        topo = "torus"
    kw = {k: v for k, v in hp.items()}
    kw["per_worker_h"] = bool(kw.get("per_worker_h", False))
    return oracle.make_problem(N, P, topo, seed=seed, torus=torus, **kw)


def make_pair(N, P, topology, seed=wl.SEED, hp=None, numels=None, Hi=None, draw_hmax=None,
              kidx=None, precision="f32"):
    hp = dict(hp or {})
    full = dict(wl.COMMON_HP)
    full.update(hp)
    ctx = g.Context(N, P, topology, seed, hparams=g.make_hparams(**full), numels=numels,
                    local_steps=Hi, draw_hmax=draw_hmax)
    st = oracle.get(precision).state(oracle_problem(N, P, topology, seed, full), kidx)
    return ctx, st


def workload_pair(name, kidx=None):
    w = wl.WORKLOADS[name]
    return w, make_pair(w.n_workers, w.n_params, w.topology, w.seed, wl.hparams_of(w), w.numels,
                        draw_hmax=w.draw_hmax, kidx=kidx)
