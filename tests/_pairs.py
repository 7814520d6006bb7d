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


U32 = 2.0 ** -24


def ce_bound(x):
    """Relative error bound of the library's consensus error of the replicas x
    ([n, P] stored values) against the exact value (the oracle's fp64 one).

    Per element the library forms dv_i = x_i - x_0 (x_0: worker 0's value),
    S1 = sum dv_i and S2 = sum dv_i^2 over ascending i and e = S2 - (S1/n) S1,
    in fp32 with one rounding per operation (u = 2^-24).  With a_i = x_i - x_0
    and D = sum a_i^2: S2 is within gamma_{n+1} D of D, S1 within gamma_n
    sum|a_i| <= gamma_n sqrt(n D) of sum a_i, so (S1/n) S1 (with the roundings
    of 1/n and of the product) is within about (2n + 2) u D of its exact value
    (S1^2 / n <= D), and the final rounding adds u e: the element's error is at
    most about (3n + 3) u D + u e; (3n + 4) u D + 2 u e is taken to cover the
    higher-order terms.  Over the elements, in fp64, the total's relative
    error is at most (3n + 4) u kappa + 2 u with kappa = sum D / sum e >= 1,
    plus the fp64 sums of both sides over P elements (2 P 2^-53)."""
    x = np.asarray(x, np.float64)
    n, P = x.shape
    e = ((x - x.mean(0)) ** 2).sum()
    if e == 0.0:
        return 0.0
    kappa = ((x - x[0]) ** 2).sum() / e
    return (3 * n + 4) * U32 * kappa + 2 * U32 + 2 * P * 2.0 ** -53


def assert_ce(got, st, x=None):
    """The library's consensus error `got` against the oracle state's, within
    ce_bound of the oracle's replicas."""
    ref = st.consensus_error()
    tol = ce_bound(st.get_all("x") if x is None else x)
    assert abs(got - ref) <= tol * abs(ref) + 1e-30, (got, ref, tol)
