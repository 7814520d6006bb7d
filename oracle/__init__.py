"""Python access to the CPU oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY: the test-suite, the smoke check and the benchmark's
CPU-baseline leg are the only users.  The product package never imports this
module, and this module imports nothing from the product package.

The oracle is compiled twice from the same source: ``f32`` (the arithmetic of
the replica store, one IEEE rounding per operation in the documented order) and
``f64`` (the same steps in double precision).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "oracle.c")
LIBS = {"f32": os.path.join(HERE, "liboracle_f32.so"),
        "f64": os.path.join(HERE, "liboracle_f64.so")}
_REAL = {"f32": "float", "f64": "double"}

TOPO = {"none": 0, "ring": 1, "complete": 2, "exp": 3, "torus": 4, "matching": 5, "2peer": 6}
WEIGHTS = {"uniform": 0, "metropolis": 1, "lazy": 2}
OUTER = {"sgd": 0, "sgdm": 1, "nesterov": 2, "eq2": 3, "dadam": 4, "local_dadam": 5}
BUF = {"x": 0, "y": 1, "m": 2, "v": 3, "b": 4, "c": 5, "h": 6}
STORAGE = {"f32": 0, "bf16": 1}


def build(force: bool = False) -> None:
    """Compiles both precision builds of the oracle with gcc (-ffp-contract=off)."""
    for prec, lib in LIBS.items():
        if (not force and os.path.exists(lib)
                and os.path.getmtime(lib) >= max(os.path.getmtime(SRC),
                                                 os.path.getmtime(os.path.join(HERE, "oracle.h")))):
            continue
        tmp = lib + ".tmp%d" % os.getpid()
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
               "-fPIC", "-shared", "-DREAL=%s" % _REAL[prec], "-o", tmp, SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, lib)


class Problem(ctypes.Structure):
    _fields_ = [
        ("n_workers", ctypes.c_int32), ("topology", ctypes.c_int32),
        ("n_params", ctypes.c_int64),
        ("torus_rows", ctypes.c_int32), ("torus_cols", ctypes.c_int32),
        ("weights", ctypes.c_int32), ("outer_mode", ctypes.c_int32),
        ("seed", ctypes.c_uint64), ("edge_prob", ctypes.c_double),
        ("lr", ctypes.c_double), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
        ("eps", ctypes.c_double), ("weight_decay", ctypes.c_double),
        ("noise_sigma", ctypes.c_double),
        ("outer_lr", ctypes.c_double), ("outer_momentum", ctypes.c_double),
        ("eta", ctypes.c_double), ("alpha", ctypes.c_double), ("gamma", ctypes.c_double),
        ("per_worker_h", ctypes.c_int32), ("storage", ctypes.c_int32),
        ("lr_total_steps", ctypes.c_int64), ("lr_warmup_frac", ctypes.c_double),
        ("lr_warmup_start", ctypes.c_double), ("lr_final_frac", ctypes.c_double),
    ]


def make_problem(n_workers: int, n_params: int, topology: str = "ring", seed: int = 0,
                 torus: Sequence[int] = (0, 0), weights: str = "uniform",
                 outer: str = "nesterov", edge_prob: float = 1.0, lr: float = 3e-4,
                 beta1: float = 0.9, beta2: float = 0.95, eps: float = 1e-8,
                 weight_decay: float = 0.1, noise_sigma: float = 0.01,
                 outer_lr: float = 0.7, outer_momentum: float = 0.9, eta: float = 1.0,
                 alpha: float = 1.0, gamma: float = 0.0, per_worker_h: bool = False,
                 storage: str = "f32", lr_total_steps: int = 0, lr_warmup_frac: float = 0.1,
                 lr_warmup_start: float = 0.01, lr_final_frac: float = 0.0) -> Problem:
    return Problem(n_workers=n_workers, topology=TOPO[topology], n_params=n_params,
                   torus_rows=torus[0], torus_cols=torus[1], weights=WEIGHTS[weights],
                   outer_mode=OUTER[outer], seed=seed, edge_prob=edge_prob, lr=lr,
                   beta1=beta1, beta2=beta2, eps=eps, weight_decay=weight_decay,
                   noise_sigma=noise_sigma, outer_lr=outer_lr, outer_momentum=outer_momentum,
                   eta=eta, alpha=alpha, gamma=gamma, per_worker_h=int(per_worker_h),
                   storage=STORAGE[storage], lr_total_steps=lr_total_steps,
                   lr_warmup_frac=lr_warmup_frac, lr_warmup_start=lr_warmup_start,
                   lr_final_frac=lr_final_frac)


_I64P = ctypes.POINTER(ctypes.c_int64)
_I32P = ctypes.POINTER(ctypes.c_int32)
_F64P = ctypes.POINTER(ctypes.c_double)


def _ptr(a: np.ndarray, t):
    return a.ctypes.data_as(t)


class Oracle:
    """One precision build of the oracle."""

    def __init__(self, precision: str = "f32"):
        if not os.path.exists(LIBS[precision]):
            build()
        self.precision = precision
        lib = ctypes.CDLL(LIBS[precision])
        self.lib = lib
        u64, i64, i32, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        sig = {
            "oc_mix64": (u64, [u64]), "oc_hash": (u64, [u64, u64, u64, u64]),
            "oc_fmix32": (ctypes.c_uint32, [ctypes.c_uint32]),
            "oc_normal": (dbl, [u64, u64, u64, u64]),
            "oc_uniform": (dbl, [u64, u64, u64, u64, dbl, dbl]),
            "oc_noise": (dbl, [u64, u64, u64, u64, i32]),
            "oc_real_size": (ctypes.c_int, []), "oc_num_threads": (ctypes.c_int, []),
            "oc_bf16_round": (dbl, [dbl]),
            "oc_permutation": (None, [u64, i64, i32, _I32P]),
            "oc_draw_local_steps": (None, [u64, i32, i32, _I32P]),
            "oc_topology": (ctypes.c_int, [ctypes.POINTER(Problem), i64, _I32P, _F64P, _I32P]),
            "oc_create": (ctypes.c_void_p, [ctypes.POINTER(Problem), _I64P, i64]),
            "oc_destroy": (None, [ctypes.c_void_p]),
            "oc_local_steps": (ctypes.c_int, [ctypes.c_void_p, i32, _I32P]),
            "oc_set_hparams": (None, [ctypes.c_void_p, ctypes.POINTER(Problem)]),
            "oc_sched_lr": (ctypes.c_double, [ctypes.POINTER(Problem), i64]),
            "oc_gossip_round": (ctypes.c_int, [ctypes.c_void_p]),
            "oc_consensus_error": (dbl, [ctypes.c_void_p]),
            "oc_average": (None, [ctypes.c_void_p, _F64P]),
            "oc_get": (ctypes.c_int, [ctypes.c_void_p, i32, i32, _F64P]),
            "oc_set": (ctypes.c_int, [ctypes.c_void_p, i32, i32, _F64P]),
            "oc_round": (i64, [ctypes.c_void_p]),
            "oc_steps_taken": (i64, [ctypes.c_void_p, i32]),
        }
        for name, (res, args) in sig.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        assert lib.oc_real_size() == (4 if precision == "f32" else 8)

    # generators -----------------------------------------------------------
    def mix64(self, z: int) -> int:
        return self.lib.oc_mix64(z)

    def hash(self, seed: int, tag: int, a: int, b: int) -> int:
        return self.lib.oc_hash(seed, tag, a, b)

    def fmix32(self, h: int) -> int:
        return self.lib.oc_fmix32(h)

    def normal(self, seed, tag, i, k) -> float:
        return self.lib.oc_normal(seed, tag, i, k)

    def uniform(self, seed, tag, i, k, lo, span) -> float:
        return self.lib.oc_uniform(seed, tag, i, k, lo, span)

    def noise(self, seed, i, n, k, storage: str = "f32") -> float:
        return self.lib.oc_noise(seed, i, n, k, STORAGE[storage])

    def sched_lr(self, pb: Problem, n: int) -> float:
        """Learning rate of a worker's n-th local step under pb's schedule."""
        return self.lib.oc_sched_lr(ctypes.byref(pb), n)

    def bf16_round(self, v: float) -> float:
        return self.lib.oc_bf16_round(v)

    def permutation(self, seed: int, t: int, n: int) -> np.ndarray:
        p = np.zeros(n, np.int32)
        self.lib.oc_permutation(seed, t, n, _ptr(p, _I32P))
        return p

    def draw_local_steps(self, seed: int, n: int, hmax: int) -> np.ndarray:
        h = np.zeros(n, np.int32)
        self.lib.oc_draw_local_steps(seed, n, hmax, _ptr(h, _I32P))
        return h

    def topology(self, pb: Problem, t: int):
        """Returns (nbr [N,N] int32, w [N,N] float64, deg [N] int32) for round t."""
        n = pb.n_workers
        nbr = np.full((n, n), -1, np.int32)
        w = np.zeros((n, n), np.float64)
        deg = np.zeros(n, np.int32)
        rc = self.lib.oc_topology(ctypes.byref(pb), t, _ptr(nbr, _I32P), _ptr(w, _F64P),
                                  _ptr(deg, _I32P))
        if rc != 0:
            raise ValueError("oc_topology failed (%d)" % rc)
        return nbr, w, deg

    def dense_w(self, pb: Problem, t: int) -> np.ndarray:
        """The round-t mixing matrix as a dense N x N array (float64)."""
        nbr, w, deg = self.topology(pb, t)
        n = pb.n_workers
        W = np.zeros((n, n))
        for i in range(n):
            for q in range(deg[i] + 1):
                W[i, nbr[i, q]] = w[i, q]
        return W

    def state(self, pb: Problem, kidx: Optional[np.ndarray] = None) -> "OracleState":
        return OracleState(self, pb, kidx)


class OracleState:
    """A replica state held by the oracle for a set of parameter indices."""

    def __init__(self, orc: Oracle, pb: Problem, kidx: Optional[np.ndarray]):
        self.orc = orc
        self.pb = pb
        if kidx is None:
            self.nk = int(pb.n_params)
            self._kidx = None
            kp = None
        else:
            self._kidx = np.ascontiguousarray(kidx, dtype=np.int64)
            self.nk = int(self._kidx.size)
            kp = _ptr(self._kidx, _I64P)
        h = orc.lib.oc_create(ctypes.byref(pb), kp, self.nk)
        if not h:
            raise MemoryError("oc_create failed")
        self.h = h

    def __del__(self):
        h = getattr(self, "h", None)
        if h:
            self.orc.lib.oc_destroy(h)
            self.h = None

    def local_steps(self, H: int, Hi: Optional[np.ndarray] = None) -> None:
        hp = None
        if Hi is not None:
            self._hi = np.ascontiguousarray(Hi, dtype=np.int32)
            hp = _ptr(self._hi, _I32P)
        if self.orc.lib.oc_local_steps(self.h, H, hp) != 0:
            raise ValueError("oc_local_steps failed")

    def set_hparams(self, pb: Problem) -> None:
        """New optimizer hyperparameters and mixing weights for the next steps
        (sizes, graph, seed and storage stay as created)."""
        self.orc.lib.oc_set_hparams(self.h, ctypes.byref(pb))

    def gossip_round(self) -> None:
        rc = self.orc.lib.oc_gossip_round(self.h)
        if rc != 0:
            raise ValueError("oc_gossip_round failed (%d)" % rc)

    def consensus_error(self) -> float:
        return self.orc.lib.oc_consensus_error(self.h)

    def average(self) -> np.ndarray:
        out = np.zeros(self.nk, np.float64)
        self.orc.lib.oc_average(self.h, _ptr(out, _F64P))
        return out

    def get(self, which: str, worker: int) -> np.ndarray:
        out = np.zeros(self.nk, np.float64)
        if self.orc.lib.oc_get(self.h, BUF[which], worker, _ptr(out, _F64P)) != 0:
            raise IndexError(which)
        return out

    def get_all(self, which: str) -> np.ndarray:
        n = self.pb.n_workers if (which != "h" or self.pb.per_worker_h) else 1
        return np.stack([self.get(which, i) for i in range(n)])

    def set(self, which: str, worker: int, values: np.ndarray) -> None:
        v = np.ascontiguousarray(values, dtype=np.float64)
        assert v.size == self.nk
        if self.orc.lib.oc_set(self.h, BUF[which], worker, _ptr(v, _F64P)) != 0:
            raise IndexError(which)

    @property
    def round(self) -> int:
        return self.orc.lib.oc_round(self.h)

    def steps_taken(self, worker: int) -> int:
        return self.orc.lib.oc_steps_taken(self.h, worker)


_CACHE = {}


def get(precision: str = "f32") -> Oracle:
    if precision not in _CACHE:
        _CACHE[precision] = Oracle(precision)
    return _CACHE[precision]
