"""GB300 (sm_103a) replica-update path of GASLoC -- Python binding of libgasloc.

A thin ctypes layer over the C ABI declared in ``include/gasloc.h``: the
functions below carry the same names and arguments and only marshal them;
every step of the path runs in the library's CUDA kernels.  There is no
fallback: importing this package without a built ``libgasloc.so`` raises.

PyTorch is used as plumbing only: its caching allocator backs the library's
device memory and its current stream is the stream work is enqueued on.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
# GASLOC_LIBRARY selects another build of the library (the index-checked one,
# libgasloc_checked.so, in its tests).
LIB_PATH = os.environ.get("GASLOC_LIBRARY") or os.path.join(HERE, "libgasloc.so")

OK, EINVAL, ENOMEM, ECUDA, ESTATE, EDEVICE, EIO = 0, -1, -2, -3, -4, -5, -6
OUTER = {"sgd": 0, "sgdm": 1, "nesterov": 2, "eq2": 3, "dadam": 4, "local_dadam": 5}
WEIGHTS = {"uniform": 0, "metropolis": 1, "lazy": 2}
BUF = {"x": 0, "y": 1, "m": 2, "v": 3, "b": 4, "c": 5, "h": 6}
STORAGE = {"f32": 0, "bf16": 1}
MAX_WORKERS = 32
PER_WORKER_STEPS = -1


class GaslocError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("gasloc error %d: %s" % (code, msg))
        self.code = code


class Hparams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eps", ctypes.c_double), ("weight_decay", ctypes.c_double),
                ("noise_sigma", ctypes.c_double), ("outer_lr", ctypes.c_double),
                ("outer_momentum", ctypes.c_double), ("eta", ctypes.c_double),
                ("alpha", ctypes.c_double), ("gamma", ctypes.c_double),
                ("edge_prob", ctypes.c_double), ("outer_mode", ctypes.c_int32),
                ("weights", ctypes.c_int32), ("per_worker_h", ctypes.c_int32),
                ("storage", ctypes.c_int32), ("lr_total_steps", ctypes.c_int64),
                ("lr_warmup_frac", ctypes.c_double), ("lr_warmup_start", ctypes.c_double),
                ("lr_final_frac", ctypes.c_double)]


ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p)

_P = ctypes.c_void_p
_I32, _I64, _U64, _DBL = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
_I32P, _I64P = ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int64)
_FP, _DP = ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_double)

# name -> (restype, argtypes): the exported symbols of include/gasloc.h
SIGNATURES = {
    "gasloc_default_hparams": (None, [ctypes.POINTER(Hparams)]),
    "gasloc_init": (ctypes.c_int, [_I32, _I64, ctypes.c_char_p, _U64, ctypes.POINTER(_P)]),
    "gasloc_set_hparams": (ctypes.c_int, [_P, ctypes.POINTER(Hparams)]),
    "gasloc_get_hparams": (ctypes.c_int, [_P, ctypes.POINTER(Hparams)]),
    "gasloc_set_layout": (ctypes.c_int, [_P, _I32, _I64P]),
    "gasloc_set_range": (ctypes.c_int, [_P, _I64, _I64]),
    "gasloc_get_range": (ctypes.c_int, [_P, _I64P, _I64P, _I64P]),
    "gasloc_set_allocator": (ctypes.c_int, [_P, ALLOC_FN, FREE_FN, _P]),
    "gasloc_set_stream": (ctypes.c_int, [_P, _P]),
    "gasloc_start": (ctypes.c_int, [_P]),
    "gasloc_set_local_steps": (ctypes.c_int, [_P, _I32P]),
    "gasloc_draw_local_steps": (ctypes.c_int, [_P, _I32]),
    "gasloc_get_local_steps": (ctypes.c_int, [_P, _I32P]),
    "gasloc_local_steps": (ctypes.c_int, [_P, _I32]),
    "gasloc_gossip_round": (ctypes.c_int, [_P]),
    "gasloc_fused_round": (ctypes.c_int, [_P, _I32]),
    "gasloc_run": (ctypes.c_int, [_P, _I32, _I32, _DP]),
    "gasloc_consensus_error": (ctypes.c_int, [_P, _DP]),
    "gasloc_consensus_error_now": (ctypes.c_int, [_P, _DP]),
    "gasloc_consensus_error_async": (ctypes.c_int, [_P, _P]),
    "gasloc_synchronize": (ctypes.c_int, [_P]),
    "gasloc_consensus_error_noalloc": (ctypes.c_int, [_P, _I32, _I64, _I64, _P, _P]),
    "gasloc_get_topology": (ctypes.c_int, [_P, _I64, _I32P, _FP, _I32P]),
    "gasloc_average": (ctypes.c_int, [_P, _P]),
    "gasloc_average_host": (ctypes.c_int, [_P, _FP]),
    "gasloc_buffer": (ctypes.c_int, [_P, _I32, _I32, ctypes.POINTER(_P), _I64P]),
    "gasloc_read": (ctypes.c_int, [_P, _I32, _I32, _FP]),
    "gasloc_write": (ctypes.c_int, [_P, _I32, _I32, _FP]),
    "gasloc_gather": (ctypes.c_int, [_P, _I32, _I32, _I64, _I64P, _FP]),
    "gasloc_round": (ctypes.c_int, [_P, _I64P]),
    "gasloc_steps_taken": (ctypes.c_int, [_P, _I32, _I64P]),
    "gasloc_save": (ctypes.c_int, [_P, ctypes.c_char_p]),
    "gasloc_load": (ctypes.c_int, [_P, ctypes.c_char_p]),
    "gasloc_launch_count": (ctypes.c_int, [_P, _I64P]),
    "gasloc_selftest_bounded_wait": (ctypes.c_int, [_P, _I64]),
    "gasloc_checked_build": (ctypes.c_int, []),
    "gasloc_selftest_index_check": (ctypes.c_int, [_P]),
    "gasloc_last_error": (ctypes.c_char_p, []),
    "gasloc_destroy": (None, [_P]),
}

_lib: Optional[ctypes.CDLL] = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Loads libgasloc.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError("libgasloc.so not found at %s: build it with "
                          "paper_2606_11081_gb300.build.build()" % path)
    try:   # share the CUDA runtime torch already loaded, if any
        import torch  # noqa: F401
    except Exception:
        pass
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(rc: int) -> None:
    if rc != OK:
        raise GaslocError(rc, _lib.gasloc_last_error().decode(errors="replace"))


def _arr(a: np.ndarray, t):
    return a.ctypes.data_as(t)


# ---------------------------------------------------------------- C names --

def gasloc_default_hparams() -> Hparams:
    hp = Hparams()
    load_library().gasloc_default_hparams(ctypes.byref(hp))
    return hp


def gasloc_init(n_workers: int, n_params: int, topology: str, seed: int) -> ctypes.c_void_p:
    lib = load_library()
    h = ctypes.c_void_p()
    _check(lib.gasloc_init(n_workers, n_params, topology.encode(), seed, ctypes.byref(h)))
    return h


def gasloc_set_hparams(ctx, hp: Hparams) -> None:
    _check(_lib.gasloc_set_hparams(ctx, ctypes.byref(hp)))


def gasloc_get_hparams(ctx) -> Hparams:
    hp = Hparams()
    _check(_lib.gasloc_get_hparams(ctx, ctypes.byref(hp)))
    return hp


def gasloc_set_layout(ctx, numels: Sequence[int]) -> None:
    a = np.ascontiguousarray(numels, dtype=np.int64)
    _check(_lib.gasloc_set_layout(ctx, int(a.size), _arr(a, _I64P)))


def gasloc_set_range(ctx, p_begin: int, p_end: int) -> None:
    _check(_lib.gasloc_set_range(ctx, p_begin, p_end))


def gasloc_get_range(ctx):
    """(p_begin, p_end, n_params of the whole problem)."""
    a, b, n = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(_lib.gasloc_get_range(ctx, ctypes.byref(a), ctypes.byref(b), ctypes.byref(n)))
    return a.value, b.value, n.value


def gasloc_set_allocator(ctx, alloc_fn, free_fn, user=None) -> None:
    _check(_lib.gasloc_set_allocator(ctx, alloc_fn, free_fn, user))


def gasloc_set_stream(ctx, stream_handle: int) -> None:
    _check(_lib.gasloc_set_stream(ctx, ctypes.c_void_p(stream_handle)))


def gasloc_start(ctx) -> None:
    _check(_lib.gasloc_start(ctx))


def gasloc_set_local_steps(ctx, H: Optional[Sequence[int]]) -> None:
    if H is None:
        _check(_lib.gasloc_set_local_steps(ctx, None))
        return
    a = np.ascontiguousarray(H, dtype=np.int32)
    _check(_lib.gasloc_set_local_steps(ctx, _arr(a, _I32P)))


def gasloc_draw_local_steps(ctx, hmax: int) -> None:
    _check(_lib.gasloc_draw_local_steps(ctx, hmax))


def gasloc_get_local_steps(ctx, n_workers: int) -> np.ndarray:
    a = np.zeros(n_workers, np.int32)
    _check(_lib.gasloc_get_local_steps(ctx, _arr(a, _I32P)))
    return a


def gasloc_local_steps(ctx, H: int) -> None:
    _check(_lib.gasloc_local_steps(ctx, H))


def gasloc_gossip_round(ctx) -> None:
    _check(_lib.gasloc_gossip_round(ctx))


def gasloc_fused_round(ctx, H: int) -> None:
    """H local steps then a gossip round, the last step fused with the gossip
    round where the store allows (a variant outside the separate kernels'
    byte model; gasloc_run and the benchmark use the separate kernels)."""
    _check(_lib.gasloc_fused_round(ctx, H))


def gasloc_run(ctx, rounds: int, H: int, trace: bool = False):
    """`rounds` complete rounds replayed from a CUDA graph; returns the
    per-round consensus errors when trace is set (synchronising)."""
    if trace:
        out = np.zeros(rounds, np.float64)
        _check(_lib.gasloc_run(ctx, rounds, H, _arr(out, _DP)))
        return out
    _check(_lib.gasloc_run(ctx, rounds, H, None))
    return None


def gasloc_consensus_error(ctx) -> float:
    out = ctypes.c_double()
    _check(_lib.gasloc_consensus_error(ctx, ctypes.byref(out)))
    return out.value


def gasloc_consensus_error_now(ctx) -> float:
    out = ctypes.c_double()
    _check(_lib.gasloc_consensus_error_now(ctx, ctypes.byref(out)))
    return out.value


def gasloc_consensus_error_async(ctx, dst_ptr: int) -> None:
    """Enqueues the copy of the consensus error to address dst_ptr (8 bytes,
    host or device; pinned host memory keeps it asynchronous)."""
    _check(_lib.gasloc_consensus_error_async(ctx, ctypes.c_void_p(dst_ptr)))


def gasloc_synchronize(ctx) -> None:
    _check(_lib.gasloc_synchronize(ctx))


def gasloc_consensus_error_noalloc(x_ptr: int, n_workers: int, n_params: int, worker_stride: int,
                                   ce_out_ptr: int, stream_handle: int = 0) -> None:
    """Consensus error of caller-owned replicas into a caller-owned device
    double, without any device allocation (asynchronous on the stream)."""
    _check(load_library().gasloc_consensus_error_noalloc(
        ctypes.c_void_p(x_ptr), n_workers, n_params, worker_stride, ctypes.c_void_p(ce_out_ptr),
        ctypes.c_void_p(stream_handle)))


def gasloc_get_topology(ctx, round_: int, n_workers: int):
    nbr = np.zeros((n_workers, n_workers), np.int32)
    w = np.zeros((n_workers, n_workers), np.float32)
    deg = np.zeros(n_workers, np.int32)
    _check(_lib.gasloc_get_topology(ctx, round_, _arr(nbr, _I32P), _arr(w, _FP), _arr(deg, _I32P)))
    return nbr, w, deg


def gasloc_average(ctx, dst_device_ptr: int) -> None:
    _check(_lib.gasloc_average(ctx, ctypes.c_void_p(dst_device_ptr)))


def gasloc_average_host(ctx, out: np.ndarray) -> np.ndarray:
    assert out.dtype == np.float32 and out.flags.c_contiguous
    _check(_lib.gasloc_average_host(ctx, _arr(out, _FP)))
    return out


def gasloc_buffer(ctx, which: str, tensor: int = 0):
    p = ctypes.c_void_p()
    stride = ctypes.c_int64()
    _check(_lib.gasloc_buffer(ctx, BUF[which], tensor, ctypes.byref(p), ctypes.byref(stride)))
    return p.value, stride.value


def gasloc_read(ctx, which: str, worker: int, out: np.ndarray) -> np.ndarray:
    assert out.dtype == np.float32 and out.flags.c_contiguous
    _check(_lib.gasloc_read(ctx, BUF[which], worker, _arr(out, _FP)))
    return out


def gasloc_write(ctx, which: str, worker: int, src: np.ndarray) -> None:
    src = np.ascontiguousarray(src, dtype=np.float32)
    _check(_lib.gasloc_write(ctx, BUF[which], worker, _arr(src, _FP)))


def gasloc_write_ptr(ctx, which: str, worker: int, host_ptr: int) -> None:
    _check(_lib.gasloc_write(ctx, BUF[which], worker, ctypes.cast(host_ptr, _FP)))


def gasloc_gather(ctx, which: str, worker: int, idx: np.ndarray) -> np.ndarray:
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    out = np.zeros(idx.size, np.float32)
    _check(_lib.gasloc_gather(ctx, BUF[which], worker, idx.size, _arr(idx, _I64P), _arr(out, _FP)))
    return out


def gasloc_round(ctx) -> int:
    r = ctypes.c_int64()
    _check(_lib.gasloc_round(ctx, ctypes.byref(r)))
    return r.value


def gasloc_steps_taken(ctx, worker: int) -> int:
    r = ctypes.c_int64()
    _check(_lib.gasloc_steps_taken(ctx, worker, ctypes.byref(r)))
    return r.value


def gasloc_save(ctx, path: str) -> None:
    _check(_lib.gasloc_save(ctx, path.encode()))


def gasloc_load(ctx, path: str) -> None:
    _check(_lib.gasloc_load(ctx, path.encode()))


def gasloc_launch_count(ctx) -> int:
    r = ctypes.c_int64()
    _check(_lib.gasloc_launch_count(ctx, ctypes.byref(r)))
    return r.value


def gasloc_selftest_bounded_wait(ctx, limit_ns: int) -> int:
    """Runs the bounded-wait self-test; returns the status code (EDEVICE is
    the expected outcome: the wait expired and was reported)."""
    return _lib.gasloc_selftest_bounded_wait(ctx, limit_ns)


def gasloc_checked_build() -> bool:
    """True if the loaded library is the index-checked build."""
    return bool(load_library().gasloc_checked_build())


def gasloc_selftest_index_check(ctx) -> int:
    """Evaluates one failing index check on the device; returns the status
    code (EDEVICE from the checked build, OK from the normal one)."""
    return _lib.gasloc_selftest_index_check(ctx)


def gasloc_last_error() -> str:
    return load_library().gasloc_last_error().decode(errors="replace")


def gasloc_destroy(ctx) -> None:
    if ctx:
        _lib.gasloc_destroy(ctx)


# ------------------------------------------------------- torch plumbing ---

class _TorchAllocator:
    """Device-memory hooks backed by torch's CUDA caching allocator."""

    def __init__(self):
        import torch
        self.torch = torch
        self.dev = torch.cuda.current_device()

        def _alloc(nbytes, stream, user):
            try:
                return self.torch.cuda.caching_allocator_alloc(int(nbytes), self.dev,
                                                               stream if stream else 0)
            except Exception:
                return None

        def _free(ptr, stream, user):
            try:
                self.torch.cuda.caching_allocator_delete(ptr)
            except Exception:
                pass

        self.alloc = ALLOC_FN(_alloc)
        self.free = FREE_FN(_free)


class Context:
    """Owns one gasloc context; methods are the C calls with the context bound."""

    def __init__(self, n_workers: int, n_params: int, topology: str, seed: int,
                 hparams: Optional[Hparams] = None, numels: Optional[Sequence[int]] = None,
                 local_steps: Optional[Sequence[int]] = None, draw_hmax: Optional[int] = None,
                 use_torch: bool = True, stream: Optional[int] = None,
                 p_range: Optional[Sequence[int]] = None):
        """p_range = (p_begin, p_end): hold only those parameters of every
        replica (gasloc_set_range); self.P is then p_end - p_begin."""
        load_library()
        self.n = n_workers
        self.P = n_params
        self.h = None
        self.h = gasloc_init(n_workers, n_params, topology, seed)
        self._alloc = None
        if hparams is not None:
            gasloc_set_hparams(self.h, hparams)
        if numels is not None:
            gasloc_set_layout(self.h, numels)
        if p_range is not None:
            gasloc_set_range(self.h, int(p_range[0]), int(p_range[1]))
            self.P = int(p_range[1]) - int(p_range[0])
        if use_torch:
            import torch
            self._alloc = _TorchAllocator()
            gasloc_set_allocator(self.h, self._alloc.alloc, self._alloc.free, None)
            if stream is None:
                stream = torch.cuda.current_stream().cuda_stream
        if stream is not None:
            gasloc_set_stream(self.h, stream)
        gasloc_start(self.h)
        if local_steps is not None:
            gasloc_set_local_steps(self.h, local_steps)
        elif draw_hmax is not None:
            gasloc_draw_local_steps(self.h, draw_hmax)

    def close(self) -> None:
        if self.h:
            gasloc_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # the calls
    def local_steps(self, H: int) -> None:
        gasloc_local_steps(self.h, H)

    def gossip_round(self) -> None:
        gasloc_gossip_round(self.h)

    def fused_round(self, H: int) -> None:
        gasloc_fused_round(self.h, H)

    def run(self, rounds: int, H: int, trace: bool = False):
        return gasloc_run(self.h, rounds, H, trace)

    def consensus_error(self) -> float:
        return gasloc_consensus_error(self.h)

    def consensus_error_now(self) -> float:
        return gasloc_consensus_error_now(self.h)

    def consensus_error_async(self, host_ptr: int) -> None:
        gasloc_consensus_error_async(self.h, host_ptr)

    def synchronize(self) -> None:
        gasloc_synchronize(self.h)

    def topology(self, round_: int):
        return gasloc_get_topology(self.h, round_, self.n)

    def read(self, which: str, worker: int) -> np.ndarray:
        return gasloc_read(self.h, which, worker, np.zeros(self.P, np.float32))

    def read_all(self, which: str) -> np.ndarray:
        rows = self.n if (which != "h" or self.hparams.per_worker_h) else 1
        return np.stack([self.read(which, i) for i in range(rows)])

    def write(self, which: str, worker: int, values: np.ndarray) -> None:
        gasloc_write(self.h, which, worker, values)

    def gather(self, which: str, worker: int, idx: np.ndarray) -> np.ndarray:
        return gasloc_gather(self.h, which, worker, idx)

    def average_host(self) -> np.ndarray:
        return gasloc_average_host(self.h, np.zeros(self.P, np.float32))

    def buffer(self, which: str, tensor: int = 0):
        return gasloc_buffer(self.h, which, tensor)

    def view(self, which: str, tensor: int, numel: int, rows: Optional[int] = None):
        """Zero-copy torch view [rows, numel] of one tensor's buffer."""
        import torch
        ptr, stride = self.buffer(which, tensor)
        if rows is None:
            rows = self.n if (which != "h" or self.hparams.per_worker_h) else 1

        if self.hparams.storage == STORAGE["bf16"]:
            raw = self.view_raw_u16(ptr, stride, rows, numel)
            return raw.view(torch.bfloat16)

        class _Cai:
            __cuda_array_interface__ = {"shape": (rows, numel), "typestr": "<f4", "data": (ptr, False),
                                        "strides": (max(stride, 1) * 4, 4), "version": 3}
        return torch.as_tensor(_Cai(), device="cuda")

    @staticmethod
    def view_raw_u16(ptr: int, stride: int, rows: int, numel: int):
        import torch

        class _Cai:
            __cuda_array_interface__ = {"shape": (rows, numel), "typestr": "<i2", "data": (ptr, False),
                                        "strides": (max(stride, 1) * 2, 2), "version": 3}
        return torch.as_tensor(_Cai(), device="cuda")

    @property
    def round(self) -> int:
        return gasloc_round(self.h)

    def steps_taken(self, worker: int) -> int:
        return gasloc_steps_taken(self.h, worker)

    @property
    def hparams(self) -> Hparams:
        return gasloc_get_hparams(self.h)

    def set_hparams(self, hp: Hparams) -> None:
        gasloc_set_hparams(self.h, hp)

    def save(self, path: str) -> None:
        gasloc_save(self.h, path)

    def load(self, path: str) -> None:
        gasloc_load(self.h, path)

    @property
    def launches(self) -> int:
        return gasloc_launch_count(self.h)


def make_hparams(**kw) -> Hparams:
    """Default hyperparameters with keyword overrides (outer/weights by name)."""
    hp = gasloc_default_hparams()
    for k, v in kw.items():
        if k == "outer":
            hp.outer_mode = OUTER[v]
        elif k == "weights":
            hp.weights = WEIGHTS[v]
        elif k == "per_worker_h":
            hp.per_worker_h = int(v)
        elif k == "storage":
            hp.storage = STORAGE[v] if isinstance(v, str) else int(v)
        else:
            if not hasattr(hp, k):
                raise KeyError(k)
            setattr(hp, k, v)
    return hp
