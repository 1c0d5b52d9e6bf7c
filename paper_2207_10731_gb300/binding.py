"""Thin ctypes binding of libpss.so (argument marshalling only).

Every step of the hot path runs in the library's CUDA kernels; this module only
checks dtypes/contiguity, passes raw pointers and the current CUDA stream, and
turns status codes into exceptions.  There is no CPU fallback: if the library
is missing or no GPU is present, calls fail loudly.

Names follow include/pss.h: ``PSS.forward`` is ``pss_forward`` and so on.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libpss.so")

PSS_OK, PSS_ERR_INVALID_ARG, PSS_ERR_OOM, PSS_ERR_CUDA, PSS_ERR_STATE, PSS_ERR_INDEX_RANGE, \
    PSS_ERR_TIMEOUT, PSS_ERR_UNSUPPORTED, PSS_ERR_CAPACITY = range(9)
PSS_SGD, PSS_ADAGRAD = 0, 1
OPT_BACKWARD_PATH, OPT_UPDATE_MODE, OPT_PROFILE, OPT_SYNC_CHECK, OPT_ACCUM = 1, 2, 3, 4, 5
OPT_SIGNED = 6
OPT_CIRCULAR = 7
OPT_SORT_DIGIT_BITS = 8
OPT_DETERMINISTIC = 9
OPT_SORT_SCOPE = 10
ACCUM_F64, ACCUM_F32 = 0, 1
PATH_AUTO, PATH_ATOMIC, PATH_SORTED = 0, 1, 2
UPDATE_AUTO, UPDATE_DENSE, UPDATE_TOUCHED = 0, 1, 2
SORT_AUTO, SORT_GLOBAL, SORT_LOCAL = 0, 1, 2
K_LOCATIONS, K_FORWARD, K_SCATTER, K_UPDATE, K_SORT, K_REDUCE, K_MISC = range(7)
KERNEL_NAMES = ["locations", "forward", "scatter", "update", "sort", "reduce", "misc"]

# Every symbol include/pss.h declares (checked by the ABI test).
EXPORTS = [
    "pss_create", "pss_destroy", "pss_set_weights", "pss_get_weights", "pss_get_state",
    "pss_set_state", "pss_compute_locations", "pss_forward", "pss_backward_update",
    "pss_backward_grad", "pss_set_option", "pss_get_option", "pss_get_error", "pss_get_info",
    "pss_get_profile", "pss_reset_profile", "pss_status_string", "pss_grad_noalloc",
    "pss_check_convert", "pss_probe_l2",
]


class PSSInfo(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d", ctypes.c_int64), ("M", ctypes.c_int64),
                ("Z", ctypes.c_int64), ("G", ctypes.c_int64), ("J", ctypes.c_int64),
                ("L", ctypes.c_int64), ("R", ctypes.c_int64), ("A", ctypes.c_uint64),
                ("B0", ctypes.c_uint64), ("optimizer", ctypes.c_int64),
                ("kernel_launches", ctypes.c_int64), ("last_path", ctypes.c_int64),
                ("last_collision_rate", ctypes.c_double), ("A2", ctypes.c_uint64),
                ("B2", ctypes.c_uint64), ("signed_hash", ctypes.c_int64),
                ("circular", ctypes.c_int64), ("last_update", ctypes.c_int64)]


class PSSError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} (status {status})")


_lock = threading.Lock()
_lib = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libpss.so (built by ``paper_2207_10731_gb300.build``)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"libpss.so not found at {p}: run paper_2207_10731_gb300.build.build() "
                               "(needs nvcc); there is no CPU fallback")
        lib = ctypes.CDLL(p)
        vp, i32, i64, u64, f32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                  ctypes.c_uint64, ctypes.c_float)
        sigs = {
            "pss_create": [vp, i32, i32, i64, i32, i32, u64, ctypes.c_int, f32, vp, vp],
            "pss_destroy": [vp],
            "pss_set_weights": [vp, vp, i64, vp],
            "pss_get_weights": [vp, vp, i64, vp],
            "pss_get_state": [vp, vp, vp, i64, vp],
            "pss_set_state": [vp, vp, vp, i64, vp],
            "pss_compute_locations": [vp, vp, i64, vp, i64, vp, vp],
            "pss_forward": [vp, vp, i64, vp, i64, vp, vp],
            "pss_backward_update": [vp, vp, f32, vp],
            "pss_backward_grad": [vp, vp, vp, vp],
            "pss_set_option": [vp, i32, i64],
            "pss_get_option": [vp, i32, vp],
            "pss_get_error": [vp, vp, vp],
            "pss_get_info": [vp, vp],
            "pss_get_profile": [vp, i32, vp, vp],
            "pss_reset_profile": [vp],
            "pss_grad_noalloc": [vp, i32, i32, i64, i32, i32, u64, vp, i64, vp, i64, vp, vp, vp,
                                 vp],
            "pss_check_convert": [i32, vp, vp, i64, vp],
            "pss_probe_l2": [i32, vp, i64, i64, i32, vp],
        }
        for name, args in sigs.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.pss_status_string.argtypes = [ctypes.c_int]
        lib.pss_status_string.restype = ctypes.c_char_p
        _lib = lib
        return lib


def probe_l2(kind: int, buf, iters: int, ctas: int, stream=None):
    """Queue one L2 rate probe kernel (pss_probe_l2) over the device tensor buf."""
    lib = load_library()
    _check(lib.pss_probe_l2(int(kind), _ptr(buf), buf.numel() * buf.element_size(), int(iters),
                            int(ctas), _stream_ptr(stream)), "pss_probe_l2")


def status_string(status: int) -> str:
    try:
        return load_library().pss_status_string(status).decode()
    except Exception:  # library not loadable: still describe the code
        return {0: "ok"}.get(status, "error")


def _check(rc: int, what: str):
    if rc != PSS_OK:
        raise PSSError(rc, what)


def _torch():
    import torch
    return torch


def _stream_ptr(stream) -> ctypes.c_void_p:
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(stream.cuda_stream))


def _ptr(t) -> ctypes.c_void_p:
    return ctypes.c_void_p(int(t.data_ptr()))


def _need(t, dtype, name):
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


class PSS:
    """One shared-array hashed embedding (see include/pss.h).

    Batch tensors may live on the GPU or in (preferably pinned) host memory;
    host batches are staged by the library on the current stream.
    """

    def __init__(self, cards, dim: int, M: int, Z: int, G: int = 4, seed: int = 0,
                 optimizer: str = "sgd", eps: float = 1e-10, stream=None):
        self._lib = load_library()
        cards = np.ascontiguousarray(np.asarray(cards, dtype=np.int64))
        self.T = int(cards.shape[0])
        self.d, self.M, self.Z, self.G = int(dim), int(M), int(Z), int(G)
        self.optimizer = optimizer
        opt = {"sgd": PSS_SGD, "adagrad": PSS_ADAGRAD}[optimizer]
        h = ctypes.c_void_p()
        _check(self._lib.pss_create(ctypes.c_void_p(cards.ctypes.data), self.T, self.d, self.M,
                                    self.Z, self.G, ctypes.c_uint64(seed), opt,
                                    ctypes.c_float(eps), _stream_ptr(stream), ctypes.byref(h)),
               "pss_create")
        self._h = h
        self._batch = None
        info = self.info()
        self.J, self.L, self.R = info["J"], info["L"], info["R"]

    # -- life cycle -------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None):
            self._lib.pss_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- state --------------------------------------------------------------
    def set_weights(self, w, stream=None):
        _need(w, _torch().float32, "w")
        _check(self._lib.pss_set_weights(self._h, _ptr(w), w.numel(), _stream_ptr(stream)),
               "pss_set_weights")

    def get_weights(self, out=None, stream=None):
        torch = _torch()
        if out is None:
            out = torch.empty(self.M, dtype=torch.float32, device="cuda")
        _need(out, torch.float32, "out")
        _check(self._lib.pss_get_weights(self._h, _ptr(out), out.numel(), _stream_ptr(stream)),
               "pss_get_weights")
        return out

    def get_state(self, stream=None):
        torch = _torch()
        w = torch.empty(self.M, dtype=torch.float32, device="cuda")
        G = torch.empty(self.M, dtype=torch.float32, device="cuda") \
            if self.optimizer == "adagrad" else None
        _check(self._lib.pss_get_state(self._h, _ptr(w), _ptr(G) if G is not None else None,
                                       self.M, _stream_ptr(stream)), "pss_get_state")
        return w, G

    def set_state(self, w, G=None, stream=None):
        _need(w, _torch().float32, "w")
        _check(self._lib.pss_set_state(self._h, _ptr(w), _ptr(G) if G is not None else None,
                                       w.numel(), _stream_ptr(stream)), "pss_set_state")

    # -- hot path -----------------------------------------------------------
    def compute_locations(self, indices, offsets, B: int, out=None, stream=None):
        torch = _torch()
        _need(indices, torch.int64, "indices")
        _need(offsets, torch.int64, "offsets")
        if out is None:
            out = torch.empty(max(1, indices.numel() * self.J), dtype=torch.int64,
                              device=indices.device if indices.is_cuda else "cuda")
        _need(out, torch.int64, "locs")
        _check(self._lib.pss_compute_locations(self._h, _ptr(indices), indices.numel(),
                                               _ptr(offsets), int(B), _ptr(out),
                                               _stream_ptr(stream)), "pss_compute_locations")
        return out[: indices.numel() * self.J]

    def forward(self, indices, offsets, B: int, out=None, stream=None):
        """Pooled embeddings [B][T][d] (fp32).  The batch is remembered for
        the next backward call (references are kept here)."""
        torch = _torch()
        _need(indices, torch.int64, "indices")
        _need(offsets, torch.int64, "offsets")
        if offsets.numel() != self.T * int(B) + 1:
            raise ValueError("offsets must have T*B+1 entries")
        if out is None:
            dev = "cuda" if (indices.is_cuda or offsets.is_cuda) else "cpu"
            out = torch.empty((int(B), self.T, self.d), dtype=torch.float32, device=dev,
                              pin_memory=(dev == "cpu"))
        _need(out, torch.float32, "out")
        _check(self._lib.pss_forward(self._h, _ptr(indices), indices.numel(), _ptr(offsets),
                                     int(B), _ptr(out), _stream_ptr(stream)), "pss_forward")
        self._batch = (indices, offsets)
        return out

    def backward_update(self, grad_out, lr: float, stream=None):
        _need(grad_out, _torch().float32, "grad_out")
        _check(self._lib.pss_backward_update(self._h, _ptr(grad_out), ctypes.c_float(lr),
                                             _stream_ptr(stream)), "pss_backward_update")

    def backward_grad(self, grad_out, grad=None, stream=None):
        torch = _torch()
        _need(grad_out, torch.float32, "grad_out")
        if grad is None:
            grad = torch.empty(self.M, dtype=torch.float32, device="cuda")
        _need(grad, torch.float32, "grad")
        _check(self._lib.pss_backward_grad(self._h, _ptr(grad_out), _ptr(grad),
                                           _stream_ptr(stream)), "pss_backward_grad")
        return grad

    # -- options, errors, introspection --------------------------------------
    def set_option(self, key: int, value: int):
        _check(self._lib.pss_set_option(self._h, int(key), int(value)), "pss_set_option")

    def get_option(self, key: int) -> int:
        v = ctypes.c_int64()
        _check(self._lib.pss_get_option(self._h, int(key), ctypes.byref(v)), "pss_get_option")
        return int(v.value)

    def get_error(self, stream=None):
        """(status, first_bad_index) after synchronising the stream."""
        fb = ctypes.c_int64(-1)
        rc = self._lib.pss_get_error(self._h, ctypes.byref(fb), _stream_ptr(stream))
        if rc not in (PSS_OK, PSS_ERR_INDEX_RANGE):
            raise PSSError(rc, "pss_get_error")
        return rc, int(fb.value)

    def info(self) -> dict:
        inf = PSSInfo()
        _check(self._lib.pss_get_info(self._h, ctypes.byref(inf)), "pss_get_info")
        return {name: getattr(inf, name) for name, _ in PSSInfo._fields_}

    def profile(self, kernel: int):
        n, ms = ctypes.c_int64(), ctypes.c_double()
        _check(self._lib.pss_get_profile(self._h, int(kernel), ctypes.byref(n), ctypes.byref(ms)),
               "pss_get_profile")
        return int(n.value), float(ms.value)

    def reset_profile(self):
        _check(self._lib.pss_reset_profile(self._h), "pss_reset_profile")
