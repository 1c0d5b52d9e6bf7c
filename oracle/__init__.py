"""CPU oracle for the PSS hashed-embedding hot path (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package.  It shares no code with the CUDA library: the
arithmetic lives in ``pss_oracle.c`` (plain C, fp64 sums, exact 128-bit hash),
compiled here with gcc and loaded through ctypes.

Passages followed: the ROBE-Z mapping and universal hashing of Sec. 2.5, the
forward/backward of a trainable PSS in Sec. 2.4, the dense branch of
Algorithm 1 (Sec. 3), and the SGD / Adagrad updates.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pss_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

P61 = (1 << 61) - 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no fused multiply-add)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Pss(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d", ctypes.c_int64), ("M", ctypes.c_int64),
                ("Z", ctypes.c_int64), ("G", ctypes.c_int64), ("J", ctypes.c_int64),
                ("L", ctypes.c_int64), ("R", ctypes.c_int64), ("A", ctypes.c_uint64),
                ("B0", ctypes.c_uint64), ("cards", ctypes.c_void_p), ("sgn", ctypes.c_int64),
                ("A2", ctypes.c_uint64), ("B2", ctypes.c_uint64), ("circ", ctypes.c_int64)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            vp, i64, u64, f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_float
            sig = {
                "oracle_splitmix64_seq": (None, [u64, i64, vp]),
                "oracle_hash_params": (None, [u64, vp, vp]),
                "oracle_sign_params": (None, [u64, vp, vp]),
                "oracle_set_signed": (None, [vp, i64]),
                "oracle_set_circular": (ctypes.c_int, [vp, i64]),
                "oracle_sign": (i64, [vp, i64, i64, i64]),
                "oracle_signs": (ctypes.c_int, [vp, vp, i64, vp, i64, vp]),
                "oracle_init": (ctypes.c_int, [vp, vp, i64, i64, i64, i64, i64, u64]),
                "oracle_location": (i64, [vp, i64, i64, i64]),
                "oracle_locations": (ctypes.c_int, [vp, vp, i64, vp, i64, vp, vp]),
                "oracle_pool": (ctypes.c_int, [vp, vp, vp, i64, vp, i64, vp, vp]),
                "oracle_forward": (ctypes.c_int, [vp, vp, vp, i64, vp, i64, vp, vp]),
                "oracle_scatter": (ctypes.c_int, [vp, vp, i64, vp, i64, vp, vp, vp]),
                "oracle_grad": (ctypes.c_int, [vp, vp, i64, vp, i64, vp, vp, vp]),
                "oracle_grad_at": (ctypes.c_int, [vp, vp, i64, vp, i64, vp, vp, i64, vp, vp]),
                "oracle_sgd": (None, [vp, vp, i64, f32]),
                "oracle_adagrad": (None, [vp, vp, vp, i64, f32, f32]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(lib, name)
                fn.restype = res
                fn.argtypes = args
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    pass


def splitmix64_seq(seed: int, n: int) -> np.ndarray:
    out = np.zeros(n, dtype=np.uint64)
    _load().oracle_splitmix64_seq(ctypes.c_uint64(seed), n, _ptr(out))
    return out


def hash_params(seed: int):
    A, B0 = ctypes.c_uint64(), ctypes.c_uint64()
    _load().oracle_hash_params(ctypes.c_uint64(seed), ctypes.byref(A), ctypes.byref(B0))
    return int(A.value), int(B0.value)


def sign_params(seed: int):
    A2, B2 = ctypes.c_uint64(), ctypes.c_uint64()
    _load().oracle_sign_params(ctypes.c_uint64(seed), ctypes.byref(A2), ctypes.byref(B2))
    return int(A2.value), int(B2.value)


class OraclePSS:
    """One PSS instance: T tables, dim d, shared array of M fp32, chunk Z,
    block-start alignment G, hash seed.  All arrays are numpy, host memory."""

    def __init__(self, cards, d: int, M: int, Z: int, G: int = 4, seed: int = 0,
                 signed: bool = False, circular: bool = False):
        self._lib = _load()
        self.cards = _c(cards, np.int64)
        self.T = int(self.cards.shape[0])
        self.d, self.M, self.Z, self.G = int(d), int(M), int(Z), int(G)
        self._p = _Pss()
        rc = self._lib.oracle_init(ctypes.byref(self._p), _ptr(self.cards), self.T, self.d,
                                   self.M, self.Z, self.G, ctypes.c_uint64(seed))
        if rc != 0:
            raise OracleError(f"oracle_init failed ({rc})")
        self.J, self.L, self.R = int(self._p.J), int(self._p.L), int(self._p.R)
        self.A, self.B0 = int(self._p.A), int(self._p.B0)
        self.A2, self.B2 = int(self._p.A2), int(self._p.B2)
        self.signed = bool(signed)
        self._lib.oracle_set_signed(ctypes.byref(self._p), 1 if signed else 0)
        self.circular = bool(circular)
        if circular:
            rc = self._lib.oracle_set_circular(ctypes.byref(self._p), 1)
            if rc != 0:
                raise OracleError(f"oracle_set_circular failed ({rc})")
            self.R = int(self._p.R)

    def _pp(self):
        return ctypes.byref(self._p)

    def location(self, i: int, t: int, j: int) -> int:
        return int(self._lib.oracle_location(self._pp(), i, t, j))

    def locations(self, indices, offsets, B: int):
        idx, off = _c(indices, np.int64), _c(offsets, np.int64)
        locs = np.zeros(max(1, idx.shape[0] * self.J), dtype=np.int64)
        bad = ctypes.c_int64(-1)
        rc = self._lib.oracle_locations(self._pp(), _ptr(idx), idx.shape[0], _ptr(off), B,
                                        _ptr(locs), ctypes.byref(bad))
        if rc:
            raise OracleError(f"oracle_locations failed ({rc})")
        return locs[: idx.shape[0] * self.J], int(bad.value)

    def sign(self, i: int, t: int, j: int) -> int:
        """+1, or -1 for a key with an odd sign hash when signed hashing is on."""
        return int(self._lib.oracle_sign(self._pp(), i, t, j))

    def signs(self, indices, offsets, B: int):
        """Sign of every (id, chunk), laid out like locations (0 for a bad id)."""
        idx, off = _c(indices, np.int64), _c(offsets, np.int64)
        sg = np.zeros(max(1, idx.shape[0] * self.J), dtype=np.int8)
        rc = self._lib.oracle_signs(self._pp(), _ptr(idx), idx.shape[0], _ptr(off), B, _ptr(sg))
        if rc:
            raise OracleError(f"oracle_signs failed ({rc})")
        return sg[: idx.shape[0] * self.J]

    def pool(self, w, locs, offsets, B: int, nnz: int, signs=None):
        w, locs, off = _c(w, np.float32), _c(locs, np.int64), _c(offsets, np.int64)
        out = np.zeros(B * self.T * self.d, dtype=np.float32)
        sg = None if signs is None else _c(signs, np.int8)
        rc = self._lib.oracle_pool(self._pp(), _ptr(w), _ptr(locs), nnz, _ptr(off), B, _ptr(out),
                                   None if sg is None else _ptr(sg))
        if rc:
            raise OracleError(f"oracle_pool failed ({rc})")
        return out

    def forward(self, w, indices, offsets, B: int):
        w, idx, off = _c(w, np.float32), _c(indices, np.int64), _c(offsets, np.int64)
        out = np.zeros(B * self.T * self.d, dtype=np.float32)
        bad = ctypes.c_int64(-1)
        rc = self._lib.oracle_forward(self._pp(), _ptr(w), _ptr(idx), idx.shape[0], _ptr(off), B,
                                      _ptr(out), ctypes.byref(bad))
        if rc:
            raise OracleError(f"oracle_forward failed ({rc})")
        return out, int(bad.value)

    def scatter(self, locs, offsets, B: int, nnz: int, grad_out, signs=None):
        locs, off, go = _c(locs, np.int64), _c(offsets, np.int64), _c(grad_out, np.float32)
        g = np.zeros(self.M, dtype=np.float64)
        sg = None if signs is None else _c(signs, np.int8)
        rc = self._lib.oracle_scatter(self._pp(), _ptr(locs), nnz, _ptr(off), B, _ptr(go), _ptr(g),
                                      None if sg is None else _ptr(sg))
        if rc:
            raise OracleError(f"oracle_scatter failed ({rc})")
        return g

    def grad(self, indices, offsets, B: int, grad_out):
        """fp64 gradient w.r.t. the whole shared array (dense, length M)."""
        idx, off, go = _c(indices, np.int64), _c(offsets, np.int64), _c(grad_out, np.float32)
        g = np.zeros(self.M, dtype=np.float64)
        bad = ctypes.c_int64(-1)
        rc = self._lib.oracle_grad(self._pp(), _ptr(idx), idx.shape[0], _ptr(off), B, _ptr(go),
                                   _ptr(g), ctypes.byref(bad))
        if rc:
            raise OracleError(f"oracle_grad failed ({rc})")
        return g

    def grad_at(self, indices, offsets, B: int, grad_out, elems):
        """fp64 gradient at sorted distinct element positions ``elems``."""
        idx, off, go = _c(indices, np.int64), _c(offsets, np.int64), _c(grad_out, np.float32)
        el = _c(elems, np.int64)
        g = np.zeros(max(1, el.shape[0]), dtype=np.float64)
        bad = ctypes.c_int64(-1)
        rc = self._lib.oracle_grad_at(self._pp(), _ptr(idx), idx.shape[0], _ptr(off), B,
                                      _ptr(go), _ptr(el), el.shape[0], _ptr(g), ctypes.byref(bad))
        if rc:
            raise OracleError(f"oracle_grad_at failed ({rc})")
        return g[: el.shape[0]]

    @staticmethod
    def sgd(w, g32, lr: float):
        """In-place SGD on fp32 arrays (returns w)."""
        assert w.dtype == np.float32 and g32.dtype == np.float32 and w.flags.c_contiguous
        g32 = _c(g32, np.float32)
        _load().oracle_sgd(_ptr(w), _ptr(g32), w.shape[0], ctypes.c_float(lr))
        return w

    @staticmethod
    def adagrad(w, Gacc, g32, lr: float, eps: float):
        """In-place Adagrad on fp32 arrays (returns (w, Gacc))."""
        assert w.dtype == np.float32 and Gacc.dtype == np.float32
        assert w.flags.c_contiguous and Gacc.flags.c_contiguous
        g32 = _c(g32, np.float32)
        _load().oracle_adagrad(_ptr(w), _ptr(Gacc), _ptr(g32), w.shape[0], ctypes.c_float(lr),
                               ctypes.c_float(eps))
        return w, Gacc

    def step(self, w, Gacc, indices, offsets, B: int, grad_out, opt: str, lr: float,
             eps: float = 1e-10):
        """One backward + update on copies of (w, Gacc); returns (w', G', g32)."""
        g32 = self.grad(indices, offsets, B, grad_out).astype(np.float32)
        w2 = np.array(w, dtype=np.float32, copy=True)
        if opt == "sgd":
            self.sgd(w2, g32, lr)
            return w2, Gacc, g32
        G2 = np.array(Gacc, dtype=np.float32, copy=True)
        self.adagrad(w2, G2, g32, lr, eps)
        return w2, G2, g32
