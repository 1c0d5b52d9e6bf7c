"""Seeded synthetic inputs shaped like the paper's Criteo workloads.

The paper trains on Criteo-Kaggle and Criteo-TB (Sec. 4, "Datasets" and
"Models": 26 categorical features, a 40M cap on ids per table, d = 128 for
Criteo-TB) and micro-benchmarks the lookup at batch 10240, d = 128 (Sec. 3,
Fig. "smallt").  Neither dataset is available here, so every input below is a
seeded synthetic stand-in with the same shapes and value distributions:
table cardinalities, Zipf-distributed ids, bag lengths, initial weights and
upstream gradients.

This module holds none of the method's arithmetic (no hashing, no pooling, no
gradient, no optimizer).  It is the one module that both the CUDA path's tests
and the CPU oracle's tests take their inputs from.

Layout conventions (shared by every consumer):
  * ``offsets`` is CSR over bags in table-major order: bag (t, b) is slot
    ``t*B + b`` and owns ``indices[offsets[s]:offsets[s+1]]``;
  * ``grad_out`` / pooled outputs are row-major ``[B][T][d]`` (DLRM concat order);
  * ids are int64, values float32.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

__all__ = [
    "Workload",
    "CONFIGS",
    "make_workload",
    "make_batch",
    "scaled_loguniform_cardinalities",
    "loguniform_cardinalities",
    "zipf_ids",
    "w0_normal",
    "w0_periodic_base",
    "dyadic",
]

# Criteo-TB shape: 26 tables capped at 40M ids, about 195M rows in total.
TB_TABLES = 26
TB_CAP = 40_000_000
TB_TOTAL_ROWS = 195_000_000

# Named workloads.  Sizes follow the paper's Criteo shapes; see module doc.
CONFIGS = {
    # 8 tables x 1000 ids, d=16, M=16384, one uniform id per bag, SGD lr 0.1.
    "tiny": dict(T=8, cards=("const", 1000), d=16, M=16384, Z=16, B=256,
                 bag=("one",), ids=("uniform",), opt="sgd", lr=0.1),
    # Criteo-Kaggle shaped: log-uniform cardinalities in [3, 10M], d=16, M=1Mi.
    "kaggle": dict(T=26, cards=("loguniform", 3, 10_000_000), d=16, M=1 << 20, Z=32,
                   B=2048, bag=("one",), ids=("zipf", 1.05), opt="adagrad", lr=0.01),
    # Criteo-TB shaped, 10000x compression: M = 2.5M fp32 (10 MB), d=128.
    "tb": dict(T=26, cards=("scaled", 3, TB_CAP, TB_TOTAL_ROWS), d=128, M=2_500_000,
               Z=32, B=65536, bag=("one",), ids=("zipf", 1.05), opt="adagrad", lr=0.01),
    # Multi-hot contention: Poisson(20) bags, Zipf(1.2) ids, d=64, SGD.
    "multihot": dict(T=26, cards=("scaled", 3, TB_CAP, TB_TOTAL_ROWS), d=64, M=2_500_000,
                     Z=32, B=16384, bag=("poisson", 20.0), ids=("zipf", 1.2), opt="sgd",
                     lr=0.1),
    # Compression sweep: the Criteo-TB shape with M chosen by the caller.
    "sweep": dict(T=26, cards=("scaled", 3, TB_CAP, TB_TOTAL_ROWS), d=128, M=None, Z=32,
                  B=65536, bag=("one",), ids=("zipf", 1.05), opt="adagrad", lr=0.01),
    # The paper's micro-benchmark shape (batch 10240, d=128, loss = sum of outputs,
    # so the upstream gradient is all ones).
    "microbench": dict(T=26, cards=("scaled", 3, TB_CAP, TB_TOTAL_ROWS), d=128,
                       M=2_500_000, Z=32, B=10240, bag=("one",), ids=("zipf", 1.05),
                       opt="sgd", lr=0.1, grad="ones"),
}

# Above this many elements the initial array is a tiled 2^24-element pattern,
# so that huge shared arrays need no multi-GB host buffer.
PERIODIC_W0_ABOVE = 1 << 28
W0_PERIOD = 1 << 24


@dataclasses.dataclass
class Workload:
    """One PSS problem instance plus one batch of inputs."""
    name: str
    T: int
    d: int
    M: int
    Z: int
    G: int
    B: int
    opt: str
    lr: float
    eps: float
    seed: int
    cards: np.ndarray                 # int64[T]
    indices: np.ndarray               # int64[nnz]
    offsets: np.ndarray               # int64[T*B+1], table-major
    grad_out: Optional[np.ndarray]    # float32[B*T*d] or None
    w0: Optional[np.ndarray]          # float32[M], or None when periodic
    w0_base: Optional[np.ndarray]     # float32[W0_PERIOD] when periodic

    @property
    def nnz(self) -> int:
        return int(self.indices.shape[0])

    def w0_at(self, elems: np.ndarray) -> np.ndarray:
        """Initial weights at the given element positions."""
        if self.w0 is not None:
            return self.w0[elems]
        return self.w0_base[np.asarray(elems, dtype=np.int64) % W0_PERIOD]


def _streams(seed: int, n: int = 6):
    """Independent generators per purpose: cards, ids, bags, w0, grad, spare."""
    return [np.random.Generator(np.random.PCG64(s))
            for s in np.random.SeedSequence(seed).spawn(n)]


def loguniform_cardinalities(rng, T: int, lo: int, hi: int) -> np.ndarray:
    """T cardinalities drawn log-uniformly in [lo, hi]."""
    u = np.exp(rng.uniform(math.log(lo), math.log(hi), size=T))
    return np.clip(np.rint(u), lo, hi).astype(np.int64)


def scaled_loguniform_cardinalities(rng, T: int, lo: int, cap: int, total: int) -> np.ndarray:
    """Log-uniform draws in [lo, cap], rescaled by one common factor so that the
    capped total is close to ``total`` rows (Criteo-TB: 26 tables, 40M cap,
    about 195M rows)."""
    u = np.exp(rng.uniform(math.log(lo), math.log(cap), size=T))

    def tot(c):
        return int(np.clip(np.rint(c * u), lo, cap).sum())

    a, b = 1e-3, 1e6
    for _ in range(200):
        m = math.sqrt(a * b)
        if tot(m) < total:
            a = m
        else:
            b = m
    return np.clip(np.rint(b * u), lo, cap).astype(np.int64)


def zipf_ids(rng, n: int, s: float, count: int) -> np.ndarray:
    """``count`` ids in [0, n) with P(id = r-1) proportional to r^-s (Zipf
    truncated at n)."""
    if count == 0:
        return np.zeros(0, dtype=np.int64)
    if n <= (1 << 22):
        r = np.arange(1, n + 1, dtype=np.float64)
        cdf = np.cumsum(r ** (-s))
        cdf /= cdf[-1]
        u = rng.random(count)
        ids = np.searchsorted(cdf, u, side="right")
        return np.minimum(ids, n - 1).astype(np.int64)
    out = np.empty(count, dtype=np.int64)
    filled = 0
    while filled < count:
        need = count - filled
        z = rng.zipf(s, size=int(need * 1.6) + 64)
        z = z[(z >= 1) & (z <= n)][:need]
        out[filled:filled + z.shape[0]] = z - 1
        filled += z.shape[0]
    return out


def dyadic(rng, size, k_max: int = 1 << 10, scale_log2: int = 8) -> np.ndarray:
    """Values k / 2^scale_log2 with |k| < k_max.  Sums of such values stay exact
    in fp32 while they are below 2^24 / 2^scale_log2 in magnitude, so any
    summation order gives the same bits."""
    k = rng.integers(-(k_max - 1), k_max, size=size)
    return (k.astype(np.float64) / float(1 << scale_log2)).astype(np.float32)


def w0_normal(rng, M: int, std: float = 0.01) -> np.ndarray:
    """N(0, std^2) fp32 initial weights (the conventional normal_(0, 0.01))."""
    return (rng.standard_normal(M, dtype=np.float32) * np.float32(std)).astype(np.float32)


def w0_periodic_base(rng, std: float = 0.01) -> np.ndarray:
    """Base pattern of a huge initial array: w0[e] = base[e mod 2^24]."""
    return w0_normal(rng, W0_PERIOD, std)


def _cards(spec, T, rng) -> np.ndarray:
    kind = spec[0]
    if kind == "const":
        return np.full(T, spec[1], dtype=np.int64)
    if kind == "loguniform":
        return loguniform_cardinalities(rng, T, spec[1], spec[2])
    if kind == "scaled":
        return scaled_loguniform_cardinalities(rng, T, spec[1], spec[2], spec[3])
    if kind == "explicit":
        return np.asarray(spec[1], dtype=np.int64)
    raise ValueError(f"unknown cardinality spec {spec!r}")


def _bag_lengths(spec, T, B, rng) -> np.ndarray:
    kind = spec[0]
    if kind == "one":
        return np.ones(T * B, dtype=np.int64)
    if kind == "poisson":
        return rng.poisson(spec[1], size=T * B).astype(np.int64)
    if kind == "uniform":            # lengths uniform in [lo, hi] (ragged tests)
        return rng.integers(spec[1], spec[2] + 1, size=T * B).astype(np.int64)
    raise ValueError(f"unknown bag spec {spec!r}")


def _ids(spec, cards, lengths, B, rng) -> np.ndarray:
    T = cards.shape[0]
    per_table = lengths.reshape(T, B).sum(axis=1)
    parts = []
    for t in range(T):
        n, cnt = int(cards[t]), int(per_table[t])
        if spec[0] == "uniform":
            parts.append(rng.integers(0, n, size=cnt).astype(np.int64))
        elif spec[0] == "zipf":
            parts.append(zipf_ids(rng, n, spec[1], cnt))
        else:
            raise ValueError(f"unknown id spec {spec!r}")
    return np.concatenate(parts) if parts else np.zeros(0, dtype=np.int64)


def make_batch(cards: np.ndarray, B: int, d: int, bag=("one",), ids=("zipf", 1.05),
               seed: int = 0, batch: int = 0, grad: str = "normal"):
    """One batch: (indices, offsets, grad_out).  ``batch`` selects an
    independent batch of the same distribution."""
    T = int(cards.shape[0])
    streams = _streams(seed * 1_000_003 + batch, 6)
    lengths = _bag_lengths(bag, T, B, streams[2])
    offsets = np.zeros(T * B + 1, dtype=np.int64)
    np.cumsum(lengths, out=offsets[1:])
    indices = _ids(ids, cards, lengths, B, streams[1])
    if grad == "normal":
        grad_out = streams[4].standard_normal(B * T * d, dtype=np.float32)
    elif grad == "ones":
        grad_out = np.ones(B * T * d, dtype=np.float32)
    elif grad == "dyadic":
        grad_out = dyadic(streams[4], B * T * d)
    elif grad == "none":
        grad_out = None
    else:
        raise ValueError(grad)
    return indices, offsets, grad_out


def make_workload(name: str, seed: int = 0, batch: int = 0, M: Optional[int] = None,
                  B: Optional[int] = None, Z: Optional[int] = None, G: int = 4,
                  grad: Optional[str] = None, w0: str = "normal",
                  eps: float = 1e-10, **overrides) -> Workload:
    """Build a named workload (see ``CONFIGS``).  ``M``, ``B`` and ``Z``
    override the config's sizes; ``w0`` is "normal" or "dyadic"."""
    cfg = dict(CONFIGS[name])
    cfg.update(overrides)
    if M is not None:
        cfg["M"] = M
    if B is not None:
        cfg["B"] = B
    if Z is not None:
        cfg["Z"] = Z
    if cfg["M"] is None:
        raise ValueError("this config needs an explicit M")
    grad = grad or cfg.get("grad", "normal")
    st = _streams(seed, 6)
    cards = _cards(cfg["cards"], cfg["T"], st[0])
    indices, offsets, grad_out = make_batch(cards, cfg["B"], cfg["d"], cfg["bag"], cfg["ids"],
                                            seed=seed, batch=batch, grad=grad)
    Mv = int(cfg["M"])
    w0_arr, base = None, None
    if w0 == "dyadic":
        w0_arr = dyadic(st[3], Mv)
    elif Mv > PERIODIC_W0_ABOVE:
        base = w0_periodic_base(st[3])
    else:
        w0_arr = w0_normal(st[3], Mv)
    return Workload(name=name, T=int(cfg["T"]), d=int(cfg["d"]), M=Mv, Z=int(cfg["Z"]), G=G,
                    B=int(cfg["B"]), opt=cfg["opt"], lr=float(cfg["lr"]), eps=eps, seed=seed,
                    cards=cards, indices=indices, offsets=offsets, grad_out=grad_out,
                    w0=w0_arr, w0_base=base)
