"""Seeded synthetic workloads for the certified cache lookup.

This module only draws random numbers. It holds none of the lookup's
arithmetic (no logits, margins, radii or distances), so both the FP64 CPU
oracle and the CUDA library consume the same FP32 bytes from here while
sharing no code with each other.

The paper evaluates on GuardNet features of CIFAR-10, SVHN and Tiny-ImageNet
(Sec. 5.1). Neither the datasets nor trained GuardNet weights are available,
so each workload is a Gaussian mixture in the GuardNet feature space with the
feature dimension d, class count C, cache size N and query batch of the
corresponding setting:

* ``m`` mixture components with equal weights; centre = R * g / ||g||,
  g ~ N(0, I_d); a sample is centre + s * N(0, I_d).
* head W ~ N(0, 1/d) (C x d); for the Lipschitz-constrained heads W is
  rescaled in FP64 so that ||W||_2 = 1 before the FP32 cast (the rescale
  uses LAPACK through ``numpy.linalg.norm``; it is input synthesis, not part
  of either implementation under test).
* bias b ~ N(0, 0.01) read as variance 0.01 (std 0.1).
* queries: a fraction ``dup`` are near-duplicates, i.e. a uniformly random
  inserted cache row plus N(0, noise^2) per dimension; the rest are fresh
  mixture draws. Which query slots are near-duplicates is a random subset.

Every draw comes from ``numpy.random.default_rng([seed, stream])`` with one
stream per role so that, e.g., the query draw does not depend on how many
cache rows were generated in chunks.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import numpy as np

# Independent random streams, one per role.
_STREAM_CENTRES = 0
_STREAM_W = 1
_STREAM_B = 2
_STREAM_ROWS = 3
_STREAM_QUERIES = 4

_ROW_CHUNK = 1 << 18  # rows generated per chunk (bounds host memory)


@dataclass(frozen=True)
class Workload:
    name: str
    d: int                 # GuardNet feature dimension
    C: int                 # classes
    components: int        # mixture components
    sphere_radius: float   # R: centres lie on the sphere of this radius
    sigma: float           # per-dimension std of a mixture draw
    N: int                 # cache rows inserted
    n_queries: int         # total queries
    batch: int             # probe batch size
    insert_batch: int      # rows per insert call
    dup_frac: float        # fraction of near-duplicate queries
    noise: float           # std of the near-duplicate perturbation
    unit_spectral: bool    # rescale W to ||W||_2 = 1
    seed: int = 0

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    # d=16, C=10, 10 components on a radius-4 sphere, sigma 0.5; N=1,024; 256 queries, half near-duplicates.
    "tiny": Workload("tiny", 16, 10, 10, 4.0, 0.5, 1024, 256, 256, 1024, 0.5, 0.05, False),
    # CIFAR-10-shaped: d=64, C=10, R=6, sigma 0.6; N=50,000; 10,000 queries in batches of 256, 40% near-duplicates.
    "cifar10": Workload("cifar10", 64, 10, 10, 6.0, 0.6, 50_000, 10_000, 256, 65_536, 0.4, 0.05, False),
    # CIFAR-100-shaped: d=128, C=100, R=8, sigma 0.7; N=50,000; 10,000 queries in batches of 1,024, 30% near-duplicates.
    "cifar100": Workload("cifar100", 128, 100, 100, 8.0, 0.7, 50_000, 10_000, 1024, 65_536, 0.3, 0.05, False),
    # Tiny-ImageNet-shaped: d=256, C=200, R=10, sigma 0.8; N=100,000; 10,000 queries in batches of 4,096, 30%
    # near-duplicates; W rescaled to ||W||_2 = 1.
    "tinyimagenet": Workload("tinyimagenet", 256, 200, 200, 10.0, 0.8, 100_000, 10_000, 4096, 65_536, 0.3, 0.05, True),
    # Scale stress: d=128 with the Tiny-ImageNet mixture and head recipe; N=4,000,000 inserted in batches of
    # 65,536; probed in batches of 4,096 queries, 25% near-duplicates.
    "scale": Workload("scale", 128, 200, 200, 10.0, 0.8, 4_000_000, 16_384, 4096, 65_536, 0.25, 0.05, True),
}


def _rng(w: Workload, stream: int) -> np.random.Generator:
    return np.random.default_rng([w.seed, stream])


def centres(w: Workload) -> np.ndarray:
    g = _rng(w, _STREAM_CENTRES).standard_normal((w.components, w.d))
    g /= np.linalg.norm(g, axis=1, keepdims=True)
    return g * w.sphere_radius  # float64, (m, d)


def head(w: Workload) -> tuple[np.ndarray, np.ndarray]:
    """Return (W, b) as contiguous FP32 arrays of shapes (C, d) and (C,)."""
    W = _rng(w, _STREAM_W).standard_normal((w.C, w.d)) / np.sqrt(w.d)
    if w.unit_spectral:
        W = W / np.linalg.norm(W, 2)
    b = _rng(w, _STREAM_B).standard_normal(w.C) * 0.1
    return np.ascontiguousarray(W, dtype=np.float32), np.ascontiguousarray(b, dtype=np.float32)


def _mixture(rng: np.random.Generator, ctr: np.ndarray, n: int, sigma: float) -> np.ndarray:
    comp = rng.integers(0, ctr.shape[0], size=n)
    x = rng.standard_normal((n, ctr.shape[1]), dtype=np.float32)
    x *= np.float32(sigma)
    x += ctr[comp].astype(np.float32)
    return x


def cache_rows(w: Workload) -> np.ndarray:
    """All N cache rows (FP32, N x d), generated in fixed-size chunks."""
    ctr = centres(w)
    rng = _rng(w, _STREAM_ROWS)
    out = np.empty((w.N, w.d), dtype=np.float32)
    for s in range(0, w.N, _ROW_CHUNK):
        e = min(w.N, s + _ROW_CHUNK)
        out[s:e] = _mixture(rng, ctr, e - s, w.sigma)
    return out


def queries(w: Workload, rows: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Return (Q, src): Q is n_queries x d FP32; src[i] is the cache row a
    near-duplicate query was drawn around, or -1 for a fresh draw."""
    ctr = centres(w)
    rng = _rng(w, _STREAM_QUERIES)
    nq = w.n_queries
    n_dup = int(round(w.dup_frac * nq))
    slots = rng.permutation(nq)[:n_dup]
    src = np.full(nq, -1, dtype=np.int64)
    src[slots] = rng.integers(0, rows.shape[0], size=n_dup)
    Q = _mixture(rng, ctr, nq, w.sigma)
    noise = rng.standard_normal((n_dup, w.d), dtype=np.float32) * np.float32(w.noise)
    Q[slots] = rows[src[slots]] + noise
    return Q, src


def batches(n: int, size: int):
    """(start, stop) pairs covering range(n) in order; the last may be ragged."""
    return [(s, min(n, s + size)) for s in range(0, n, size)]
