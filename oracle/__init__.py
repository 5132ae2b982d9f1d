"""FP64 CPU oracle of the certified cache lookup — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline /
reference arm may import this package. It wraps ``lipcache_oracle.c`` (plain
C, FP64) through ctypes and shares no code with the CUDA library.

Functions (each follows the passage cited in the C source):
  sigma_max / singular_values   Sec. 4.1, Eqs. 17-19
  logits                        Eq. 5
  certify                       Algorithm 1 with Eqs. 6, 20, 21 and Eq. 29
  probe                         Algorithm 2 with Eqs. 13-15
  pair_dist                     ||q - k||_2 for given pairs
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from .build import build as _build

_lib = None

_f32p = np.ctypeslib.ndpointer(dtype=np.float32, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")
_i32p = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(dtype=np.int64, flags="C_CONTIGUOUS")

RADIUS_CONSERVATIVE = 0
RADIUS_TIGHT = 1


def lib():
    global _lib
    if _lib is None:
        path = _build()
        L = C.CDLL(path)
        L.orc_threads.restype = C.c_int
        L.orc_singular_values.argtypes = [_f32p, C.c_int, C.c_int, _f64p, C.c_int]
        L.orc_singular_values.restype = C.c_int
        L.orc_sigma_max.argtypes = [_f32p, C.c_int, C.c_int]
        L.orc_sigma_max.restype = C.c_double
        L.orc_logits.argtypes = [_f32p, _f32p, C.c_int, C.c_int, _f32p, _f64p]
        L.orc_certify.argtypes = [_f32p, _f32p, C.c_int, C.c_int, C.c_double, C.c_int, C.c_double, _f32p,
                                  C.c_int64, C.c_void_p, C.c_int, _i32p, _i32p, _f64p, _f64p, _i32p]
        L.orc_probe.argtypes = [_f32p, _f64p, _i32p, C.c_int64, C.c_int, _f32p, C.c_int64, _i64p, _i32p, _f64p,
                                _i32p, _i32p, _i32p, C.c_double]
        L.orc_pair_dist.argtypes = [_f32p, _f32p, C.c_int, _i64p, _i64p, C.c_int64, _f64p]
        _lib = L
    return _lib


def threads() -> int:
    return int(lib().orc_threads())


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def singular_values(W) -> np.ndarray:
    W = _f32(W)
    Cn, d = W.shape
    sv = np.zeros(min(Cn, d), dtype=np.float64)
    rc = lib().orc_singular_values(W, Cn, d, sv, 100)
    if rc < 0:
        raise RuntimeError("oracle Jacobi SVD did not converge")
    return sv


def sigma_max(W) -> float:
    W = _f32(W)
    s = lib().orc_sigma_max(W, W.shape[0], W.shape[1])
    if s < 0:
        raise RuntimeError("oracle Jacobi SVD did not converge")
    return float(s)


def logits(W, b, z) -> np.ndarray:
    W, b, z = _f32(W), _f32(b), _f32(z)
    s = np.zeros(W.shape[0], dtype=np.float64)
    lib().orc_logits(W, b, W.shape[0], W.shape[1], z, s)
    return s


def certify(W, b, sigma, H, payload=None, require_consistency=False, radius_mode=RADIUS_CONSERVATIVE,
            scale=1.0) -> dict:
    """Algorithm 1 for every row of H. Returns per-row arrays: yG, label,
    margin, radius (FP64) and accept (bool)."""
    W, b, H = _f32(W), _f32(b), _f32(H)
    Cn, d = W.shape
    n = H.shape[0]
    yG = np.zeros(n, np.int32)
    label = np.zeros(n, np.int32)
    margin = np.zeros(n, np.float64)
    radius = np.zeros(n, np.float64)
    accept = np.zeros(n, np.int32)
    pl = None
    if payload is not None:
        pl = np.ascontiguousarray(payload, dtype=np.int32)
    if n:
        lib().orc_certify(W, b, Cn, d, float(sigma), int(radius_mode), float(scale), H, n,
                          pl.ctypes.data if pl is not None else None, int(bool(require_consistency)),
                          yG, label, margin, radius, accept)
    return {"yG": yG, "label": label, "margin": margin, "radius": radius, "accept": accept.astype(bool)}


def build_cache(W, b, sigma, rows, payload=None, require_consistency=False, radius_mode=RADIUS_CONSERVATIVE,
                scale=1.0) -> dict:
    """Certify rows in order and keep the accepted ones in insertion order
    (the cache C of Algorithm 1 with every candidate selected)."""
    cert = certify(W, b, sigma, rows, payload, require_consistency, radius_mode, scale)
    acc = cert["accept"]
    index = np.full(len(acc), -1, dtype=np.int64)
    index[acc] = np.arange(int(acc.sum()), dtype=np.int64)
    return {
        "keys": _f32(np.asarray(rows, dtype=np.float32)[acc]),
        "radius": np.ascontiguousarray(cert["radius"][acc]),
        "label": np.ascontiguousarray(cert["label"][acc]),
        "yG": np.ascontiguousarray(cert["yG"][acc]),
        "index": index,
        "cert": cert,
    }


def probe(keys, radius, labels, Q, band_rel=1e-5) -> dict:
    """Algorithm 2 for every query. Returns index (-1 = miss), label,
    dist (FP64, +inf on a miss), n_hits, decision_band, selection_band."""
    keys, Q = _f32(keys), _f32(Q)
    radius = np.ascontiguousarray(radius, dtype=np.float64)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    N = keys.shape[0]
    B, d = Q.shape
    if N:
        assert keys.shape[1] == d
    out = {
        "index": np.full(B, -1, np.int64), "label": np.full(B, -1, np.int32),
        "dist": np.full(B, np.inf, np.float64), "n_hits": np.zeros(B, np.int32),
        "decision_band": np.zeros(B, np.int32), "selection_band": np.zeros(B, np.int32),
    }
    if B == 0:
        return out
    if N == 0:
        keys = np.zeros((1, d), np.float32)
    lib().orc_probe(keys, radius if N else np.zeros(1), labels if N else np.zeros(1, np.int32), N, d, Q, B,
                    out["index"], out["label"], out["dist"], out["n_hits"], out["decision_band"],
                    out["selection_band"], float(band_rel))
    return out


def pair_dist(Q, K, qi, ki) -> np.ndarray:
    Q, K = _f32(Q), _f32(K)
    qi = np.ascontiguousarray(qi, dtype=np.int64)
    ki = np.ascontiguousarray(ki, dtype=np.int64)
    out = np.zeros(len(qi), np.float64)
    if len(qi):
        lib().orc_pair_dist(Q, K, Q.shape[1], qi, ki, len(qi), out)
    return out
