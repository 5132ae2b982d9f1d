"""FP64 CPU oracle of the certified cache lookup — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline /
reference arm may import this package. It wraps ``lipcache_oracle.c`` (plain
C, FP64) through ctypes and shares no code with the CUDA library.

Functions (each follows the passage cited in the C source):
  sigma_max / singular_values   Sec. 4.1, Eqs. 17-19
  logits                        Eq. 5
  certify                       Algorithm 1 with Eqs. 6, 20, 21 and Eq. 29
  probe                         Algorithm 2 with Eqs. 13-15
  probe_writeback               Algorithm 2 with write-back of certified misses
  consistency                   certified-consistency rate of the hits (Sec. 5)
  interclass_radius             empirical inter-class-distance radius (Sec. 5.4)
  global_radius                 one global threshold for every entry (Sec. 5.4)
  select_radius_dedup           selection S: radius-prioritised de-duplication (Algorithm 1, Sec. 5.5)
  radius_rz32                   FP32 radius rounded toward zero (the order key of the selection)
  select_kcenter                selection S: K-center per class (Sec. 5.5)
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


def probe_writeback(cache, W, b, sigma, Q, payload=None, require_consistency=False,
                    radius_mode=RADIUS_CONSERVATIVE, scale=1.0, band_rel=1e-5) -> dict:
    """Algorithm 2 with write-back enabled. The distances D_{k,i} are formed
    once for the whole batch against the cache as it stood when the batch
    arrived, so no query of a batch sees another query's write-back. Every
    missed query is then certified as in Algorithm 1 (payload: the given
    labels, else the proxy label y^G) and, if accepted, appended in query
    order. ``cache`` holds keys / radius / label / yG as returned by
    build_cache. Returns the probe result, ``inserted`` (new cache index of
    each written-back query, -1 otherwise) and the grown cache."""
    res = probe(cache["keys"], cache["radius"], cache["label"], Q, band_rel)
    Q = _f32(Q)
    cert = certify(W, b, sigma, Q, payload, require_consistency, radius_mode, scale)
    add = (res["index"] < 0) & cert["accept"]
    n0 = int(np.asarray(cache["keys"]).shape[0])
    inserted = np.full(Q.shape[0], -1, dtype=np.int64)
    inserted[add] = n0 + np.arange(int(add.sum()), dtype=np.int64)
    grown = {
        "keys": _f32(np.concatenate([np.asarray(cache["keys"], np.float32).reshape(n0, Q.shape[1]), Q[add]])),
        "radius": np.concatenate([np.asarray(cache["radius"], np.float64), cert["radius"][add]]),
        "label": np.concatenate([np.asarray(cache["label"], np.int32), cert["label"][add]]).astype(np.int32),
        "yG": np.concatenate([np.asarray(cache["yG"], np.int32), cert["yG"][add]]).astype(np.int32),
    }
    return {"probe": res, "inserted": inserted, "cert": cert, "cache": grown}


def consistency(W, b, Q, hit_index, yG_table) -> dict:
    """Certified-consistency check of the hits (the rate reported in Sec. 5):
    for every query with hit_index >= 0, whether the head's argmax on the
    query (FP64 logits, Eq. 5; lowest class on ties) equals y^G of the hit
    entry. ``consistent`` is 1 / 0 per hit and -1 on a miss; ``gap`` is the
    query's FP64 top-two logit gap (+inf on a miss), for band exclusion."""
    Q = _f32(Q)
    hit_index = np.asarray(hit_index, dtype=np.int64)
    yG_table = np.asarray(yG_table, dtype=np.int32)
    B = Q.shape[0]
    out = np.full(B, -1, dtype=np.int8)
    gap = np.full(B, np.inf)
    for k in np.nonzero(hit_index >= 0)[0]:
        s = logits(W, b, Q[k])
        y = int(np.argmax(s))
        top = np.sort(s)
        gap[k] = top[-1] - top[-2]
        out[k] = 1 if y == int(yG_table[hit_index[k]]) else 0
    n_hits = int((hit_index >= 0).sum())
    return {"consistent": out, "n_hits": n_hits, "n_consistent": int((out == 1).sum()), "gap": gap}


def global_radius(n, tau) -> np.ndarray:
    """The global nearest-neighbour threshold compared with the certified
    radius in Sec. 5.4: one radius tau for every cache entry, so a query hits
    its nearest entry iff that entry is closer than tau."""
    return np.full(int(n), float(tau), dtype=np.float64)


def interclass_radius(keys, labels, n_classes, beta=1.0) -> dict:
    """The empirical inter-class-distance radius compared with the certified
    radius in Sec. 5.4. Reading (the paper names only "inter-class distance
    statistics"): mu_c = mean of the cached keys with label c (FP64);
    rho_c = beta / 2 * min over present classes c' != c of ||mu_c - mu_c'||,
    i.e. beta times half the distance to the nearest other class centroid;
    every entry gets rho of its label. Labels outside [0, C), classes without
    entries, and classes with no other class present get radius 0."""
    keys = np.asarray(keys, dtype=np.float64)
    labels = np.asarray(labels, dtype=np.int64)
    C = int(n_classes)
    n, d = keys.shape if keys.ndim == 2 else (0, 0)
    count = np.zeros(C, dtype=np.int64)
    total = np.zeros((C, d), dtype=np.float64)
    for i in range(n):
        c = int(labels[i])
        if 0 <= c < C:
            count[c] += 1
            total[c] += keys[i]
    present = count > 0
    mu = np.zeros_like(total)
    mu[present] = total[present] / count[present][:, None]
    rho = np.zeros(C, dtype=np.float64)
    for c in range(C):
        if not present[c]:
            continue
        best = np.inf
        for c2 in range(C):
            if c2 != c and present[c2]:
                best = min(best, float(np.sqrt(np.sum((mu[c] - mu[c2]) ** 2))))
        rho[c] = 0.0 if not np.isfinite(best) else beta * 0.5 * best
    radius = np.zeros(n, dtype=np.float64)
    ok = (labels >= 0) & (labels < C)
    radius[ok] = rho[labels[ok]]
    return {"rho": rho, "radius": radius, "centroid": mu, "count": count}


def radius_rz32(r) -> np.ndarray:
    """FP64 radii rounded toward zero to FP32 (NaN stays NaN)."""
    r = np.asarray(r, dtype=np.float64)
    with np.errstate(over="ignore"):
        f = r.astype(np.float32)  # beyond the FP32 range: inf, corrected below
    over = np.isfinite(r) & (np.abs(f.astype(np.float64)) > np.abs(r))
    f[over] = np.nextafter(f[over], np.float32(0))
    return f


def select_radius_dedup(rows, cert, keys0=None, radius0=None, budget_total=0, budget_per_class=0, n_classes=0):
    """Selection strategy S of Algorithm 1, read as radius-prioritised
    de-duplication (the default strategy of Sec. 5.5; the paper gives no
    formula). The certified candidates (cert["accept"]) are visited in order
    of decreasing radius, the radius rounded toward zero to FP32 (ties: lower
    row first). A candidate is skipped if it lies strictly inside the
    certified ball of an entry already kept -- an entry of the existing cache
    (keys0, radius0) or one selected earlier in this pass -- i.e. if the
    lookup would already hit it (Eq. 13), or if its class (payload label in
    [0, C)) has budget_per_class selected entries or the pass has
    budget_total (0 = unlimited). Returns the selected rows in visiting
    order."""
    rows = np.asarray(rows, dtype=np.float32)
    acc = np.asarray(cert["accept"], dtype=bool)
    r64 = np.asarray(cert["radius"], dtype=np.float64)
    lab = np.asarray(cert["label"], dtype=np.int64)
    r32 = radius_rz32(r64)
    cand = np.nonzero(acc)[0]
    order = sorted(cand.tolist(), key=lambda i: (-float(r32[i]), i))
    k0 = np.asarray(keys0 if keys0 is not None else np.zeros((0, rows.shape[1])), dtype=np.float64)
    r0 = np.asarray(radius0 if radius0 is not None else np.zeros(0), dtype=np.float64)
    kept_z = np.zeros((len(k0) + len(cand), rows.shape[1]), dtype=np.float64)  # entries kept so far
    kept_r = np.zeros(len(k0) + len(cand), dtype=np.float64)
    kept_z[:len(k0)] = k0
    kept_r[:len(k0)] = r0
    m = len(k0)
    per = {}
    out = []
    for i in order:
        if budget_total and len(out) >= budget_total:
            break
        c = int(lab[i])
        if budget_per_class and 0 <= c < max(n_classes, 1) and per.get(c, 0) >= budget_per_class:
            continue
        z = rows[i].astype(np.float64)
        # the lookup of Eq. 13 against every entry kept so far (direct differences, FP64)
        if m and np.any(np.sqrt(np.sum((kept_z[:m] - z) ** 2, axis=1)) < kept_r[:m]):
            continue
        out.append(i)
        kept_z[m] = z
        kept_r[m] = r64[i]
        m += 1
        per[c] = per.get(c, 0) + 1
    return np.asarray(out, dtype=np.int64)


def select_kcenter(rows, cert, budget_per_class, n_classes) -> dict:
    """Selection strategy S read as K-center (the alternative named in
    Sec. 5.5; no formula given): for each class c (payload label in [0, C))
    among the certified candidates, Gonzalez's farthest-point greedy: the
    first centre is the candidate with the largest certified radius, each
    next one the candidate farthest (Euclidean, FP64) from the centres chosen
    so far; ties go to the lower row; stop at budget_per_class centres or
    when the class is exhausted. Returns the selected rows (classes in
    ascending order, each class in selection order) and, per step, the
    relative gap between the chosen candidate's distance and the runner-up's
    (to tell near-ties apart)."""
    rows = np.asarray(rows, dtype=np.float32)
    acc = np.asarray(cert["accept"], dtype=bool)
    lab = np.asarray(cert["label"], dtype=np.int64)
    rad = np.asarray(cert["radius"], dtype=np.float64)
    out, gaps = [], []
    for c in range(int(n_classes)):
        cand = np.nonzero(acc & (lab == c))[0]
        if len(cand) == 0 or budget_per_class <= 0:
            continue
        Z = rows[cand].astype(np.float64)
        r = rad[cand]
        first = int(np.lexsort((cand, -r))[0])  # largest radius, then lowest row
        chosen = [first]
        mind = np.sqrt(np.sum((Z - Z[first]) ** 2, axis=1))
        mind[first] = -1.0
        while len(chosen) < min(budget_per_class, len(cand)):
            best = float(mind.max())
            j = int(np.nonzero(mind == best)[0][0])  # candidates are in row order: lowest row on ties
            rest = np.delete(mind, j)
            second = float(rest.max()) if len(rest) else -1.0
            gaps.append((best - second) / best if best > 0 else 0.0)
            chosen.append(j)
            mind = np.minimum(mind, np.sqrt(np.sum((Z - Z[j]) ** 2, axis=1)))
            mind[chosen] = -1.0
        out.extend(cand[chosen].tolist())
    return {"selected": np.asarray(out, dtype=np.int64), "gaps": np.asarray(gaps)}


def pair_dist(Q, K, qi, ki) -> np.ndarray:
    Q, K = _f32(Q), _f32(K)
    qi = np.ascontiguousarray(qi, dtype=np.int64)
    ki = np.ascontiguousarray(ki, dtype=np.int64)
    out = np.zeros(len(qi), np.float64)
    if len(qi):
        lib().orc_pair_dist(Q, K, Q.shape[1], qi, ki, len(qi), out)
    return out
