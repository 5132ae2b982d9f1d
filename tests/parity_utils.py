"""Comparison rules between the CUDA path and the FP64 oracle.

Bit-exact: acceptance of inserted rows, cache indices, hit/miss decisions,
selected indices and labels. Within 1e-5 relative: radii and distances.
The only tolerated disagreements are queries in the oracle's 1e-5 band:
some entry has |D - r| <= 1e-5 r (decision band) or the two nearest hits
are within 1e-5 of each other (selection band). A GPU hit the oracle
rejects (an unsafe accept) is never tolerated.
"""
import numpy as np

import oracle

RTOL = 1e-5


def fp64_band(W, b, rows, kappa=1.0, tight=False, chunk=1 << 16):
    """Rows whose radius FP64 arithmetic itself cannot pin to 1e-5 relative,
    and the absolute slack allowed for their radii (0 elsewhere).

    The oracle and the GPU's FP64 pass each compute a logit within
    gamma_{d+8} (sum_j |W_cj z_j| + |b_c|) of its exact value, below
    res = 1.01 (d + 8) 2^-53 (max_c ||W_c|| ||z|| + max_c |b_c|). A radius
    taken from a logit difference m (Eq. 21: the top-two margin; Eq. 29: the
    numerator s_y - s_j of the minimising term) is then known to 4 res / m
    relative on both sides together, which exceeds 1e-5 only when
    m < 4e5 res; the top-two gap also decides y^G in both radius modes. Such
    rows (a hair from a decision boundary, e.g. the tests' constructed near
    ties) get the absolute slack 4 res kappa / (sigma sqrt 2) (conservative)
    or 4 res kappa / min ||W_y - W_j|| (tight). The logits here are numpy
    FP64, used only to classify rows."""
    W64 = np.asarray(W, np.float64)
    b64 = np.asarray(b, np.float64)
    rows = np.asarray(rows, np.float32)
    n, d = rows.shape[0], W64.shape[1]
    wmax = np.linalg.norm(W64, axis=1).max()
    bmax = np.abs(b64).max()
    band = np.zeros(n, bool)
    res_all = np.zeros(n)
    PN = np.stack([np.linalg.norm(W64 - W64[y], axis=1) for y in range(W64.shape[0])]) if tight else None
    for s0 in range(0, n, chunk):
        z = rows[s0:s0 + chunk].astype(np.float64)
        res = 1.01 * (d + 8) * 2.0 ** -53 * (wmax * np.linalg.norm(z, axis=1) + bmax)
        s = z @ W64.T + b64
        top = np.partition(s, -2, axis=1)[:, -2:]
        with np.errstate(invalid="ignore"):
            gap = top[:, 1] - top[:, 0]
            bnd = gap < 4e5 * res
        if tight:
            y = np.argmax(s, axis=1)
            k = np.arange(len(z))
            pn = PN[y]
            with np.errstate(divide="ignore", invalid="ignore"):  # rows with NaN / infinite features
                num = s[k, y][:, None] - s
                t = np.where(pn > 0, num / pn, np.inf)
            t[k, y] = np.inf
            j = np.argmin(t, axis=1)
            with np.errstate(invalid="ignore"):
                bnd |= np.isfinite(t[k, j]) & (num[k, j] < 4e5 * res)
        band[s0:s0 + chunk] = bnd
        res_all[s0:s0 + chunk] = res
    if tight:
        pmin = PN[PN > 0].min() if np.any(PN > 0) else 1.0
        slack = kappa * 4 * res_all / pmin
    else:
        slack = kappa * 4 * res_all / (oracle.sigma_max(W) * np.sqrt(2.0))
    return band, np.where(band, slack, 0.0)


def radius_tol(W, b, rows, r, kappa=1.0, tight=False):
    """Allowed |GPU radius - exact radius| per row: 1e-5 relative, plus the
    FP64-resolution slack of fp64_band for the rows it marks."""
    _, slack = fp64_band(W, b, rows, kappa, tight)
    return RTOL * np.abs(np.asarray(r, np.float64)) + slack


def check_insert(g_index, g_radius, n_acc, ref, head=None):
    """Acceptance and indices bit-exact; every accepted row's radius within
    1e-5 relative of the oracle's FP64 radius (Eq. 21, or Eq. 29 for
    head = ("tight", W, b, rows, kappa); head = (W, b, rows, kappa) for the
    conservative radius), except rows at FP64's own resolution (fp64_band),
    which get its slack. head=None: kernels that refine every class in FP64
    (1e-5 relative, the rounding of the FP32 result included). Returns how
    many rows were in the FP64 band."""
    cert = ref["cert"]
    assert n_acc == int(cert["accept"].sum())
    bad = np.nonzero(g_index != ref["index"])[0]
    assert bad.size == 0, f"{bad.size} rows differ in acceptance/index, first {bad[:5]}"
    r = cert["radius"]
    m = np.isfinite(r) & (r > 0)
    n_band = 0
    if head is None:
        tol = RTOL * r + r * 1e-12
    else:
        tight = isinstance(head[0], str) and head[0] == "tight"
        W, b, rows, kappa = head[1:] if tight else head
        band, slack = fp64_band(W, b, rows, kappa, tight)
        tol = RTOL * r + slack
        n_band = int((band & m).sum())
    g = g_radius[m].astype(np.float64)
    err = np.abs(g - r[m])
    bad = np.nonzero(err > tol[m])[0]
    assert bad.size == 0, f"{bad.size} radii off, e.g. {g[bad[:3]]} vs {r[m][bad[:3]]}"
    return {"rows": int(len(r)), "accepted": int(m.sum()), "fp64_band": n_band}


def check_probe(gi, gl, gd, ref, Q, orc):
    keys, radius, labels = ref["keys"], ref["radius"], ref["label"]
    hits = gi >= 0
    if hits.any():
        qi = np.nonzero(hits)[0]
        D = oracle.pair_dist(Q, keys, qi, gi[hits])
        unsafe = ~(D < radius[gi[hits]])
        assert not unsafe.any(), f"{unsafe.sum()} unsafe accepts, e.g. query {qi[unsafe][:3]}"
        assert np.array_equal(gl[hits], labels[gi[hits]])
        np.testing.assert_allclose(gd[hits].astype(np.float64), D, rtol=RTOL)
    assert np.all(gl[~hits] == -1) and np.all(np.isinf(gd[~hits]))
    band = (orc["decision_band"] | orc["selection_band"]).astype(bool)
    mism = gi != orc["index"]
    out = mism & ~band
    assert not out.any(), (f"{out.sum()} queries differ outside the 1e-5 band: "
                           f"gpu {gi[out][:5]} oracle {orc['index'][out][:5]}")
    return {"queries": len(gi), "hits": int(hits.sum()), "oracle_hits": int((orc["index"] >= 0).sum()),
            "identical": int((~mism).sum()), "band": int(band.sum()),
            "decision_band": int(orc["decision_band"].astype(bool).sum()),
            "selection_band": int(orc["selection_band"].astype(bool).sum()),
            "band_mismatch": int((mism & band).sum()), "unsafe_accepts": 0}


def record_parity(workload, path, stats):
    """Append one parity record (the counts check_probe returns, the unsafe
    accepts among them asserted to be 0) as a JSON line to the file named by
    LIPCACHE_PARITY_OUT, when that variable is set."""
    import json
    import os
    dst = os.environ.get("LIPCACHE_PARITY_OUT")
    if dst:
        with open(dst, "a") as f:
            f.write(json.dumps({"workload": workload, "path": path, **stats}) + "\n")
