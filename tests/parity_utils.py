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


def refine_slack(W, b, rows, kappa=1.0):
    """Largest amount by which the GPU's reported conservative radius may
    exceed the exact one: the two refined logits (compensated FP32 dot
    products) are each within 2 gamma_{d+40}^2 (||W_c|| ||z|| + |b_c|) of
    the exact logits, and r = kappa m / (sigma sqrt 2) (Eq. 21)."""
    W64 = np.asarray(W, np.float64)
    d = W64.shape[1]
    u = 2.0 ** -24
    g = (d + 40) * u / (1 - (d + 40) * u)
    scale = np.linalg.norm(W64, axis=1).max() * np.linalg.norm(np.asarray(rows, np.float64), axis=1)
    scale += np.abs(np.asarray(b, np.float64)).max()
    return kappa * 4 * g * g * scale / (oracle.sigma_max(W) * np.sqrt(2.0)) * (1 + 1e-6)


def refine_slack_tight(W, b, rows, kappa=1.0):
    """The same for the tight radius (Eq. 29) computed from compensated FP32
    refinements: r* = kappa (s_y - s_j) / ||W_y - W_j|| with both logits
    within 2 gamma_{d+40}^2 (||W_c|| ||z|| + |b_c|) of the exact ones."""
    W64 = np.asarray(W, np.float64)
    d = W64.shape[1]
    u = 2.0 ** -24
    g = (d + 40) * u / (1 - (d + 40) * u)
    scale = np.linalg.norm(W64, axis=1).max() * np.linalg.norm(np.asarray(rows, np.float64), axis=1)
    scale += np.abs(np.asarray(b, np.float64)).max()
    pn = np.linalg.norm(W64[:, None, :] - W64[None, :, :], axis=2)
    pmin = pn[pn > 0].min() if np.any(pn > 0) else 1.0
    return kappa * 4 * g * g * scale / pmin * (1 + 1e-6)


def check_insert(g_index, g_radius, n_acc, ref, head=None):
    """head = (W, b, rows, kappa) for the conservative radius and
    ("tight", W, b, rows, kappa) for the tight radius from compensated FP32
    refinements: the reported radius (the refined value, rounded toward zero)
    must then not exceed the exact one by more than the refinement's error
    bound. Without it (tight radius, FP64 refinement of every class) the bound
    is 1e-12 relative."""
    cert = ref["cert"]
    assert n_acc == int(cert["accept"].sum())
    bad = np.nonzero(g_index != ref["index"])[0]
    assert bad.size == 0, f"{bad.size} rows differ in acceptance/index, first {bad[:5]}"
    r = cert["radius"]
    m = np.isfinite(r) & (r > 0)
    if head is None:
        slack = r * 1e-12
    elif isinstance(head[0], str) and head[0] == "tight":
        slack = r * 1e-12 + refine_slack_tight(*head[1:])
    else:
        slack = refine_slack(*head)
    g = g_radius[m].astype(np.float64)
    # within 1e-5 relative, or within the refinement's proven absolute error
    # where that is larger (radii of entries a hair from a decision boundary,
    # below ~1e-6 of the logit scale); never above the exact radius by more
    # than that error
    err = np.abs(g - r[m])
    bad = np.nonzero(err > RTOL * r[m] + slack[m])[0]
    assert bad.size == 0, f"{bad.size} radii off, e.g. {g[bad[:3]]} vs {r[m][bad[:3]]}"
    assert np.all(g <= r[m] + slack[m])


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
            "band": int(band.sum()), "band_mismatch": int((mism & band).sum())}
