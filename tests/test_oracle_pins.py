"""Pins for the FP64 oracle against what the paper and the mathematics fix.

None of these checks re-states the oracle's own formulas: they use closed
forms, hand-derived golden values (tests/golden), invariants the paper
proves (Lemma 4.1, Remark 4.2), and independent library routines (LAPACK
SVD through numpy, scipy's cKDTree — the lookup structure the paper's
device measurement uses).
"""
import numpy as np
import pytest
from scipy.spatial import cKDTree

import oracle
import synth
from conftest import golden


# ---------------------------------------------------------------- sigma_max
def test_sigma_diagonal():
    a = np.array([0.5, -3.25, 2.0, 1.0], np.float32)
    W = np.diag(a).astype(np.float32)
    assert oracle.sigma_max(W) == pytest.approx(3.25, rel=1e-15)
    sv = oracle.singular_values(W)
    np.testing.assert_allclose(sv, np.sort(np.abs(a))[::-1], rtol=1e-15)


def test_sigma_scaled_orthogonal():
    rng = np.random.default_rng(1)
    Qm, _ = np.linalg.qr(rng.standard_normal((8, 8)))
    W = (2.5 * Qm).astype(np.float32)
    # FP32 rounding of an orthogonal matrix perturbs singular values by ~1e-7.
    np.testing.assert_allclose(oracle.singular_values(W), 2.5, rtol=1e-6)


def test_sigma_rank_one():
    rng = np.random.default_rng(2)
    u = rng.standard_normal(5).astype(np.float32)
    v = rng.standard_normal(7).astype(np.float32)
    W = np.outer(u, v).astype(np.float32)
    W64 = W.astype(np.float64)
    # rank one: sigma = ||u|| ||v|| (up to the FP32 rounding of W's entries)
    assert oracle.sigma_max(W) == pytest.approx(np.linalg.norm(u.astype(np.float64)) *
                                                np.linalg.norm(v.astype(np.float64)), rel=1e-6)
    assert oracle.sigma_max(W) == pytest.approx(np.sqrt((W64 ** 2).sum()), rel=1e-13)  # rank one: ||W||_F


def test_sigma_two_rows_closed_form():
    rng = np.random.default_rng(3)
    for d in (1, 2, 5, 16):
        W = rng.standard_normal((2, d)).astype(np.float32)
        w1, w2 = W.astype(np.float64)
        a, e, c = w1 @ w1, w2 @ w2, w1 @ w2
        s2 = (a + e) / 2 + np.sqrt(((a - e) / 2) ** 2 + c * c)
        assert oracle.sigma_max(W) == pytest.approx(np.sqrt(s2), rel=1e-13)


@pytest.mark.parametrize("shape", [(10, 16), (10, 64), (100, 128), (200, 256), (40, 12), (3, 3)])
def test_sigma_vs_lapack(shape):
    rng = np.random.default_rng(shape[0] * 1000 + shape[1])
    W = (rng.standard_normal(shape) / np.sqrt(shape[1])).astype(np.float32)
    ref = np.linalg.svd(W.astype(np.float64), compute_uv=False)
    np.testing.assert_allclose(oracle.singular_values(W), ref, rtol=1e-12, atol=1e-14 * ref[0])


@pytest.mark.parametrize("name", ["tinyimagenet", "scale"])
def test_sigma_unit_spectral_heads(name):
    W, _ = synth.head(synth.WORKLOADS[name])
    assert oracle.sigma_max(W) == pytest.approx(1.0, abs=2e-6)


def test_sigma_zero_head():
    g = golden("certify_skip_rules.json")["degenerate"]
    assert oracle.sigma_max(np.array(g["W"], np.float32)) == g["sigma"]


# ---------------------------------------------------------------- radius
def test_golden_two_class():
    g = golden("radius_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    s = oracle.sigma_max(W)
    assert s == pytest.approx(g["sigma"], rel=1e-15)
    rows = np.array(g["rows"], np.float32)
    c = oracle.certify(W, b, s, rows)
    assert list(c["yG"]) == g["yG"]
    np.testing.assert_allclose(c["margin"], g["margin"], rtol=1e-15)
    np.testing.assert_allclose(c["radius"], g["radius"], rtol=1e-15)
    ct = oracle.certify(W, b, s, rows, radius_mode=oracle.RADIUS_TIGHT)
    np.testing.assert_allclose(ct["radius"], g["radius_tight"], rtol=1e-15)
    cache = oracle.build_cache(W, b, s, rows)
    out = oracle.probe(cache["keys"], cache["radius"], cache["label"], np.array(g["queries"], np.float32))
    assert list(out["index"]) == g["expect_index"]
    for dist, exp in zip(out["dist"], g["expect_dist"]):
        if exp is None:
            assert dist == np.inf
        else:
            assert dist == pytest.approx(exp, rel=1e-6)


def test_golden_three_class():
    for case in golden("radius_three_class.json")["cases"]:
        W, b = np.array(case["W"], np.float32), np.array(case["b"], np.float32)
        z = np.array([case["z"]], np.float32)
        s = oracle.sigma_max(W)
        assert s == pytest.approx(case["sigma"], rel=1e-15)
        c = oracle.certify(W, b, s, z)
        assert c["yG"][0] == case["yG"]
        assert c["margin"][0] == pytest.approx(case["margin"], rel=1e-15)
        assert c["radius"][0] == pytest.approx(case["radius"], rel=1e-15)
        ct = oracle.certify(W, b, s, z, radius_mode=oracle.RADIUS_TIGHT)
        assert ct["radius"][0] == pytest.approx(case["radius_tight"], rel=1e-15)
        assert ct["radius"][0] >= c["radius"][0]


def test_golden_radius_tightening():
    """Sec. 5.6: kappa multiplies the radius itself (not r^2), in both radius
    modes, after certification: a row's acceptance does not depend on kappa
    in (0, 1], and a hit needs D < kappa r (strict)."""
    for case in golden("radius_tightening.json")["cases"]:
        W, b = np.array(case["W"], np.float32), np.array(case["b"], np.float32)
        rows = np.array(case["rows"], np.float32)
        s = oracle.sigma_max(W)
        assert s == pytest.approx(case["sigma"], rel=1e-15)
        kappa = case["kappa"]
        for mode, key in ((oracle.RADIUS_CONSERVATIVE, "radius"), (oracle.RADIUS_TIGHT, "radius_tight")):
            c = oracle.certify(W, b, s, rows, radius_mode=mode, scale=kappa)
            assert list(c["accept"]) == case["accept"]
            np.testing.assert_allclose(c["radius"], case[key], rtol=1e-15, atol=0)
            # acceptance is the same at kappa = 1 and the radius is kappa times it
            c1 = oracle.certify(W, b, s, rows, radius_mode=mode)
            assert list(c1["accept"]) == case["accept"]
            np.testing.assert_allclose(c["radius"], kappa * c1["radius"], rtol=1e-15, atol=0)
        if "queries" in case:
            Q = np.array(case["queries"], np.float32)
            cache = oracle.build_cache(W, b, s, rows, scale=kappa)
            out = oracle.probe(cache["keys"], cache["radius"], cache["label"], Q)
            assert list(out["index"]) == case["expect_index"]
            cache1 = oracle.build_cache(W, b, s, rows)
            out1 = oracle.probe(cache1["keys"], cache1["radius"], cache1["label"], Q)
            assert list(out1["index"]) == case["expect_index_kappa1"]


def test_golden_skip_rules():
    g = golden("certify_skip_rules.json")
    t = g["tie"]
    W, b = np.array(t["W"], np.float32), np.array(t["b"], np.float32)
    c = oracle.certify(W, b, oracle.sigma_max(W), np.array(t["rows"], np.float32))
    assert list(c["accept"].astype(int)) == t["accept"]
    np.testing.assert_array_equal(c["radius"], t["radius"])
    k = g["consistency"]
    W, b = np.array(k["W"], np.float32), np.array(k["b"], np.float32)
    rows = np.array(k["rows"], np.float32)
    pl = np.array(k["payload"], np.int32)
    req = oracle.certify(W, b, 1.0, rows, payload=pl, require_consistency=True)
    free = oracle.certify(W, b, 1.0, rows, payload=pl, require_consistency=False)
    assert list(req["yG"]) == k["yG"]
    assert list(req["accept"].astype(int)) == k["accept_required"]
    assert list(free["accept"].astype(int)) == k["accept_free"]
    assert list(free["label"]) == k["label"]
    proxy = oracle.certify(W, b, 1.0, rows)
    assert list(proxy["label"]) == k["yG"]  # proxy payload = y^G


def _random_head(rng, C, d, antisymmetric=False):
    if antisymmetric:
        w = rng.standard_normal(d)
        beta = rng.standard_normal() * 0.3
        return np.stack([w, -w]).astype(np.float32), np.array([beta, -beta], np.float32)
    return rng.standard_normal((C, d)).astype(np.float32), (rng.standard_normal(C) * 0.3).astype(np.float32)


def _argmax_fp64(W, b, Z):
    return np.argmax(Z.astype(np.float64) @ W.astype(np.float64).T + b.astype(np.float64), axis=1)


def _ball_points(rng, centre, radius, n):
    d = centre.shape[0]
    u = rng.standard_normal((n, d))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    rad = radius * rng.random(n) ** (1.0 / d)
    rad[: n // 4] = radius  # a quarter on the sphere itself
    return centre[None, :] + u * rad[:, None]


@pytest.mark.parametrize("C,d,anti", [(2, 2, True), (2, 3, True), (2, 4, False), (3, 2, False), (5, 4, False),
                                      (4, 3, False)])
def test_lemma_label_invariant(C, d, anti):
    """Lemma 4.1: every point strictly inside r keeps the cached GuardNet
    label. For the antisymmetric 2-class heads r equals the distance to the
    decision hyperplane, so an r that is too large (e.g. a dropped sqrt 2)
    is caught here."""
    rng = np.random.default_rng(C * 100 + d + 7 * anti)
    for _ in range(20):
        W, b = _random_head(rng, C, d, anti)
        s = oracle.sigma_max(W)
        rows = (rng.standard_normal((8, d)) * 2).astype(np.float32)
        c = oracle.certify(W, b, s, rows)
        for i in np.nonzero(c["accept"])[0]:
            pts = _ball_points(rng, rows[i].astype(np.float64), c["radius"][i] * (1 - 1e-9), 400)
            assert np.all(_argmax_fp64(W, b, pts) == c["yG"][i])


@pytest.mark.parametrize("C,d", [(2, 3), (3, 2), (4, 4), (6, 3)])
def test_tight_radius_is_boundary_distance(C, d):
    """Remark 4.2: r* >= r, the label is kept strictly inside r*, and r* is
    attained: just beyond r* along the minimising facet normal the label
    flips (the decision region is an intersection of half-spaces)."""
    rng = np.random.default_rng(C * 10 + d)
    for _ in range(25):
        W, b = _random_head(rng, C, d)
        s = oracle.sigma_max(W)
        rows = (rng.standard_normal((6, d)) * 2).astype(np.float32)
        cons = oracle.certify(W, b, s, rows)
        tight = oracle.certify(W, b, s, rows, radius_mode=oracle.RADIUS_TIGHT)
        for i in range(len(rows)):
            if not tight["accept"][i]:
                continue
            r, rs, y = cons["radius"][i], tight["radius"][i], tight["yG"][i]
            assert rs >= r * (1 - 1e-12)
            z = rows[i].astype(np.float64)
            pts = _ball_points(rng, z, rs * (1 - 1e-9), 300)
            assert np.all(_argmax_fp64(W, b, pts) == y)
            # Find the facet that is reached first by moving against W_y - W_j.
            flipped = False
            for j in range(C):
                if j == y:
                    continue
                n = W[y].astype(np.float64) - W[j].astype(np.float64)
                p = z - n / np.linalg.norm(n) * rs * (1 + 1e-7)
                if _argmax_fp64(W, b, p[None, :])[0] != y:
                    flipped = True
            assert flipped


# ---------------------------------------------------------------- probe
def test_golden_probe_selection():
    g = golden("probe_selection.json")
    out = oracle.probe(np.array(g["keys"], np.float32), np.array(g["radius"]), np.array(g["labels"], np.int32),
                       np.array(g["queries"], np.float32))
    assert list(out["index"]) == g["expect_index"]
    assert list(out["label"]) == g["expect_label"]
    assert list(out["n_hits"]) == g["expect_n_hits"]
    for dist, exp in zip(out["dist"], g["expect_dist"]):
        assert (dist == np.inf) if exp is None else (dist == exp)


@pytest.mark.parametrize("N,d,B", [(200, 3, 100), (500, 8, 64), (64, 16, 32)])
def test_probe_vs_ckdtree(N, d, B):
    """Nearest certified hit from scipy's cKDTree (all neighbours sorted by
    distance; the first one inside its own radius)."""
    rng = np.random.default_rng(N + d)
    keys = rng.standard_normal((N, d)).astype(np.float32)
    radius = rng.random(N) * 1.2
    labels = rng.integers(0, 10, N).astype(np.int32)
    Q = np.concatenate([keys[rng.integers(0, N, B // 2)] + 0.1 * rng.standard_normal((B // 2, d)),
                        rng.standard_normal((B - B // 2, d))]).astype(np.float32)
    out = oracle.probe(keys, radius, labels, Q)
    tree = cKDTree(keys.astype(np.float64))
    dist, idx = tree.query(Q.astype(np.float64), k=N)
    for q in range(B):
        hit = dist[q] < radius[idx[q]]
        assert out["n_hits"][q] == hit.sum()
        if hit.any():
            j = np.argmax(hit)
            assert out["index"][q] == idx[q][j]
            assert out["label"][q] == labels[idx[q][j]]
            assert out["dist"][q] == pytest.approx(dist[q][j], rel=1e-12)
        else:
            assert out["index"][q] == -1 and out["label"][q] == -1 and out["dist"][q] == np.inf


def test_probe_band_flags():
    keys = np.zeros((2, 2), np.float32)
    keys[1] = [4.0, 0.0]
    radius = np.array([1.0, 1.0])
    labels = np.array([1, 2], np.int32)
    Q = np.array([[1.0 + 5e-6, 0.0], [0.5, 0.0], [2.0, 0.0], [0.3, 0.0]], np.float32)
    out = oracle.probe(keys, radius, labels, Q, band_rel=1e-5)
    assert list(out["decision_band"]) == [1, 0, 0, 0]
    assert list(out["index"]) == [-1, 0, -1, 0]
    # two equidistant hits -> selection band
    keys2 = np.array([[0.0, 0.0], [1.0, 0.0]], np.float32)
    out2 = oracle.probe(keys2, np.array([1.0, 1.0]), labels, np.array([[0.5, 0.0]], np.float32))
    assert out2["selection_band"][0] == 1 and out2["index"][0] == 0


def test_empty_cache_and_batch():
    out = oracle.probe(np.zeros((0, 4), np.float32), np.zeros(0), np.zeros(0, np.int32),
                       np.ones((3, 4), np.float32))
    assert list(out["index"]) == [-1, -1, -1]
    out = oracle.probe(np.ones((3, 4), np.float32), np.ones(3), np.zeros(3, np.int32), np.zeros((0, 4), np.float32))
    assert len(out["index"]) == 0


def test_pair_dist_matches_probe():
    rng = np.random.default_rng(5)
    K = rng.standard_normal((50, 6)).astype(np.float32)
    Q = rng.standard_normal((4, 6)).astype(np.float32)
    out = oracle.probe(K, np.full(50, 10.0), np.zeros(50, np.int32), Q)
    d = oracle.pair_dist(Q, K, np.arange(4), out["index"])
    np.testing.assert_array_equal(d, out["dist"])


def test_certify_logits_vs_matmul():
    rng = np.random.default_rng(9)
    W = rng.standard_normal((7, 13)).astype(np.float32)
    b = rng.standard_normal(7).astype(np.float32)
    z = rng.standard_normal(13).astype(np.float32)
    ref = W.astype(np.float64) @ z.astype(np.float64) + b
    np.testing.assert_allclose(oracle.logits(W, b, z), ref, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("mode", [oracle.RADIUS_CONSERVATIVE, oracle.RADIUS_TIGHT])
def test_non_finite_rows_skipped(mode):
    """A row with an infinite or NaN feature has no defined margin (Eq. 20)
    nor terms of Eq. 29, so it is skipped in either mode. The first row makes
    exactly one logit +inf and the others -inf (margin inf - (-inf) = +inf,
    which a plain evaluation would accept with an infinite radius); the
    finite rows are certified as usual."""
    W = np.array([[1, 0], [-1, 0], [-1, 1]], np.float32)
    b = np.zeros(3, np.float32)
    H = np.array([[np.inf, 0], [np.nan, 1], [2, -np.inf], [3, 1], [-2, 0.5]], np.float32)
    cert = oracle.certify(W, b, oracle.sigma_max(W), H, radius_mode=mode)
    assert cert["accept"].tolist() == [False, False, False, True, True]
    assert np.all(np.isnan(cert["radius"][:3]))
    assert np.all(np.isfinite(cert["radius"][3:])) and np.all(cert["radius"][3:] > 0)
