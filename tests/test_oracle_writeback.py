"""Pins for the oracle's write-back (Algorithm 2, miss branch) and its
certified-consistency check (Sec. 5 metrics, Lemma of Sec. 4.2).

Hand-derived golden values (tests/golden), the Lemma as an invariant, and an
independent FP64 argmax through numpy's matmul.
"""
import numpy as np
import pytest

import oracle
from conftest import golden


def _cache(W, b, sigma, rows):
    c = oracle.build_cache(np.array(W, np.float32), np.array(b, np.float32), sigma, np.array(rows, np.float32))
    return {"keys": c["keys"], "radius": c["radius"], "label": c["label"], "yG": c["yG"]}


def test_golden_writeback_proxy_labels():
    g = golden("writeback_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache = _cache(W, b, g["sigma"], g["rows"])
    r = oracle.probe_writeback(cache, W, b, g["sigma"], np.array(g["queries"], np.float32))
    assert r["probe"]["index"].tolist() == g["expect_index"]
    assert r["inserted"].tolist() == g["expect_inserted"]
    np.testing.assert_allclose(r["cache"]["radius"], g["expect_radius"], rtol=1e-15)
    assert r["cache"]["yG"].tolist() == g["expect_yG"]
    assert r["cache"]["label"].tolist() == g["expect_yG"]  # proxy label = y^G
    q = np.array(g["queries"], np.float32)
    np.testing.assert_array_equal(r["cache"]["keys"][1:], q[r["inserted"] >= 0])


def test_golden_writeback_require_consistency():
    g = golden("writeback_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache = _cache(W, b, g["sigma"], g["rows"])
    r = oracle.probe_writeback(cache, W, b, g["sigma"], np.array(g["queries"], np.float32),
                               payload=np.array(g["payload"], np.int32), require_consistency=True)
    assert r["inserted"].tolist() == g["expect_inserted_consistent"]
    assert r["cache"]["label"].tolist() == g["expect_label_consistent"]


@pytest.mark.parametrize("which", ["inflated", "certified"])
def test_golden_consistency(which):
    g = golden("consistency_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    keys = np.array(g["keys"], np.float32)
    Q = np.array(g["queries"], np.float32)
    radius = np.array([g["radius_" + which]], np.float64)
    p = oracle.probe(keys, radius, np.array(g["yG"], np.int32), Q)
    assert p["index"].tolist() == g["expect_hit_" + which]
    c = oracle.consistency(W, b, Q, p["index"], np.array(g["yG"], np.int32))
    assert c["consistent"].tolist() == g["expect_consistent_" + which]
    exp = np.array(g["expect_consistent_" + which])
    assert c["n_hits"] == int((exp >= 0).sum()) and c["n_consistent"] == int((exp == 1).sum())


def _instance(seed, C, d, n_rows, n_q):
    rng = np.random.default_rng(seed)
    W = rng.standard_normal((C, d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = (2 * rng.standard_normal((n_rows, d))).astype(np.float32)
    return rng, W, b, rows


@pytest.mark.parametrize("seed,C,d", [(0, 3, 2), (1, 5, 4), (2, 4, 8)])
def test_writeback_batch_semantics(seed, C, d):
    """The batch is probed against the old cache (same result as a plain
    probe), only misses are written back, in query order, and each
    written-back query hits the grown cache (it lies at distance 0 from its
    own entry, whose radius is positive)."""
    rng, W, b, rows = _instance(seed, C, d, 24, 64)
    s = oracle.sigma_max(W)
    cache = _cache(W, b, s, rows)
    Q = (2 * rng.standard_normal((64, d))).astype(np.float32)
    Q[::4] = rows[rng.integers(0, len(rows), 16)] + 0.01  # some hits
    r = oracle.probe_writeback(cache, W, b, s, Q)
    plain = oracle.probe(cache["keys"], cache["radius"], cache["label"], Q)
    np.testing.assert_array_equal(r["probe"]["index"], plain["index"])
    ins = r["inserted"]
    assert np.all(ins[plain["index"] >= 0] == -1)
    n0 = len(cache["keys"])
    new = ins[ins >= 0]
    np.testing.assert_array_equal(new, n0 + np.arange(len(new)))
    assert np.all(r["cache"]["radius"][n0:] > 0)
    again = oracle.probe(r["cache"]["keys"], r["cache"]["radius"], r["cache"]["label"], Q[ins >= 0])
    assert np.all(again["index"] >= 0)
    assert np.all(again["dist"] == 0.0)


def _argmax_numpy(W, b, Q):
    s = Q.astype(np.float64) @ W.astype(np.float64).T + b.astype(np.float64)
    return np.argmax(s, axis=1)


@pytest.mark.parametrize("seed,C,d", [(3, 2, 2), (4, 3, 3), (5, 6, 4)])
def test_consistency_lemma_and_planted_radius(seed, C, d):
    """Certified radii: every hit strictly inside r(1 - 1e-9) is consistent
    (the Lemma). Radii inflated 4x: the check flags exactly the hits whose
    numpy FP64 argmax differs from the entry's y^G."""
    rng, W, b, rows = _instance(seed, C, d, 16, 0)
    s = oracle.sigma_max(W)
    cache = _cache(W, b, s, rows)
    n = len(cache["keys"])
    assert n > 0
    pick = rng.integers(0, n, 400)
    u = rng.standard_normal((400, d))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    Q = (cache["keys"][pick] + u * (cache["radius"][pick] * rng.random(400) * 3.5)[:, None]).astype(np.float32)

    p = oracle.probe(cache["keys"], cache["radius"], cache["label"], Q)
    c = oracle.consistency(W, b, Q, p["index"], cache["yG"])
    hit = p["index"] >= 0
    assert c["n_hits"] == int(hit.sum()) > 0
    inner = hit & (p["dist"] < cache["radius"][np.maximum(p["index"], 0)] * (1 - 1e-9))
    assert np.all(c["consistent"][inner] == 1)

    big = cache["radius"] * 4
    p4 = oracle.probe(cache["keys"], big, cache["label"], Q)
    c4 = oracle.consistency(W, b, Q, p4["index"], cache["yG"])
    h4 = p4["index"] >= 0
    want = (_argmax_numpy(W, b, Q) == cache["yG"][np.maximum(p4["index"], 0)]).astype(np.int8)
    clear = h4 & (c4["gap"] > 1e-9)
    np.testing.assert_array_equal(c4["consistent"][clear], want[clear])
    assert np.all(c4["consistent"][~h4] == -1)
    assert c4["n_consistent"] < c4["n_hits"]  # the inflated radii do cross the boundary


# ---------------------------------------------------------------- empirical radii
def test_golden_interclass_radius():
    g = golden("interclass_radius.json")
    r = oracle.interclass_radius(np.array(g["keys"], np.float32), g["labels"], g["C"], g["beta"])
    np.testing.assert_allclose(r["rho"], g["expect_rho"], rtol=1e-15)
    np.testing.assert_allclose(r["radius"], g["expect_radius"], rtol=1e-15)
    half = oracle.interclass_radius(np.array(g["keys"], np.float32), g["labels"], g["C"], 0.5 * g["beta"])
    np.testing.assert_allclose(half["rho"], 0.5 * np.array(g["expect_rho"]), rtol=1e-15)
    one = oracle.interclass_radius(np.array(g["single_class_keys"], np.float32), g["single_class_labels"], g["C"])
    assert one["rho"].tolist() == g["expect_single_class_rho"]


def test_interclass_radius_invariances():
    """Centroid distances are invariant under a common translation and entry
    order and scale with the keys; checked against a numpy centroid
    computation (np.add.at) of the same statistic."""
    rng = np.random.default_rng(9)
    keys = rng.standard_normal((300, 5)) * 3
    labels = rng.integers(0, 6, 300)
    base = oracle.interclass_radius(keys, labels, 7, 0.8)
    sums = np.zeros((7, 5))
    np.add.at(sums, labels, keys)
    cnt = np.bincount(labels, minlength=7)
    mu = sums[:6] / cnt[:6, None]
    D = np.sqrt(((mu[:, None, :] - mu[None, :, :]) ** 2).sum(-1)) + np.diag(np.full(6, np.inf))
    np.testing.assert_allclose(base["rho"][:6], 0.4 * D.min(1), rtol=1e-12)
    assert base["rho"][6] == 0.0  # class 6 has no entries
    perm = rng.permutation(300)
    np.testing.assert_allclose(oracle.interclass_radius(keys[perm], labels[perm], 7, 0.8)["rho"], base["rho"],
                               rtol=1e-12)
    np.testing.assert_allclose(oracle.interclass_radius(keys + 7.5, labels, 7, 0.8)["rho"], base["rho"], rtol=1e-9)
    np.testing.assert_allclose(oracle.interclass_radius(keys * 4, labels, 7, 0.8)["rho"], 4 * base["rho"],
                               rtol=1e-12)


def test_global_radius_hits_nearest_within_tau():
    """With one global radius, a query hits iff its nearest cached entry is
    closer than tau (checked with scipy's cKDTree)."""
    from scipy.spatial import cKDTree
    rng = np.random.default_rng(4)
    keys = rng.standard_normal((200, 3)).astype(np.float32)
    Q = rng.standard_normal((300, 3)).astype(np.float32)
    tau = 0.3
    p = oracle.probe(keys, oracle.global_radius(200, tau), np.arange(200, dtype=np.int32), Q)
    dist, idx = cKDTree(keys.astype(np.float64)).query(Q.astype(np.float64))
    clear = np.abs(dist - tau) > 1e-9
    np.testing.assert_array_equal((p["index"] >= 0)[clear], (dist < tau)[clear])
    hit = (p["index"] >= 0) & clear
    np.testing.assert_array_equal(p["index"][hit], idx[hit])


# ---------------------------------------------------------------- selection strategy S
def test_golden_select_radius_dedup():
    g = golden("select_radius_dedup.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    rows = np.array(g["rows"], np.float32)
    cert = oracle.certify(W, b, g["sigma"], rows)
    assert oracle.select_radius_dedup(rows, cert).tolist() == g["expect"]
    assert oracle.select_radius_dedup(rows, cert, budget_per_class=1, n_classes=2).tolist() == g["expect_per_class_1"]
    assert oracle.select_radius_dedup(rows, cert, budget_total=2).tolist() == g["expect_total_2"]
    sel = oracle.select_radius_dedup(rows, cert, keys0=np.array(g["existing_keys"], np.float32),
                                     radius0=np.array(g["existing_radius"]))
    assert sel.tolist() == g["expect_with_existing"]


def _check_greedy(rows, cert, sel, keys0, radius0, budget_total, budget_per_class, C):
    """The selection is the unique greedy result for the visiting order iff
    (i) no kept entry lies inside the ball of an entry kept before it and
    (ii) every candidate not kept lies inside such a ball or met an
    exhausted budget at its turn. Checked here by brute force over the order."""
    r32 = oracle.radius_rz32(cert["radius"])
    order = sorted(np.nonzero(cert["accept"])[0].tolist(), key=lambda i: (-float(r32[i]), i))
    chosen = set(sel.tolist())
    kept_z = [z.astype(np.float64) for z in keys0]
    kept_r = list(radius0)
    per, total, pos = {}, 0, 0
    for i in order:
        z = rows[i].astype(np.float64)
        covered = any(np.linalg.norm(z - kz) < kr for kz, kr in zip(kept_z, kept_r))
        c = int(cert["label"][i])
        full = (budget_total and total >= budget_total) or (budget_per_class and per.get(c, 0) >= budget_per_class)
        if i in chosen:
            assert not covered and not full
            assert sel[pos] == i  # kept entries come out in visiting order
            pos += 1
            kept_z.append(z)
            kept_r.append(float(cert["radius"][i]))
            per[c] = per.get(c, 0) + 1
            total += 1
        else:
            assert covered or full
    assert pos == len(sel)


@pytest.mark.parametrize("seed,C,d,bt,bc", [(0, 3, 2, 0, 0), (1, 4, 3, 0, 3), (2, 5, 2, 7, 0), (3, 2, 4, 0, 0),
                                            (4, 6, 3, 10, 2)])
def test_select_radius_dedup_is_the_greedy(seed, C, d, bt, bc):
    rng, W, b, rows = _instance(seed, C, d, 300, 0)
    rows = (0.5 * rows).astype(np.float32)  # dense enough that balls overlap
    s = oracle.sigma_max(W)
    cert = oracle.certify(W, b, s, rows)
    keys0 = rows[:5] + np.float32(0.01)
    radius0 = np.full(5, 0.3)
    sel = oracle.select_radius_dedup(rows, cert, keys0, radius0, bt, bc, C)
    assert 0 < len(sel) < int(cert["accept"].sum())
    _check_greedy(rows, cert, sel, keys0, radius0, bt, bc, C)
    if bt:
        assert len(sel) <= bt
    if bc:
        assert np.bincount(cert["label"][sel], minlength=C).max() <= bc


def test_radius_rz32_rounds_toward_zero():
    r = np.array([1.0, 0.1, 1 / 3, 2.0 ** -130, 3.5e38, 0.0, np.inf])
    f = oracle.radius_rz32(r)
    assert np.all(f.astype(np.float64)[:6] <= r[:6]) and f[6] == np.inf
    with np.errstate(over="ignore"):
        nxt = np.nextafter(f[:6], np.float32(np.inf)).astype(np.float64)
    assert np.all(nxt > r[:6])  # the largest FP32 value not above r


def test_golden_select_kcenter():
    g = golden("select_kcenter.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    rows = np.array(g["rows"], np.float32)
    cert = oracle.certify(W, b, g["sigma"], rows)
    assert oracle.select_kcenter(rows, cert, 3, 2)["selected"].tolist() == g["budget_3"]
    assert oracle.select_kcenter(rows, cert, 1, 2)["selected"].tolist() == g["budget_1"]
    tie = np.array(g["tie_rows"], np.float32)
    ct = oracle.certify(W, b, g["sigma"], tie)
    assert oracle.select_kcenter(tie, ct, 2, 2)["selected"].tolist() == g["tie_budget_2"]


@pytest.mark.parametrize("seed,C,d,k", [(0, 3, 2, 5), (1, 4, 3, 8), (2, 2, 5, 20)])
def test_select_kcenter_farthest_point(seed, C, d, k):
    """Brute force: per class the first centre has the largest radius and
    every next centre is at least as far from the earlier centres as any
    other candidate; a class with fewer candidates than the budget keeps all."""
    rng, W, b, rows = _instance(seed, C, d, 200, 0)
    cert = oracle.certify(W, b, oracle.sigma_max(W), rows)
    sel = oracle.select_kcenter(rows, cert, k, C)["selected"]
    for c in range(C):
        cand = np.nonzero(cert["accept"] & (cert["label"] == c))[0]
        mine = [i for i in sel.tolist() if cert["label"][i] == c]
        assert len(mine) == min(k, len(cand))
        if not mine:
            continue
        assert cert["radius"][mine[0]] == cert["radius"][cand].max()
        for t in range(1, len(mine)):
            centres = rows[mine[:t]].astype(np.float64)
            dmin = lambda i: np.min(np.linalg.norm(centres - rows[i].astype(np.float64), axis=1))
            others = [i for i in cand if i not in mine[:t]]
            assert dmin(mine[t]) >= max(dmin(i) for i in others) - 1e-12
