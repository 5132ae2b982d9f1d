"""Selection strategy S (radius-prioritised de-duplication), CUDA path vs the
FP64 oracle through the C ABI (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from conftest import golden

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def T(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def make_cache(dev, W, b, capacity):
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], capacity, device=dev)
    c.set_head(T(W, dev), T(b, dev))
    return c


def kept_in_order(index):
    """Rows kept by the GPU, in the order they were appended."""
    rows = np.nonzero(index >= 0)[0]
    return rows[np.argsort(index[rows])]


@pytest.mark.parametrize("variant", ["plain", "per_class", "total", "existing"])
def test_golden_select(dev, variant):
    g = golden("select_radius_dedup.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    rows = np.array(g["rows"], np.float32)
    cache = make_cache(dev, W, b, 16)
    kw = {}
    if variant == "per_class":
        kw = {"budget_per_class": 1}
    elif variant == "total":
        kw = {"budget_total": 2}
    elif variant == "existing":
        cache.insert(T(np.array(g["existing_keys"], np.float32), dev))  # radius |y| = 1.5 under this head
    idx, rad, n = cache.insert_select(T(rows, dev), **kw)
    idx = idx.cpu().numpy()
    want = {"plain": g["expect"], "per_class": g["expect_per_class_1"], "total": g["expect_total_2"],
            "existing": g["expect_with_existing"]}[variant]
    assert kept_in_order(idx).tolist() == want
    assert n == len(want)
    base = 1 if variant == "existing" else 0
    assert sorted(idx[idx >= 0].tolist()) == list(range(base, base + len(want)))
    np.testing.assert_allclose(rad.cpu().numpy()[:6], np.abs(rows[:6, 1]), rtol=1e-6)
    # the kept rows are looked up as themselves
    gi, _, gd = cache.probe(T(rows[want], dev))
    assert gi.cpu().numpy().tolist() == list(range(base, base + len(want)))
    cache.close()


def check_selection(rows, cert, g_index, g_radius, keys0, radius0, budget_total=0, budget_per_class=0, C=0):
    """The GPU's choice is a greedy selection in its own visiting order (its
    FP32 radii, ties to the lower row) whose coverage decisions agree with
    FP64 distances and radii outside the 1e-5 band: a skipped row is always
    exactly covered (or over budget); a kept row is never covered unless it
    sits in the band of a ball. Returns the number of band events."""
    acc = np.nonzero(cert["accept"])[0]
    order = sorted(acc.tolist(), key=lambda i: (-float(g_radius[i]), i))
    kept = kept_in_order(g_index)
    pos = {r: k for k, r in enumerate(kept.tolist())}
    z_k = np.zeros((len(keys0) + len(order), rows.shape[1]))
    r_k = np.zeros(len(keys0) + len(order))
    z_k[:len(keys0)] = np.asarray(keys0, np.float64)
    r_k[:len(keys0)] = radius0
    m = len(keys0)
    per, total, nxt, band = {}, 0, 0, 0
    for i in order:
        z = rows[i].astype(np.float64)
        D = np.sqrt(np.sum((z_k[:m] - z) ** 2, axis=1))
        R = r_k[:m]
        covered = bool(np.any(D < R))
        inband = bool(np.any(np.abs(D - R) <= 1e-5 * R))
        c = int(cert["label"][i])
        full = (budget_total and total >= budget_total) or (budget_per_class and 0 <= c < C and
                                                          per.get(c, 0) >= budget_per_class)
        if i in pos:
            assert pos[i] == nxt, "kept rows must be appended in visiting order"
            nxt += 1
            assert not full
            if covered:
                assert inband, f"row {i} kept inside a ball"
                band += 1
            z_k[m] = z
            r_k[m] = cert["radius"][i]
            m += 1
            per[c] = per.get(c, 0) + 1
            total += 1
        else:
            assert covered or full, f"row {i} skipped without cover or budget"
    assert nxt == len(kept)
    return band


def _pool(w, n, seed):
    """n candidates: half mixture draws, half near-duplicates of them (the
    workload's duplicate noise), shuffled, so that balls overlap."""
    base = synth.cache_rows(w)[: n // 2]
    rng = np.random.default_rng(seed)
    dup = base[rng.integers(0, len(base), n - len(base))] + \
        rng.standard_normal((n - len(base), w.d)).astype(np.float32) * np.float32(w.noise)
    pool = np.concatenate([base, dup]).astype(np.float32)
    return pool[rng.permutation(n)]


@pytest.mark.parametrize("name,n,bt,bc", [("tiny", 1024, 0, 0), ("cifar10", 6000, 0, 0), ("cifar10", 6000, 0, 40),
                                          ("cifar100", 5000, 800, 0), ("tinyimagenet", 3000, 0, 3)])
def test_select_workload(dev, name, n, bt, bc):
    w = synth.WORKLOADS[name]
    W, b = synth.head(w)
    rows = _pool(w, n, 7)
    s = oracle.sigma_max(W)
    cert = oracle.certify(W, b, s, rows)
    cache = make_cache(dev, W, b, n + 100)
    # a few existing entries first (they cover part of the pool)
    pre = rows[:50] + np.float32(0.01)
    pidx, _, npre = cache.insert(T(pre, dev))
    pcert = oracle.certify(W, b, s, pre)
    idx, rad, got = cache.insert_select(T(rows, dev), budget_total=bt, budget_per_class=bc)
    idx, rad = idx.cpu().numpy(), rad.cpu().numpy()
    assert got == int((idx >= 0).sum()) and got > 0
    assert got < int(cert["accept"].sum())  # the pool does hold covered candidates
    assert sorted(idx[idx >= 0].tolist()) == list(range(npre, npre + got))
    band = check_selection(rows, cert, idx, rad, pre[pcert["accept"]], pcert["radius"][pcert["accept"]], bt, bc, w.C)
    ref = oracle.select_radius_dedup(rows, cert, pre[pcert["accept"]], pcert["radius"][pcert["accept"]], bt, bc, w.C)
    if band == 0:
        np.testing.assert_array_equal(kept_in_order(idx), ref)
    if bt:
        assert got <= bt
    if bc:
        assert np.bincount(cert["label"][idx >= 0], minlength=w.C).max() <= bc
    # the grown cache answers like the oracle's cache of the same entries
    kept = kept_in_order(idx)
    keys = np.concatenate([pre[pcert["accept"]], rows[kept]])
    radius = np.concatenate([pcert["radius"][pcert["accept"]], cert["radius"][kept]])
    labels = np.concatenate([pcert["label"][pcert["accept"]], cert["label"][kept]])
    Q, _ = synth.queries(w, rows)
    Q = Q[:1000]
    from parity_utils import check_probe
    gi, gl, gd = cache.probe(T(Q, dev))
    check_probe(gi.cpu().numpy(), gl.cpu().numpy(), gd.cpu().numpy(),
                {"keys": keys, "radius": radius, "label": labels}, Q, oracle.probe(keys, radius, labels, Q))
    assert cache.info()["device_errors"] == 0
    cache.close()


def test_select_errors_and_all(dev):
    from paper_2608_13144_gb300._lib import LipCacheError, check
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:200]
    cache = make_cache(dev, W, b, 100)
    with pytest.raises(LipCacheError) as e:
        cache.insert_select(T(rows, dev))  # 200 candidates could exceed 100
    assert e.value.status == 4 and cache.size == 0
    idx, _, n = cache.insert_select(T(rows, dev), budget_total=100)
    assert 0 < n <= 100
    with pytest.raises(LipCacheError) as e:
        check(cache.L.lipcache_insert_select(cache._h, None, 0, None, 0, 9, 0, 0, None, None, None, None))
    assert e.value.status == 1
    with pytest.raises(LipCacheError) as e:
        cache.insert_select(T(rows[:10], dev), strategy="all", budget_total=3)
    assert e.value.status == 1
    cache.set_radius_policy("global", 1.0)
    with pytest.raises(LipCacheError) as e:
        cache.insert_select(T(rows[:10], dev), budget_total=5)
    assert e.value.status == 2
    cache.close()
    # strategy "all" is the plain insert
    c1, c2 = make_cache(dev, W, b, 300), make_cache(dev, W, b, 300)
    i1, r1, n1 = c1.insert(T(rows, dev))
    i2, r2, n2 = c2.insert_select(T(rows, dev), strategy="all")
    assert n1 == n2 and torch.equal(i1, i2) and torch.equal(r1, r2)
    c1.close()
    c2.close()


# ---------------------------------------------------------------- K-center
def test_golden_kcenter(dev):
    g = golden("select_kcenter.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    rows = np.array(g["rows"], np.float32)
    for k, key in ((3, "budget_3"), (1, "budget_1")):
        cache = make_cache(dev, W, b, 16)
        idx, _, n = cache.insert_select(T(rows, dev), strategy="kcenter", budget_per_class=k)
        assert kept_in_order(idx.cpu().numpy()).tolist() == g[key] and n == len(g[key])
        cache.close()
    tie = np.array(g["tie_rows"], np.float32)
    cache = make_cache(dev, W, b, 16)
    idx, _, n = cache.insert_select(T(tie, dev), strategy="kcenter", budget_per_class=2)
    assert kept_in_order(idx.cpu().numpy()).tolist() == g["tie_budget_2"]
    cache.close()


@pytest.mark.parametrize("name,n,k", [("tiny", 1024, 20), ("cifar10", 6000, 50), ("cifar100", 5000, 10),
                                      ("tinyimagenet", 4000, 5)])
def test_kcenter_workload(dev, name, n, k):
    """Per class the GPU's centres are a farthest-point sequence (each at
    least (1 - 1e-5) as far from the earlier centres as any other candidate,
    FP64), the first has the class's largest radius, and the whole selection
    equals the oracle's whenever no step was a near-tie."""
    w = synth.WORKLOADS[name]
    W, b = synth.head(w)
    rows = _pool(w, n, 11)
    cert = oracle.certify(W, b, oracle.sigma_max(W), rows)
    cache = make_cache(dev, W, b, n)
    idx, rad, got = cache.insert_select(T(rows, dev), strategy="kcenter", budget_per_class=k)
    idx = idx.cpu().numpy()
    sel = kept_in_order(idx)
    assert got == len(sel)
    ref = oracle.select_kcenter(rows, cert, k, w.C)
    for c in range(w.C):
        cand = np.nonzero(cert["accept"] & (cert["label"] == c))[0]
        mine = [i for i in sel.tolist() if cert["label"][i] == c]
        assert len(mine) == min(k, len(cand))
        if not mine:
            continue
        assert cert["radius"][mine[0]] >= cert["radius"][cand].max() * (1 - 1e-6)
        Z = rows[cand].astype(np.float64)
        mind = np.full(len(cand), np.inf)
        pos = {r: j for j, r in enumerate(cand.tolist())}
        for t, r in enumerate(mine):
            if t:
                avail = np.ones(len(cand), bool)
                avail[[pos[x] for x in mine[:t]]] = False
                assert mind[pos[r]] >= mind[avail].max() * (1 - 1e-5)
            mind = np.minimum(mind, np.linalg.norm(Z - Z[pos[r]], axis=1))
    # classes come out in ascending order
    labs = cert["label"][sel]
    assert np.all(np.diff(labs) >= 0)
    if len(ref["gaps"]) == 0 or ref["gaps"].min() > 1e-5:
        np.testing.assert_array_equal(sel, ref["selected"])
    # the kept entries carry their certified radii
    gi, _, gd = cache.probe(T(rows[sel], dev))
    assert np.array_equal(gi.cpu().numpy(), idx[sel]) or np.all(gd.cpu().numpy() == 0)
    cache.close()


def test_kcenter_errors(dev):
    from paper_2608_13144_gb300._lib import LipCacheError
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:100]
    cache = make_cache(dev, W, b, 1000)
    for kw in ({}, {"budget_per_class": 0}, {"budget_per_class": 2, "budget_total": 5}):
        with pytest.raises(LipCacheError) as e:
            cache.insert_select(T(rows, dev), strategy="kcenter", **kw)
        assert e.value.status == 1
    small = make_cache(dev, W, b, 15)
    with pytest.raises(LipCacheError) as e:
        small.insert_select(T(rows, dev), strategy="kcenter", budget_per_class=2)  # 10 classes x 2 > 15
    assert e.value.status == 4
    cache.close()
    small.close()
