"""Write-back (Algorithm 2's miss branch) and the certified-consistency check,
CUDA path vs the FP64 oracle through the C ABI (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from conftest import golden
from parity_utils import RTOL, check_insert, check_probe, radius_tol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

PATHS = ["exact", "tensor"]


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def T(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def make_cache(dev, W, b, capacity, path="auto", mode="conservative"):
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], capacity, mode, device=dev)
    sigma = c.set_head(T(W, dev), T(b, dev))
    c.set_probe_path(path)
    return c, sigma


def np_(*ts):
    return [t.cpu().numpy() for t in ts]


# ---------------------------------------------------------------- write-back
@pytest.mark.parametrize("path", PATHS)
def test_golden_writeback(dev, path):
    g = golden("writeback_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    Q = np.array(g["queries"], np.float32)
    cache, _ = make_cache(dev, W, b, 16, path)
    cache.insert(T(np.array(g["rows"], np.float32), dev))
    gi, gl, gd, ins, n = cache.probe_writeback(T(Q, dev))
    gi, gl, ins = np_(gi, gl, ins)
    assert gi.tolist() == g["expect_index"]
    assert ins.tolist() == g["expect_inserted"]
    assert n == 3 and cache.size == 4
    # each written-back query now hits itself (distance 0) with its proxy label
    qi, ql, qd = np_(*cache.probe(T(Q[ins >= 0], dev)))
    assert qi.tolist() == ins[ins >= 0].tolist()
    assert ql.tolist() == g["expect_yG"][1:] and np.all(qd == 0)
    # the new radii: probes 0.1% inside / outside r, in a direction where the
    # entry is the nearest hit (entry 1 down, entries 2 and 3 up)
    for k, r, up in zip(ins[ins >= 0], g["expect_radius"][1:], (-1.0, 1.0, 1.0)):
        z = Q[np.nonzero(ins == k)[0][0]]
        inside = (z + np.array([0.0, up * r * 0.999], np.float32))[None]
        outside = (z + np.array([0.0, up * r * 1.001], np.float32))[None]
        ri, _, _ = np_(*cache.probe(T(inside, dev)))
        ro, _, _ = np_(*cache.probe(T(outside, dev)))
        assert ri[0] == k and ro[0] != k
    cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_golden_writeback_require_consistency(dev, path):
    g = golden("writeback_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    Q = np.array(g["queries"], np.float32)
    cache, _ = make_cache(dev, W, b, 16, path)
    cache.insert(T(np.array(g["rows"], np.float32), dev))
    _, _, _, ins, n = cache.probe_writeback(T(Q, dev), T(np.array(g["payload"], np.int32), dev), True)
    assert ins.cpu().numpy().tolist() == g["expect_inserted_consistent"]
    assert n == 2
    _, ql, _ = np_(*cache.probe(T(Q[ins.cpu().numpy() >= 0], dev)))
    assert ql.tolist() == g["expect_label_consistent"][1:]
    cache.close()


def test_writeback_full_is_all_or_nothing(dev):
    from paper_2608_13144_gb300._lib import LipCacheError
    g = golden("writeback_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache, _ = make_cache(dev, W, b, 6)
    cache.insert(T(np.array(g["rows"], np.float32), dev))
    with pytest.raises(LipCacheError) as e:
        cache.probe_writeback(T(np.array(g["queries"], np.float32), dev))  # 1 + 6 > 6
    assert e.value.status == 4 and cache.size == 1
    cache.close()


def _workload(name, n_rows, n_q):
    w = synth.WORKLOADS[name]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:n_rows]
    Q, _ = synth.queries(w, rows)
    return w, W, b, rows, Q[:n_q]


@pytest.mark.parametrize("name,path", [("tiny", "exact"), ("cifar10", "tensor"), ("cifar100", "tensor"),
                                       ("cifar100", "exact")])
def test_writeback_workload(dev, name, path):
    """Batches of the workload's size, each probed and written back; the
    probe must match the oracle outside the 1e-5 band, and the set written
    back must be exactly the GPU's misses that Algorithm 1 accepts, appended
    in query order. A final probe of every query against the grown cache
    matches the oracle's probe of the same grown cache."""
    w, W, b, rows, Q = _workload(name, 3000 if name != "tiny" else 1024, 2000 if name != "tiny" else 256)
    sigma = oracle.sigma_max(W)
    ref = oracle.build_cache(W, b, sigma, rows)
    cache, _ = make_cache(dev, W, b, len(rows) + len(Q), path)
    gidx, grad, nacc = cache.insert(T(rows, dev))
    check_insert(gidx.cpu().numpy(), grad.cpu().numpy(), nacc, ref, (W, b, rows, 1.0))
    cur = {k: ref[k] for k in ("keys", "radius", "label", "yG")}
    total_ins = 0
    for s, e in synth.batches(len(Q), w.batch):
        q = Q[s:e]
        gi, gl, gd, ins, n = cache.probe_writeback(T(q, dev))
        gi, gl, gd, ins = np_(gi, gl, gd, ins)
        orc = oracle.probe(cur["keys"], cur["radius"], cur["label"], q)
        check_probe(gi, gl, gd, cur, q, orc)
        cert = oracle.certify(W, b, sigma, q)
        add = (gi < 0) & cert["accept"]
        n0 = len(cur["keys"])
        exp = np.full(len(q), -1, np.int64)
        exp[add] = n0 + np.arange(int(add.sum()))
        assert np.array_equal(ins, exp), f"{(ins != exp).sum()} write-back indices differ"
        assert n == int(add.sum())
        total_ins += n
        cur = {"keys": np.concatenate([cur["keys"], q[add]]), "radius": np.concatenate([cur["radius"],
               cert["radius"][add]]), "label": np.concatenate([cur["label"], cert["label"][add]]),
               "yG": np.concatenate([cur["yG"], cert["yG"][add]])}
    assert total_ins > 0 and cache.size == len(cur["keys"])
    gi, gl, gd = np_(*cache.probe(T(Q, dev)))
    orc = oracle.probe(cur["keys"], cur["radius"], cur["label"], Q)
    check_probe(gi, gl, gd, cur, Q, orc)
    assert cache.info()["device_errors"] == 0
    cache.close()


@pytest.mark.parametrize("name,path", [("tiny", "exact"), ("cifar100", "tensor"), ("tinyimagenet", "tensor")])
def test_writeback_tight_radius(dev, name, path):
    """Write-back with the tight radius (Eq. 29): the misses Algorithm 1
    accepts are certified on the same kernels as an insert, so the set
    written back is exactly the oracle's, in query order, and each new radius
    is within 1e-5 relative of the FP64 one (rows at FP64's own resolution
    get its slack). The grown cache then probes like the oracle's
    outside the 1e-5 band."""
    w, W, b, rows, Q = _workload(name, 2000, 1500)
    sigma = oracle.sigma_max(W)
    ref = oracle.build_cache(W, b, sigma, rows, radius_mode=oracle.RADIUS_TIGHT)
    cache, _ = make_cache(dev, W, b, len(rows) + len(Q), path, "tight")
    gidx, grad, nacc = cache.insert(T(rows, dev))
    check_insert(gidx.cpu().numpy(), grad.cpu().numpy(), nacc, ref, ("tight", W, b, rows, 1.0))
    cur = {k: ref[k] for k in ("keys", "radius", "label", "yG")}
    n_base = len(cur["keys"])
    for s, e in synth.batches(len(Q), w.batch):
        q = Q[s:e]
        gi, gl, gd, ins, n = cache.probe_writeback(T(q, dev))
        gi, gl, gd, ins = np_(gi, gl, gd, ins)
        res = oracle.probe_writeback(cur, W, b, sigma, q, radius_mode=oracle.RADIUS_TIGHT)
        check_probe(gi, gl, gd, cur, q, res["probe"])
        # the oracle's write-back set follows its own probe; the GPU's follows
        # the GPU probe, which agrees outside the band (checked above)
        add = (gi < 0) & res["cert"]["accept"]
        exp = np.full(len(q), -1, np.int64)
        exp[add] = len(cur["keys"]) + np.arange(int(add.sum()))
        assert np.array_equal(ins, exp), f"{(ins != exp).sum()} write-back indices differ"
        assert n == int(add.sum())
        cert = res["cert"]
        cur = {"keys": np.concatenate([cur["keys"], q[add]]), "radius": np.concatenate([cur["radius"],
               cert["radius"][add]]), "label": np.concatenate([cur["label"], cert["label"][add]]),
               "yG": np.concatenate([cur["yG"], cert["yG"][add]])}
    assert cache.size == len(cur["keys"]) > n_base
    ent = cache.entries(n_base)
    r = cur["radius"][n_base:]
    assert np.array_equal(ent["keys"], cur["keys"][n_base:])
    assert np.array_equal(ent["label"], cur["label"][n_base:]) and np.array_equal(ent["yG"], cur["yG"][n_base:])
    g_r = ent["radius"].astype(np.float64)
    np.testing.assert_allclose(g_r, r, rtol=RTOL)
    assert np.all(np.abs(g_r - r) <= radius_tol(W, b, cur["keys"][n_base:], r, 1.0, tight=True))
    gi, gl, gd = np_(*cache.probe(T(Q, dev)))
    orc = oracle.probe(cur["keys"], cur["radius"], cur["label"], Q)
    check_probe(gi, gl, gd, cur, Q, orc)
    assert cache.info()["device_errors"] == 0
    cache.close()


# ---------------------------------------------------------------- consistency
def test_golden_consistency(dev):
    g = golden("consistency_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache, _ = make_cache(dev, W, b, 4)
    cache.insert(T(np.array(g["keys"], np.float32), dev))
    Q = T(np.array(g["queries"], np.float32), dev)
    for which in ("inflated", "certified"):
        hit = T(np.array(g["expect_hit_" + which], np.int64), dev)
        out, nh, nc = cache.consistency(Q, hit)
        exp = np.array(g["expect_consistent_" + which])
        assert out.cpu().numpy().tolist() == exp.tolist()
        assert nh == int((exp >= 0).sum()) and nc == int((exp == 1).sum())
    # the certified radius, through the probe itself
    gi, _, _ = cache.probe(Q)
    assert gi.cpu().numpy().tolist() == g["expect_hit_certified"]
    cache.close()


def test_consistency_rejects_bad_index(dev):
    from paper_2608_13144_gb300._lib import LipCacheError
    g = golden("consistency_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache, _ = make_cache(dev, W, b, 4)
    cache.insert(T(np.array(g["keys"], np.float32), dev))
    Q = T(np.array(g["queries"][:3], np.float32), dev)
    with pytest.raises(LipCacheError) as e:
        cache.consistency(Q, T(np.array([0, 1, -2], np.int64), dev))  # size is 1
    assert e.value.status == 1
    cache.close()


@pytest.mark.parametrize("name", ["tiny", "cifar10", "cifar100", "tinyimagenet"])
def test_consistency_workload(dev, name):
    """Probe hits with certified radii are all consistent (the Lemma); with
    arbitrary entries in place of the hits the check agrees with the
    oracle's FP64 argmax wherever the top-two logit gap exceeds 1e-6 of the
    logit scale."""
    w, W, b, rows, Q = _workload(name, 2000, 1024)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    cache, _ = make_cache(dev, W, b, len(rows))
    cache.insert(T(rows, dev))
    gi, _, _ = cache.probe(T(Q, dev))
    out, nh, nc = cache.consistency(T(Q, dev), gi)
    gi, out = gi.cpu().numpy(), out.cpu().numpy()
    assert nh == int((gi >= 0).sum()) and nc == nh
    if name in ("tiny", "cifar10"):
        assert nh > 50
    assert np.all(out[gi < 0] == -1) and np.all(out[gi >= 0] == 1)

    rng = np.random.default_rng(5)
    fake = rng.integers(-1, len(ref["keys"]), len(Q)).astype(np.int64)
    out, nh, nc = cache.consistency(T(Q, dev), T(fake, dev))
    out = out.cpu().numpy()
    orc = oracle.consistency(W, b, Q, fake, ref["yG"])
    s = Q.astype(np.float64) @ W.astype(np.float64).T + b
    scale = np.abs(s).max(axis=1)
    clear = orc["gap"] > 1e-6 * scale
    np.testing.assert_array_equal(out[clear], orc["consistent"][clear])
    assert nh == orc["n_hits"]
    assert abs(nc - orc["n_consistent"]) <= int((~clear).sum())
    cache.close()


def test_read_entries_roundtrip(dev):
    """Entries read back equal the accepted rows, their radii and labels; a
    cache rebuilt from them (keys + labels as payload) answers identically."""
    w = synth.WORKLOADS["cifar10"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:3000]
    Q, _ = synth.queries(w, rows)
    Q = Q[:1000]
    payload = (np.arange(len(rows)) % 7).astype(np.int32)
    cache, _ = make_cache(dev, W, b, 4000)
    idx, rad, n = cache.insert(T(rows, dev), T(payload, dev))
    idx, rad = idx.cpu().numpy(), rad.cpu().numpy()
    e = cache.entries()
    acc = idx >= 0
    np.testing.assert_array_equal(e["keys"], rows[acc])
    np.testing.assert_array_equal(e["radius"], rad[acc])
    np.testing.assert_array_equal(e["label"], payload[acc])
    ref = oracle.certify(W, b, oracle.sigma_max(W), rows)
    np.testing.assert_array_equal(e["yG"], ref["yG"][acc])
    part = cache.entries(10, 5)
    np.testing.assert_array_equal(part["keys"], e["keys"][10:15])
    from paper_2608_13144_gb300._lib import LipCacheError
    with pytest.raises(LipCacheError):
        cache.entries(n - 2, 5)
    again, _ = make_cache(dev, W, b, 4000)
    again.insert(T(e["keys"], dev), T(e["label"], dev))
    a = [t.cpu().numpy() for t in cache.probe(T(Q, dev))]
    c = [t.cpu().numpy() for t in again.probe(T(Q, dev))]
    for x, y in zip(a, c):
        np.testing.assert_array_equal(x, y)
    cache.close()
    again.close()


@pytest.mark.parametrize("mode,policy", [("conservative", "certified"), ("tight", "interclass")])
def test_checkpoint_roundtrip(dev, tmp_path, mode, policy):
    """save / load: the restored cache has the same head, entries (keys,
    radii re-certified to the same bits, labels, y^G), probe path and radius
    policy, and answers every probe identically."""
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS["cifar10"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:5000]
    Q, _ = synth.queries(w, rows)
    Q = Q[:1500]
    cache = LipCache(w.d, w.C, 6000, mode, device=dev)
    cache.set_radius_scale(0.9)
    cache.set_head(T(W, dev), T(b, dev))
    cache.insert(T(rows, dev), T((np.arange(len(rows)) % 3).astype(np.int32), dev))
    cache.set_probe_path("exact")
    if policy != "certified":
        cache.set_radius_policy(policy, 0.8)
    path = str(tmp_path / "cache.npz")
    cache.save(path)
    again = LipCache.load(path, device=dev)
    a, c = cache.info(), again.info()
    for k in ("d", "C", "capacity", "size", "radius_mode", "radius_scale", "sigma", "probe_path", "radius_policy",
              "policy_param"):
        assert a[k] == c[k], k
    Wa, ba = again.head()
    np.testing.assert_array_equal(Wa, W)
    np.testing.assert_array_equal(ba, b)
    ea, ec = cache.entries(), again.entries()
    for k in ("keys", "radius", "label", "yG"):
        np.testing.assert_array_equal(ea[k], ec[k])
    for x, y in zip(cache.probe(T(Q, dev)), again.probe(T(Q, dev))):
        np.testing.assert_array_equal(x.cpu().numpy(), y.cpu().numpy())
    cache.close()
    again.close()
