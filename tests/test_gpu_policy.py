"""Empirical radius policies (Sec. 5.4) through the unchanged probe kernels,
CUDA path vs the FP64 oracle (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from conftest import golden
from parity_utils import check_probe

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


def probe_np(cache, Q, dev, batch=4096):
    outs = [[], [], []]
    for s, e in synth.batches(len(Q), batch):
        o = cache.probe(T(Q[s:e], dev))
        for k in range(3):
            outs[k].append(o[k].cpu().numpy())
    return [np.concatenate(x) for x in outs]


def _golden_cache(dev, path):
    from paper_2608_13144_gb300.lipcache import LipCache
    g = golden("interclass_radius.json")
    # a 3-class head under which every golden key has a positive margin
    W = np.array([[1.0, 0.0], [0.0, 1.0], [-1.0, -1.0]], np.float32)
    b = np.array([0.1, 0.05, 0.0], np.float32)
    keys = np.array(g["keys"], np.float32)
    labels = np.array(g["labels"], np.int32)
    c = LipCache(2, 3, 64, device=dev)
    c.set_head(T(W, dev), T(b, dev))
    c.set_probe_path(path)
    _, _, n = c.insert(T(keys, dev), T(labels, dev))
    assert n == len(keys)
    return g, c, W, b, keys, labels


def _ring_queries(keys, radii, rng, per=40):
    """Queries around each key at 0.2 .. 1.8 times its radius."""
    out = []
    for z, r in zip(keys, radii):
        u = rng.standard_normal((per, keys.shape[1]))
        u /= np.linalg.norm(u, axis=1, keepdims=True)
        out.append(z + u * (max(r, 0.05) * rng.uniform(0.2, 1.8, per))[:, None])
    return np.concatenate(out).astype(np.float32)


@pytest.mark.parametrize("path", PATHS)
def test_golden_interclass_policy(dev, path):
    g, cache, W, b, keys, labels = _golden_cache(dev, path)
    rho = cache.set_radius_policy("interclass", g["beta"])
    np.testing.assert_allclose(rho, g["expect_rho"], rtol=1e-13)
    info = cache.info()
    assert info["radius_policy"] == 2 and info["policy_param"] == g["beta"]
    radius = np.array(g["expect_radius"])
    Q = _ring_queries(keys, radius, np.random.default_rng(1))
    gi, gl, gd = probe_np(cache, Q, dev)
    ref = {"keys": keys, "radius": radius, "label": labels}
    stats = check_probe(gi, gl, gd, ref, Q, oracle.probe(keys, radius, labels, Q))
    assert stats["hits"] > 50
    cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_global_policy_and_back(dev, path):
    g, cache, W, b, keys, labels = _golden_cache(dev, path)
    Q = _ring_queries(keys, np.full(len(keys), 0.8), np.random.default_rng(2))
    rho = cache.set_radius_policy("global", 0.8)
    assert np.all(rho == 0.8)
    gi, gl, gd = probe_np(cache, Q, dev)
    rad = oracle.global_radius(len(keys), 0.8)
    ref = {"keys": keys, "radius": rad, "label": labels}
    check_probe(gi, gl, gd, ref, Q, oracle.probe(keys, rad, labels, Q))
    # back to the certified radii
    assert np.all(cache.set_radius_policy("certified") == 0)
    cert = oracle.certify(W, b, oracle.sigma_max(W), keys, labels)
    gi, gl, gd = probe_np(cache, Q, dev)
    ref = {"keys": keys, "radius": cert["radius"], "label": labels}
    check_probe(gi, gl, gd, ref, Q, oracle.probe(keys, cert["radius"], labels, Q))
    assert cache.info()["radius_policy"] == 0
    cache.close()


def test_policy_rejects_bad_arguments(dev):
    from paper_2608_13144_gb300._lib import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    g, cache, *_ = _golden_cache(dev, "auto")
    for pol, p in [("global", 0.0), ("global", -1.0), ("interclass", float("nan")), ("global", float("inf"))]:
        with pytest.raises(LipCacheError) as e:
            cache.set_radius_policy(pol, p)
        assert e.value.status == 1
    from paper_2608_13144_gb300._lib import check
    with pytest.raises(LipCacheError) as e:
        check(cache.L.lipcache_set_radius_policy(cache._h, 7, 1.0, None, None))  # unknown policy
    assert e.value.status == 1
    cache.close()
    c2 = LipCache(2, 3, 8, device=dev)
    with pytest.raises(LipCacheError) as e:
        c2.set_radius_policy("global", 1.0)
    assert e.value.status == 2  # no head yet
    c2.close()


@pytest.mark.parametrize("name,path", [("cifar10", "tensor"), ("cifar100", "exact"), ("tinyimagenet", "tensor")])
def test_policies_workload(dev, name, path):
    """Both empirical boundaries against the oracle on a workload, plus the
    comparison of Sec. 5.4 in shape: the certified radius keeps every hit
    consistent; the empirical boundaries reuse more and give some of it up."""
    from scipy.spatial import cKDTree
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS[name]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:3000]
    Q, _ = synth.queries(w, rows)
    Q = Q[:1000]
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    keys, labels, yG = ref["keys"], ref["label"], ref["yG"]
    cache = LipCache(w.d, w.C, len(rows), device=dev)
    cache.set_head(T(W, dev), T(b, dev))
    cache.set_probe_path(path)
    cache.insert(T(rows, dev))
    dist, _ = cKDTree(keys.astype(np.float64)).query(Q.astype(np.float64))
    tau = float(np.median(dist))
    summary = {}
    for pol, param in [("certified", 0.0), ("global", tau), ("interclass", 1.0)]:
        rho = cache.set_radius_policy(pol, param)
        if pol == "certified":
            rad = ref["radius"]
        elif pol == "global":
            rad = oracle.global_radius(len(keys), tau)
        else:
            o = oracle.interclass_radius(keys, labels, w.C, 1.0)
            rad = o["radius"]
            np.testing.assert_allclose(rho, o["rho"], rtol=1e-10)
        gi, gl, gd = probe_np(cache, Q, dev, w.batch)
        r = {"keys": keys, "radius": rad, "label": labels}
        check_probe(gi, gl, gd, r, Q, oracle.probe(keys, rad, labels, Q))
        _, nh, nc = cache.consistency(T(Q, dev), T(gi, dev))
        summary[pol] = (nh, nc)
    nh, nc = summary["certified"]
    assert nc == nh
    if name == "cifar10":
        for pol in ("global", "interclass"):
            assert summary[pol][0] > nh and summary[pol][1] < summary[pol][0], summary
    cache.close()


def test_policy_applies_to_later_inserts(dev):
    """Entries inserted (or written back) after a policy is set get its
    radius: tau under GLOBAL, rho of their label from the snapshot under
    INTERCLASS."""
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS["cifar10"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:2000]
    Q, _ = synth.queries(w, rows)
    Q = Q[:600]
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    for pol, param in [("global", 1.5), ("interclass", 0.7)]:
        cache = LipCache(w.d, w.C, 4000, device=dev)
        cache.set_head(T(W, dev), T(b, dev))
        cache.insert(T(rows[:1000], dev))
        rho = cache.set_radius_policy(pol, param)
        cache.insert(T(rows[1000:1500], dev))
        _, _, _, ins, n = cache.probe_writeback(T(rows[1500:], dev))
        ins = ins.cpu().numpy()
        first = ref["index"][:1500]
        keys = np.concatenate([rows[:1500][first >= 0], rows[1500:][ins >= 0]])
        labels = np.concatenate([ref["label"][:int((first >= 0).sum())],
                                 oracle.certify(W, b, oracle.sigma_max(W), rows[1500:])["label"][ins >= 0]])
        assert cache.size == len(keys)
        if pol == "global":
            rad = oracle.global_radius(len(keys), param)
        else:
            snap = oracle.interclass_radius(rows[:1000][ref["index"][:1000] >= 0],
                                            ref["label"][:int((ref["index"][:1000] >= 0).sum())], w.C, param)
            np.testing.assert_allclose(rho, snap["rho"], rtol=1e-10)
            rad = snap["rho"][labels]
        gi, gl, gd = probe_np(cache, Q, dev)
        r = {"keys": keys, "radius": rad, "label": labels}
        check_probe(gi, gl, gd, r, Q, oracle.probe(keys, rad, labels, Q))
        cache.close()
