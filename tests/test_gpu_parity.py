"""CUDA path vs the FP64 oracle, through the C ABI (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from conftest import golden
from parity_utils import check_insert, check_probe, record_parity

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

PATHS = ["exact", "tensor", "tensor_single", "tensor_pair"]


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def T(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def make_cache(dev, W, b, capacity, mode="conservative", kappa=None):
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], capacity, mode, device=dev)
    if kappa is not None:
        c.set_radius_scale(kappa)
    sigma = c.set_head(T(W, dev), T(b, dev))
    return c, sigma


def run_probe(cache, Q, dev, batch, path):
    cache.set_probe_path(path)
    outs = [[], [], []]
    for s, e in synth.batches(len(Q), batch):
        o = cache.probe(T(Q[s:e], dev))
        for k in range(3):
            outs[k].append(o[k].cpu().numpy())
    info = cache.info()
    assert info["device_errors"] == 0 and info["last_probe_path"] in {"exact": (2,), "tensor": (3, 4), "tensor_single": (3,), "tensor_pair": (4,)}[path]
    return [np.concatenate(x) if x else np.zeros(0) for x in outs]


# ---------------------------------------------------------------- spectral norm
def _heads():
    rng = np.random.default_rng(11)
    hs = []
    for C, d in [(10, 16), (10, 64), (100, 128), (200, 256), (3, 3), (2, 2), (40, 12), (2, 100), (7, 33)]:
        hs.append(((C, d), (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)))
    Qm, _ = np.linalg.qr(rng.standard_normal((16, 16)))
    hs.append(("orthogonal", (3.0 * Qm).astype(np.float32)))  # all singular values equal
    hs.append(("rank1", np.outer(rng.standard_normal(12), rng.standard_normal(20)).astype(np.float32)))
    hs.append(("close_top", np.diag([1.0, 1.0 - 1e-7, 0.5, 0.2]).astype(np.float32)))
    for name in ("tinyimagenet", "scale", "cifar100"):
        hs.append((name, synth.head(synth.WORKLOADS[name])[0]))
    return hs


@pytest.mark.parametrize("name,W", _heads(), ids=lambda x: str(x) if not isinstance(x, np.ndarray) else "")
def test_sigma_vs_oracle_svd(dev, name, W):
    b = np.zeros(W.shape[0], np.float32)
    cache, sigma = make_cache(dev, W, b, 8)
    ref = oracle.sigma_max(W)
    assert abs(sigma - ref) <= 1e-10 * ref, (sigma, ref)
    info = cache.info()
    assert info["sigma_residual"] <= 1e-10
    cache.close()


def test_degenerate_head(dev):
    from paper_2608_13144_gb300 import LipCacheError
    W = np.array(golden("certify_skip_rules.json")["degenerate"]["W"], np.float32)
    with pytest.raises(LipCacheError) as e:
        make_cache(dev, W, np.zeros(2, np.float32), 4)
    assert e.value.status == 3


def test_not_converged(dev):
    from paper_2608_13144_gb300 import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    W, b = synth.head(synth.WORKLOADS["cifar100"])
    c = LipCache(W.shape[1], W.shape[0], 4, device=dev)
    c.set_spectral_options(0, 1)
    with pytest.raises(LipCacheError) as e:
        c.set_head(T(W, dev), T(b, dev))
    assert e.value.status == 5
    with pytest.raises(LipCacheError) as e:  # no head installed -> insert refused
        c.insert(T(np.zeros((1, W.shape[1]), np.float32), dev))
    assert e.value.status == 2
    c.set_spectral_options(40, 1000)
    c.set_head(T(W, dev), T(b, dev))
    c.close()


# ---------------------------------------------------------------- golden cases
@pytest.mark.parametrize("path", PATHS)
def test_golden_two_class(dev, path):
    g = golden("radius_two_class.json")
    W, b = np.array(g["W"], np.float32), np.array(g["b"], np.float32)
    cache, sigma = make_cache(dev, W, b, 4)
    assert sigma == pytest.approx(g["sigma"], rel=1e-14)
    idx, rad, n = cache.insert(T(np.array(g["rows"], np.float32), dev))
    assert n == 1 and rad.cpu().numpy()[0] == pytest.approx(g["radius"][0], rel=1e-7)
    gi, gl, gd = run_probe(cache, np.array(g["queries"], np.float32), dev, 8, path)
    exp = np.array(g["expect_index"])
    # (3, 1e-6) sits 1e-6 inside r = 1: outside the 1e-5 band only in the
    # oracle's FP64 sense, so the GPU's conservative threshold may miss it.
    assert list(gi[:5]) == list(exp[:5])
    assert gi[5] in (0, -1)
    cache.close()


@pytest.mark.parametrize("mode", ["conservative", "tight"])
def test_golden_three_class(dev, mode):
    for case in golden("radius_three_class.json")["cases"]:
        W, b = np.array(case["W"], np.float32), np.array(case["b"], np.float32)
        cache, sigma = make_cache(dev, W, b, 4, mode)
        assert sigma == pytest.approx(case["sigma"], rel=1e-14)
        _, rad, n = cache.insert(T(np.array([case["z"]], np.float32), dev))
        exp = case["radius"] if mode == "conservative" else case["radius_tight"]
        assert n == 1 and rad.cpu().numpy()[0] == pytest.approx(exp, rel=1e-7)
        cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_golden_probe_selection(dev, path):
    """Hand-built strict-inequality and lowest-index cases of Eqs. 13-14,
    with radii produced by a 2-class antisymmetric head (r = distance to the
    hyperplane x_1 = c)."""
    # keys on the x axis; head W = [[1,0],[-1,0]], b = [-c, c] gives
    # s_0 - s_1 = 2(x - c), sigma = sqrt 2, r = |x - c| (Eq. 21).
    keys = np.array([[0.0, 0.0], [0.0, 0.0], [1.0, 0.0], [0.25, 0.0]], np.float32)
    W = np.array([[1.0, 0.0], [-1.0, 0.0]], np.float32)
    b = np.array([0.5, -0.5], np.float32)  # boundary at x = -0.5: r = x + 0.5
    cache, _ = make_cache(dev, W, b, 8)
    idx, rad, n = cache.insert(T(keys, dev))
    assert n == 4
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), keys)
    Q = np.array([[0.125, 0.0], [0.75, 0.0], [5.0, 5.0], [0.25, 0.0625], [0.0, 0.25]], np.float32)
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
    gi, gl, gd = run_probe(cache, Q, dev, 8, path)
    check_probe(gi, gl, gd, ref, Q, orc)
    assert gi[0] == 0  # keys 0 and 1 are identical: lowest index wins
    cache.close()


def test_skip_rules(dev):
    g = golden("certify_skip_rules.json")
    t = g["tie"]
    W, b = np.array(t["W"], np.float32), np.array(t["b"], np.float32)
    cache, _ = make_cache(dev, W, b, 8)
    idx, rad, n = cache.insert(T(np.array(t["rows"], np.float32), dev))
    assert n == 0 and list(idx.cpu().numpy()) == [-1, -1]
    cache.close()
    k = g["consistency"]
    W, b = np.array(k["W"], np.float32), np.array(k["b"], np.float32)
    rows = T(np.array(k["rows"], np.float32), dev)
    pl = T(np.array(k["payload"], np.int32), dev)
    for req, exp in ((True, k["accept_required"]), (False, k["accept_free"])):
        cache, _ = make_cache(dev, W, b, 8)
        idx, _, n = cache.insert(rows, payload=pl, require_consistency=req)
        assert list((idx.cpu().numpy() >= 0).astype(int)) == exp
        gi, gl, _ = cache.probe(rows)
        acc = np.nonzero(exp)[0]
        assert list(gl.cpu().numpy()[acc]) == [k["label"][i] for i in acc]  # payload passes through
        cache.close()


# ---------------------------------------------------------------- workloads
WORKLOADS = ["tiny", "cifar10", "cifar100", "tinyimagenet"]


@pytest.fixture(scope="module")
def built(dev):
    """GPU cache + oracle cache per workload, built once."""
    store = {}

    def get(name, mode="conservative"):
        key = (name, mode)
        if key not in store:
            w = synth.WORKLOADS[name]
            W, b = synth.head(w)
            rows = synth.cache_rows(w)
            Q, _ = synth.queries(w, rows)
            cache, sigma = make_cache(dev, W, b, w.N, mode)
            parts = [cache.insert(T(rows[s:e], dev)) for s, e in synth.batches(w.N, w.insert_batch)]
            g_index = np.concatenate([p[0].cpu().numpy() for p in parts])
            g_index_local = g_index.copy()
            g_radius = np.concatenate([p[1].cpu().numpy() for p in parts])
            n_acc = sum(p[2] for p in parts)
            s_ref = oracle.sigma_max(W)
            ref = oracle.build_cache(W, b, s_ref, rows,
                                     radius_mode=oracle.RADIUS_TIGHT if mode == "tight" else oracle.RADIUS_CONSERVATIVE)
            orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
            store[key] = dict(w=w, W=W, b=b, rows=rows, Q=Q, cache=cache, sigma=sigma, s_ref=s_ref,
                              g_index=g_index_local, g_radius=g_radius, n_acc=n_acc, ref=ref, orc=orc)
        return store[key]

    yield get
    for v in store.values():
        v["cache"].close()


@pytest.mark.parametrize("name", WORKLOADS)
def test_insert_parity(built, name):
    s = built(name)
    assert abs(s["sigma"] - s["s_ref"]) <= 1e-10 * s["s_ref"]
    check_insert(s["g_index"], s["g_radius"], s["n_acc"], s["ref"], (s["W"], s["b"], s["rows"], 1.0))


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("name", WORKLOADS)
def test_probe_parity(built, dev, name, path):
    s = built(name)
    gi, gl, gd = run_probe(s["cache"], s["Q"], dev, s["w"].batch, path)
    stats = check_probe(gi, gl, gd, s["ref"], s["Q"], s["orc"])
    record_parity(name, path, stats)
    print(name, path, stats)


@pytest.mark.parametrize("name", WORKLOADS)
def test_tensor_equals_exact(built, dev, name):
    """Both probe kernels evaluate the same canonical FP32 distance for every
    pair they accept, so their outputs agree bit for bit; a screen that
    dropped an accepted pair would show up here."""
    s = built(name)
    a = run_probe(s["cache"], s["Q"], dev, s["w"].batch, "exact")
    for path in ("tensor", "tensor_single", "tensor_pair"):
        b = run_probe(s["cache"], s["Q"], dev, s["w"].batch, path)
        for x, y in zip(a, b):
            assert np.array_equal(x.view(np.uint8) if x.dtype == np.float32 else x,
                                  y.view(np.uint8) if y.dtype == np.float32 else y), path


@pytest.mark.parametrize("name", ["tiny", "cifar100"])
def test_tight_radius_parity(built, dev, name):
    s = built(name, "tight")
    check_insert(s["g_index"], s["g_radius"], s["n_acc"], s["ref"], ("tight", s["W"], s["b"], s["rows"], 1.0))
    for path in PATHS:
        gi, gl, gd = run_probe(s["cache"], s["Q"], dev, s["w"].batch, path)
        check_probe(gi, gl, gd, s["ref"], s["Q"], s["orc"])


def test_radius_scale(dev):
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    cache, sigma = make_cache(dev, W, b, w.N, kappa=0.5)
    idx, rad, n = cache.insert(T(rows, dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, scale=0.5)
    check_insert(idx.cpu().numpy(), rad.cpu().numpy(), n, ref, (W, b, rows, 0.5))
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
    for path in PATHS:
        gi, gl, gd = run_probe(cache, Q, dev, w.batch, path)
        check_probe(gi, gl, gd, ref, Q, orc)
    cache.close()


# ---------------------------------------------------------------- edge cases
@pytest.mark.parametrize("path", PATHS)
def test_empty_and_zero_sizes(dev, path):
    from paper_2608_13144_gb300 import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    c = LipCache(w.d, w.C, 10, device=dev)
    with pytest.raises(LipCacheError) as e:
        c.probe(T(np.zeros((2, w.d), np.float32), dev))
    assert e.value.status == 2  # before set_head
    c.set_head(T(W, dev), T(b, dev))
    c.set_probe_path(path)
    gi, gl, gd = c.probe(T(np.ones((3, w.d), np.float32), dev))  # empty cache: all misses
    assert list(gi.cpu().numpy()) == [-1, -1, -1] and list(gl.cpu().numpy()) == [-1, -1, -1]
    assert np.all(np.isinf(gd.cpu().numpy()))
    gi, _, _ = c.probe(T(np.zeros((0, w.d), np.float32), dev))
    assert gi.numel() == 0
    _, _, n = c.insert(T(np.zeros((0, w.d), np.float32), dev))
    assert n == 0 and c.size == 0
    rows = synth.cache_rows(w)[:12]
    with pytest.raises(LipCacheError) as e:  # 12 > capacity 10: nothing inserted
        c.insert(T(rows, dev))
    assert e.value.status == 4 and c.size == 0
    idx, _, n = c.insert(T(rows[:10], dev))
    assert c.size == n
    with pytest.raises(LipCacheError) as e:
        c.set_head(T(W, dev), T(b, dev))
    assert e.value.status == 2
    c.close()


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("d,C,N,B", [(20, 5, 300, 77), (33, 3, 1000, 130), (1, 2, 50, 10), (256, 7, 513, 129),
                                     (96, 12, 2049, 300), (64, 300, 700, 100), (160, 40, 900, 260)])
def test_ragged_shapes(dev, path, d, C, N, B):
    w = synth.WORKLOADS["tiny"].scaled(d=d, C=C, components=C, N=N, n_queries=B, sphere_radius=3.0)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    cache, sigma = make_cache(dev, W, b, N + 5)
    idx, rad, n = cache.insert(T(rows, dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(idx.cpu().numpy(), rad.cpu().numpy(), n, ref, (W, b, rows, 1.0))
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
    gi, gl, gd = run_probe(cache, Q, dev, 64, path)
    check_probe(gi, gl, gd, ref, Q, orc)
    cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_duplicate_keys_lowest_index(dev, path):
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:40]
    dup = np.concatenate([rows, rows, rows])  # every key three times
    cache, _ = make_cache(dev, W, b, len(dup))
    idx, _, n = cache.insert(T(dup, dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), dup)
    Q = rows + np.float32(1e-3)
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
    gi, gl, gd = run_probe(cache, Q, dev, 64, path)
    check_probe(gi, gl, gd, ref, Q, orc)
    hit = gi >= 0
    assert np.all(gi[hit] < 40)  # the first copy always wins
    cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_probe_host_matches_device(dev, path):
    w = synth.WORKLOADS["cifar10"].scaled(N=5000, n_queries=700)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    cache, _ = make_cache(dev, W, b, w.N)
    cache.insert(T(rows, dev))
    cache.set_probe_path(path)
    a = [t.cpu().numpy() for t in cache.probe(T(Q, dev))]
    hq = torch.from_numpy(Q).pin_memory()
    b2 = [t.numpy() for t in cache.probe_host(hq)]
    for x, y in zip(a, b2):
        assert np.array_equal(x, y)
    cache.close()


@pytest.mark.parametrize("mode", ["conservative", "tight"])
def test_many_tied_runners_up(dev, mode):
    """19 identical head rows: every row has at least 19 classes whose FP32
    intervals overlap (more than the insert kernel's per-row candidate
    slots), so the whole-warp fallback decides them. Rows whose best class
    is unique keep an exact margin; rows won by the tied group are skipped
    (m = 0) on both sides."""
    rng = np.random.default_rng(21)
    d, C = 32, 24
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    W[1:20] = W[1]
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    b[1:20] = b[1]
    rows = np.concatenate([3 * W[0] + 0.3 * rng.standard_normal((150, d)),
                           3 * W[1] + 0.3 * rng.standard_normal((150, d)),
                           rng.standard_normal((100, d))]).astype(np.float32)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=int(mode == "tight"))
    cache, _ = make_cache(dev, W, b, len(rows), mode)
    idx, rad, n = cache.insert(T(rows, dev))
    check_insert(idx.cpu().numpy(), rad.cpu().numpy(), n, ref,
                 ("tight", W, b, rows, 1.0) if mode == "tight" else (W, b, rows, 1.0))
    assert n > 100
    if mode == "conservative":
        assert n < len(rows)  # rows won by the tied group are skipped
    # (the tight radius skips classes with W_j = W_y, Eq. 29, so it keeps them)
    cache.close()


def test_large_dim_exact_path(dev):
    """d = 1024 (the largest supported): the streaming certify kernel and the
    exact probe; the tensor paths refuse d > 256."""
    from paper_2608_13144_gb300._lib import LipCacheError
    w = synth.WORKLOADS["tiny"].scaled(d=1024, C=12, components=12, N=600, n_queries=150, sphere_radius=6.0)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    cache, sigma = make_cache(dev, W, b, w.N)
    idx, rad, n = cache.insert(T(rows, dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(idx.cpu().numpy(), rad.cpu().numpy(), n, ref, (W, b, rows, 1.0))
    with pytest.raises(LipCacheError):
        cache.set_probe_path("tensor")
    gi, gl, gd = run_probe(cache, Q, dev, 64, "exact")
    check_probe(gi, gl, gd, ref, Q, oracle.probe(ref["keys"], ref["radius"], ref["label"], Q))
    cache.close()


def test_auto_path_choice(dev):
    """"auto" takes the exact kernel below 2^24 multiply-adds per batch (its
    fixed cost is smaller) and the tensor kernel above; both give the same
    bits."""
    for name, N, B, expect in [("tiny", 1024, 256, 2), ("cifar10", 5000, 256, 3)]:
        w = synth.WORKLOADS[name].scaled(N=N, n_queries=B)
        W, b = synth.head(w)
        rows = synth.cache_rows(w)
        Q, _ = synth.queries(w, rows)
        cache, _ = make_cache(dev, W, b, N)
        cache.insert(T(rows, dev))
        cache.set_probe_path("auto")
        a = [t.cpu().numpy() for t in cache.probe(T(Q, dev))]
        assert cache.info()["last_probe_path"] == expect, name
        cache.set_probe_path("tensor" if expect == 2 else "exact")
        c = [t.cpu().numpy() for t in cache.probe(T(Q, dev))]
        for x, y in zip(a, c):
            assert np.array_equal(x.view(np.uint8), y.view(np.uint8))
        cache.close()


@pytest.mark.parametrize("path", PATHS)
def test_probe_special_queries(dev, path):
    """Queries with NaN or infinite features, and of magnitude 1e30, miss on
    every path (the strict test fails; nothing is accepted that the oracle
    rejects); a zero query and tiny ones get the oracle's answer."""
    w = synth.WORKLOADS["cifar10"].scaled(N=4000, n_queries=64)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    cache, _ = make_cache(dev, W, b, w.N)
    cache.insert(T(rows, dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    q = np.tile(rows[:1], (8, 1)).astype(np.float32)
    q[0, 3] = np.nan
    q[1, :] = np.inf
    q[2, 7] = -np.inf
    q[3] *= np.float32(1e30)
    q[4] = 0
    q[5] *= np.float32(1e-30)
    # q[6], q[7]: the cached row itself and a copy
    gi, gl, gd = run_probe(cache, q, dev, 64, path)
    assert np.all(gi[:4] == -1) and np.all(gl[:4] == -1) and np.all(np.isinf(gd[:4]))
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], q)
    check_probe(gi, gl, gd, ref, q, orc)
    assert gi[6] == 0 and gi[7] == 0
    cache.close()
