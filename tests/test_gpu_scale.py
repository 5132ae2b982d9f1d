"""The 4M-entry scale workload at full size, in the launch configuration the
benchmark times (insert batches of 65,536, probe batches of 4,096 on the
default path), against the FP64 oracle: every row's certification and every
one of the 16,384 queries against the whole cache (the oracle's brute force
takes about 5 minutes on 16 cores) (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from parity_utils import check_probe, record_parity

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def scale():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_13144_gb300.lipcache import LipCache
    dev = torch.device("cuda", 0)
    w = synth.WORKLOADS["scale"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, src = synth.queries(w, rows)
    cache = LipCache(w.d, w.C, w.N, device=dev)
    sigma = cache.set_head(torch.from_numpy(W).to(dev), torch.from_numpy(b).to(dev))
    rows_d = torch.from_numpy(rows).to(dev)
    idx, rad = [], []
    for s, e in synth.batches(w.N, w.insert_batch):
        i, r, _ = cache.insert(rows_d[s:e])
        idx.append(i.cpu().numpy())
        rad.append(r.cpu().numpy())
    del rows_d
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    yield dict(w=w, W=W, b=b, rows=rows, Q=Q, src=src, cache=cache, dev=dev, sigma=sigma,
               g_index=np.concatenate(idx), g_radius=np.concatenate(rad), ref=ref)
    cache.close()


def test_scale_insert_full(scale):
    """Every one of the 4M rows: acceptance and cache index bit-exact, radius
    within 1e-5 (the oracle's FP64 certification of all rows)."""
    s = scale
    ref = s["ref"]
    assert abs(s["sigma"] - oracle.sigma_max(s["W"])) <= 1e-10
    np.testing.assert_array_equal(s["g_index"], ref["index"])
    r = ref["cert"]["radius"]
    m = np.isfinite(r) & (r > 0)
    np.testing.assert_allclose(s["g_radius"][m], r[m], rtol=1e-5)
    assert s["cache"].size == len(ref["keys"])


def test_scale_probe_all_queries(scale):
    """All 16,384 queries (four batches of 4,096 on the default path) against
    the oracle's brute force over the whole 4M-entry cache: every GPU hit an
    exact FP64 hit, labels and distances as the oracle's, and every decision
    and selected index identical outside the 1e-5 band (Algorithm 2,
    Eqs. 13-15). The band counts are recorded (LIPCACHE_PARITY_OUT)."""
    s = scale
    w, ref, Q = s["w"], s["ref"], s["Q"]
    cache = s["cache"]
    cache.set_probe_path("auto")
    out = [[], [], []]
    for a, e in synth.batches(len(Q), w.batch):
        for k, t in enumerate(cache.probe(torch.from_numpy(Q[a:e]).to(s["dev"]))):
            out[k].append(t.cpu().numpy())
        assert cache.info()["device_errors"] == 0 and cache.info()["last_probe_path"] == 3
    gi, gl, gd = (np.concatenate(x) for x in out)
    assert (gi >= 0).sum() > 0
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q)
    stats = check_probe(gi, gl, gd, ref, Q, orc)
    record_parity("scale", "tensor", stats)
    print("scale", stats)


def test_scale_probe_hit_rich(scale):
    """A hit-rich batch against the 4M-entry cache (35 % near-duplicates with
    noise 0.002 per feature, so that most of them fall inside their entry's
    radius, as at the paper's operating points where a third to a half of the
    queries hit): every GPU hit is an exact FP64 hit with the oracle's label
    and distance, and the near-duplicates of the first 1,024 queries plus 64
    fresh ones match the oracle's brute force over the whole cache outside
    the 1e-5 band. The exact kernel gives the same bits."""
    s = scale
    w = s["w"].scaled(noise=0.002, dup_frac=0.35)
    ref = s["ref"]
    Q, src = synth.queries(w, s["rows"])
    q = Q[: w.batch]
    cache = s["cache"]
    cache.set_probe_path("auto")
    gi, gl, gd = [t.cpu().numpy() for t in cache.probe(torch.from_numpy(q).to(s["dev"]))]
    assert cache.info()["device_errors"] == 0 and cache.info()["last_probe_path"] == 3
    hits = gi >= 0
    assert hits.mean() > 0.3, hits.mean()
    D = oracle.pair_dist(q, ref["keys"], np.nonzero(hits)[0], gi[hits])
    assert np.all(D < ref["radius"][gi[hits]])
    np.testing.assert_array_equal(gl[hits], ref["label"][gi[hits]])
    np.testing.assert_allclose(gd[hits].astype(np.float64), D, rtol=1e-5)
    rng = np.random.default_rng(4)
    dup = np.nonzero(src[:1024] >= 0)[0]
    fresh = np.nonzero(src[:1024] < 0)[0]
    pick = np.sort(np.concatenate([dup, rng.choice(fresh, 64, replace=False)]))
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], q[pick])
    stats = check_probe(gi[pick], gl[pick], gd[pick], ref, q[pick], orc)
    record_parity("scale-hit-rich (sample)", "tensor", stats)
    cache.set_probe_path("exact")
    ge = [t.cpu().numpy() for t in cache.probe(torch.from_numpy(q).to(s["dev"]))]
    cache.set_probe_path("auto")
    assert np.array_equal(ge[0], gi) and np.array_equal(ge[2].view(np.uint32), gd.view(np.uint32))
    print("scale hit-rich", stats, "batch hit rate", hits.mean())


def test_scale_tensor_equals_exact(scale):
    """The same batch through the exact kernel (every pair on CUDA cores) and
    both tensor kernels: bit-identical outputs at full size."""
    s = scale
    q = torch.from_numpy(s["Q"][: s["w"].batch]).to(s["dev"])
    cache = s["cache"]
    outs = {}
    for path in ("exact", "tensor_single", "tensor_pair"):
        cache.set_probe_path(path)
        outs[path] = [t.cpu().numpy() for t in cache.probe(q)]
        assert cache.info()["device_errors"] == 0
    cache.set_probe_path("auto")
    for path in ("tensor_single", "tensor_pair"):
        for x, y in zip(outs["exact"], outs[path]):
            assert np.array_equal(x.view(np.uint8) if x.dtype == np.float32 else x,
                                  y.view(np.uint8) if y.dtype == np.float32 else y), path


def test_scale_tight_radius_rows(scale):
    """The tight radius (Eq. 29) on 262,144 rows of the 4M-entry workload
    (four 65,536-row launches, the benchmark's batch): acceptance and indices
    bit-exact, radii within the compensated refinement's bound of the oracle's
    FP64 tight radius."""
    from paper_2608_13144_gb300.lipcache import LipCache
    from parity_utils import check_insert
    s = scale
    w = s["w"]
    rows = s["rows"][:262144]
    c = LipCache(w.d, w.C, len(rows), "tight", device=s["dev"])
    c.set_head(torch.from_numpy(s["W"]).to(s["dev"]), torch.from_numpy(s["b"]).to(s["dev"]))
    rd = torch.from_numpy(rows).to(s["dev"])
    idx, rad, n = [], [], 0
    for a, e in synth.batches(len(rows), w.insert_batch):
        i, r, k = c.insert(rd[a:e])
        idx.append(i.cpu().numpy())
        rad.append(r.cpu().numpy())
        n += k
    assert c.info()["last_insert_kernel"] == 4  # the tensor certify kernel
    ref = oracle.build_cache(s["W"], s["b"], oracle.sigma_max(s["W"]), rows, radius_mode=oracle.RADIUS_TIGHT)
    check_insert(np.concatenate(idx), np.concatenate(rad), n, ref, ("tight", s["W"], s["b"], rows, 1.0))
    c.close()
