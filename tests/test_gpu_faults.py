"""Failure detection on the GPU without a fault: a probe whose MMA issuer
waits on a barrier nothing arrives on must give up after its bounded wait,
report the batch as misses and an error, and leave the context usable
(pytest -m gpu)."""
import time

import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

STALL = 1  # LIPCACHE_DEBUG_STALL_PROBE


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


@pytest.mark.parametrize("path", ["tensor_single", "tensor_pair"])
def test_stalled_probe_aborts_and_recovers(dev, path):
    from paper_2608_13144_gb300._lib import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    cache = LipCache(w.d, w.C, w.N + w.n_queries, device=dev)
    cache.set_head(torch.from_numpy(W).to(dev), torch.from_numpy(b).to(dev))
    cache.insert(torch.from_numpy(rows).to(dev))
    cache.set_probe_path(path)
    q = torch.from_numpy(Q).to(dev)
    base = [t.cpu().numpy() for t in cache.probe(q)]
    assert (base[0] >= 0).sum() > 0

    cache.set_debug(STALL)
    cache.reset_stats()
    t0 = time.perf_counter()
    gi, gl, gd = [t.cpu().numpy() for t in cache.probe(q)]
    waited = time.perf_counter() - t0
    assert np.all(gi == -1) and np.all(gl == -1) and np.all(np.isinf(gd))
    assert cache.info()["device_errors"] > 0
    assert 0.05 < waited < 30  # the bounded wait, not a hang
    with pytest.raises(LipCacheError) as e:
        cache.probe_host(torch.from_numpy(Q))
    assert e.value.status == 8  # LIPCACHE_E_DEVICE
    size = cache.size
    with pytest.raises(LipCacheError) as e:
        cache.probe_writeback(q)
    assert e.value.status == 8 and cache.size == size  # nothing written back
    cache.set_probe_path("exact")  # no waits in the exact kernel: unaffected
    ge = cache.probe(q)[0].cpu().numpy()
    np.testing.assert_array_equal(ge, base[0])

    cache.set_debug(0)
    cache.set_probe_path(path)
    cache.reset_stats()
    again = [t.cpu().numpy() for t in cache.probe(q)]
    for x, y in zip(base, again):
        np.testing.assert_array_equal(x, y)
    assert cache.info()["device_errors"] == 0
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    hits = again[0] >= 0
    D = oracle.pair_dist(Q, ref["keys"], np.nonzero(hits)[0], again[0][hits])
    assert np.all(D < ref["radius"][again[0][hits]])
    cache.close()


def test_debug_flags_validated(dev):
    from paper_2608_13144_gb300._lib import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(4, 2, 8, device=dev)
    with pytest.raises(LipCacheError) as e:
        c.set_debug(6)
    assert e.value.status == 1
    c.close()
