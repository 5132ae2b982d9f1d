"""Failure detection on the GPU without a fault: a probe or a tensor certify
kernel whose MMA issuer waits on a barrier nothing arrives on must give up
after its bounded wait, report an error (the probe's batch as misses, no
inserted row), and leave the context usable (pytest -m gpu)."""
import time

import numpy as np
import pytest

import oracle
import synth
from parity_utils import check_insert

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
        c.set_debug(32)
    assert e.value.status == 1
    c.set_debug(2 | 4 | 8 | 16)  # every known flag together is accepted
    c.set_debug(0)
    c.close()


def test_certify_stall_aborts_cleanly(dev):
    """A bounded wait of the tensor certify kernel that expires (a barrier
    nothing arrives on) aborts the kernel: the insert returns E_DEVICE,
    appends nothing and counts a device error; the next insert works and
    matches the oracle."""
    from paper_2608_13144_gb300._lib import LipCacheError
    from paper_2608_13144_gb300.lipcache import LipCache
    w = synth.WORKLOADS["cifar100"].scaled(N=2000)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    c = LipCache(w.d, w.C, 2 * len(rows), device=dev)
    c.set_head(torch.from_numpy(W).to(dev), torch.from_numpy(b).to(dev))
    c.set_debug(8)
    with pytest.raises(LipCacheError) as e:
        c.insert(torch.from_numpy(rows).to(dev))
    assert e.value.status == 8 and c.size == 0  # LIPCACHE_E_DEVICE
    assert c.info()["last_insert_kernel"] == 4 and c.info()["device_errors"] >= 1
    c.set_debug(0)
    idx, rad, n = c.insert(torch.from_numpy(rows).to(dev))
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(idx.cpu().numpy(), rad.cpu().numpy(), n, ref, (W, b, rows, 1.0))
    assert c.size == n
    c.close()
