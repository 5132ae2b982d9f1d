"""lipcache_probe_noalloc, the lookup for callers that cannot allocate device
memory while they run (their device memory belongs to another allocator, or
their latency budget cannot absorb a cudaMalloc/cudaFree, which may block and
synchronise the device). It uses one fixed scratch array compiled into the
library instead of scratch grown with cudaMalloc.

Through the C ABI, two calls in a row must return what lipcache_probe returns
for the same batches (indices and labels exactly, distances within the 1e-5
relative tolerance of the parity tests), on both probe kernels; batches too
large for the array must be refused with E_INVALID. This file is collected
last and also passes on its own in a fresh process.
"""
import ctypes as C

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def _cache(dev, w):
    from paper_2608_13144_gb300.lipcache import LipCache
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    c = LipCache(w.d, w.C, w.N, device=dev)
    c.set_head(torch.from_numpy(W).to(dev), torch.from_numpy(b).to(dev))
    c.insert(torch.from_numpy(rows).to(dev))
    return c, torch.from_numpy(Q).to(dev)


def _noalloc(c, Qb, dev):
    B = Qb.shape[0]
    out = (torch.full((B,), -7, dtype=torch.int64, device=dev), torch.full((B,), -7, dtype=torch.int32, device=dev),
           torch.full((B,), -7.0, dtype=torch.float32, device=dev))
    st = c.L.lipcache_probe_noalloc(c._h, C.c_void_p(Qb.data_ptr()), B, C.c_void_p(out[0].data_ptr()),
                                    C.c_void_p(out[1].data_ptr()), C.c_void_p(out[2].data_ptr()),
                                    C.c_void_p(torch.cuda.current_stream(dev).cuda_stream))
    assert st == 0, c.L.lipcache_last_error()
    return [t.cpu().numpy() for t in out]


@pytest.mark.parametrize("path", ["tensor", "exact"])
def test_noalloc_matches_probe_twice(dev, path):
    w = synth.WORKLOADS["cifar100"].scaled(N=20000, n_queries=3000)
    c, Q = _cache(dev, w)
    c.set_probe_path(path)
    hits = 0
    for s, e in [(0, 1500), (1500, 3000)]:  # two calls in a row, different batches
        Qb = Q[s:e].contiguous()
        ref = [t.cpu().numpy() for t in c.probe(Qb)]
        got = _noalloc(c, Qb, dev)
        assert np.array_equal(got[0], ref[0])
        assert np.array_equal(got[1], ref[1])
        hit = ref[0] >= 0
        np.testing.assert_allclose(got[2][hit], ref[2][hit], rtol=1e-5)
        assert np.all(np.isinf(got[2][~hit]))
        hits += int(hit.sum())
    assert hits > 0
    assert c.info()["device_errors"] == 0
    c.close()


def test_noalloc_rejects_oversized_batch(dev):
    from paper_2608_13144_gb300 import _lib
    w = synth.WORKLOADS["cifar100"].scaled(N=1000, n_queries=10)
    c, _ = _cache(dev, w)
    dpad = 128
    too_many = _lib.NOALLOC_SCRATCH_BYTES // (4 * dpad + 12) + 256
    Qbig = torch.zeros((too_many, w.d), dtype=torch.float32, device=dev)
    out = [torch.empty(too_many, dtype=torch.int64, device=dev), None, None]
    st = c.L.lipcache_probe_noalloc(c._h, C.c_void_p(Qbig.data_ptr()), too_many, C.c_void_p(out[0].data_ptr()),
                                    None, None, C.c_void_p(torch.cuda.current_stream(dev).cuda_stream))
    assert st == _lib.E_INVALID
    assert b"too large" in c.L.lipcache_last_error()
    c.close()
