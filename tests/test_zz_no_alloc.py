"""lipcache_probe_noalloc, the lookup for callers that cannot allocate device
memory while they run (their device memory belongs to another allocator, or
their latency budget cannot absorb a cudaMalloc/cudaFree, which may block and
synchronise the device). It uses one fixed scratch array compiled into the
library instead of scratch grown with cudaMalloc.

Through the C ABI, two calls in a row must return what lipcache_probe returns
for the same batches (indices and labels exactly, distances within the 1e-5
relative tolerance of the parity tests), on every probe kernel, for the
largest documented batch and a ragged one; nothing may be allocated on a
fresh handle; batches too large for the array must be refused with
E_INVALID. This file is collected
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


def _compare(c, Q, dev, spans):
    """Two or more calls in a row on different batches: the no-allocation
    probe returns what lipcache_probe returns."""
    hits = 0
    for s, e in spans:
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


@pytest.mark.parametrize("path", ["tensor", "tensor_pair", "exact"])
def test_noalloc_matches_probe_twice(dev, path):
    w = synth.WORKLOADS["cifar100"].scaled(N=20000, n_queries=3000)
    c, Q = _cache(dev, w)
    c.set_probe_path(path)
    _compare(c, Q, dev, [(0, 1500), (1500, 3000)])
    c.close()


@pytest.mark.parametrize("path", ["tensor", "tensor_pair"])
def test_noalloc_largest_batch_and_ragged(dev, path):
    """d = 256 (d_pad = 256): the documented largest batch, 4,096 queries,
    fills the array; then a batch of 1,100 queries (padded to 1,152 rows, not
    a multiple of 256) exercises the kernels' row guards on the array's
    exactly sized regions."""
    from paper_2608_13144_gb300 import _lib
    # near-duplicates close enough to hit (the head's radii are ~0.1 here)
    w = synth.WORKLOADS["tinyimagenet"].scaled(N=20000, n_queries=5196, noise=0.002)
    assert (4096 * (4 * 256 + 12) + 512) <= _lib.NOALLOC_SCRATCH_BYTES
    c, Q = _cache(dev, w)
    c.set_probe_path(path)
    _compare(c, Q, dev, [(0, 4096), (4096, 5196)])
    c.close()


def test_noalloc_allocates_nothing_on_a_fresh_handle(dev):
    """On a handle whose probe scratch was never grown, the no-allocation
    probe leaves the device's free memory and torch's allocator unchanged,
    while an ordinary probe of the same batch then allocates its scratch."""
    w = synth.WORKLOADS["tinyimagenet"].scaled(N=5000, n_queries=4096, noise=0.002)
    # warm-up on another handle: loads the kernels' modules and resolves the
    # array's device address, both of which may take device memory once
    warm, Qw = _cache(dev, w)
    _noalloc(warm, Qw, dev)
    warm.probe(Qw)
    torch.cuda.synchronize(dev)
    warm.close()
    c, Q = _cache(dev, w)
    torch.cuda.synchronize(dev)
    free0 = torch.cuda.mem_get_info(dev)[0]
    alloc0 = torch.cuda.memory_stats(dev).get("allocation.all.allocated", 0)
    out = (torch.empty(4096, dtype=torch.int64, device=dev), torch.empty(4096, dtype=torch.int32, device=dev),
           torch.empty(4096, dtype=torch.float32, device=dev))
    alloc1 = torch.cuda.memory_stats(dev).get("allocation.all.allocated", 0)
    torch.cuda.synchronize(dev)
    free1 = torch.cuda.mem_get_info(dev)[0]
    for _ in range(2):
        st = c.L.lipcache_probe_noalloc(c._h, C.c_void_p(Q.data_ptr()), 4096, C.c_void_p(out[0].data_ptr()),
                                        C.c_void_p(out[1].data_ptr()), C.c_void_p(out[2].data_ptr()),
                                        C.c_void_p(torch.cuda.current_stream(dev).cuda_stream))
        assert st == 0, c.L.lipcache_last_error()
    torch.cuda.synchronize(dev)
    assert torch.cuda.mem_get_info(dev)[0] == free1
    assert torch.cuda.memory_stats(dev).get("allocation.all.allocated", 0) == alloc1
    assert int((out[0] >= 0).sum()) > 0
    # the check can see an allocation: the ordinary probe grows ~4 MB of scratch
    c.probe(Q)
    torch.cuda.synchronize(dev)
    assert torch.cuda.mem_get_info(dev)[0] < free1
    assert alloc1 >= alloc0 and free1 <= free0
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
