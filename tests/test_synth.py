import numpy as np

import synth


def test_workload_shapes_and_determinism():
    w = synth.WORKLOADS["tiny"]
    W, b = synth.head(w)
    assert W.shape == (w.C, w.d) and b.shape == (w.C,) and W.dtype == np.float32
    rows = synth.cache_rows(w)
    assert rows.shape == (w.N, w.d) and rows.dtype == np.float32
    Q, src = synth.queries(w, rows)
    assert Q.shape == (w.n_queries, w.d)
    assert (src >= 0).sum() == round(w.dup_frac * w.n_queries)
    rows2 = synth.cache_rows(w)
    np.testing.assert_array_equal(rows, rows2)
    Q2, _ = synth.queries(w, rows2)
    np.testing.assert_array_equal(Q, Q2)
    dup = src >= 0
    # near-duplicates sit about noise * sqrt(d) from their source row
    dist = np.linalg.norm(Q[dup] - rows[src[dup]], axis=1)
    assert abs(dist.mean() - w.noise * np.sqrt(w.d)) < 0.05


def test_mixture_geometry():
    w = synth.WORKLOADS["cifar10"].scaled(N=4000)
    ctr = synth.centres(w)
    np.testing.assert_allclose(np.linalg.norm(ctr, axis=1), w.sphere_radius)
    rows = synth.cache_rows(w)
    nearest = np.min(((rows[:, None, :] - ctr[None]) ** 2).sum(-1), axis=1)
    assert abs(nearest.mean() / w.d - w.sigma ** 2) < 0.05 * w.sigma ** 2


def test_batches_ragged():
    assert synth.batches(10, 4) == [(0, 4), (4, 8), (8, 10)]
    assert synth.batches(0, 4) == []
