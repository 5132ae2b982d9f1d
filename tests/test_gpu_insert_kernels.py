"""The certify kernels against each other and the FP64 oracle (pytest -m
gpu). The wide-tile kernel (128-row tiles, logits in registers) and the
64-row-tile kernel form the same FP32 logit chains, candidate sets,
compensated refinements and FP64 finals, so their outputs agree bit for bit.
The tensor kernel (TF32 tcgen05 screen) picks its candidates from wider
intervals but refines them in the same order, so its radii, labels and
entries agree bit for bit with the wide-tile kernel too; the oracle pins the
values."""
import numpy as np
import pytest

import oracle
import synth
from parity_utils import check_insert, radius_tol

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

WIDE_TILE, TILE64, STREAMED, TENSOR = 1, 2, 3, 4
DEBUG_INSERT_TILE64, DEBUG_INSERT_WIDE_TILE, DEBUG_INSERT_FIX_STANDALONE = 2, 4, 16


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def T(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def build(dev, W, b, rows, batch, tile64, payload=None, consistency=False):
    """tile64: True forces the 64-row-tile kernel, "wide" the wide-tile one,
    False leaves the choice to the library."""
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], len(rows), device=dev)
    c.set_head(T(W, dev), T(b, dev))
    if tile64 == "wide":
        c.set_debug(DEBUG_INSERT_WIDE_TILE)
    elif tile64:
        c.set_debug(DEBUG_INSERT_TILE64)
    idx, rad, n = [], [], 0
    for s, e in synth.batches(len(rows), batch):
        p = None if payload is None else T(payload[s:e], dev)
        i, r, k = c.insert(T(rows[s:e], dev), p, consistency)
        idx.append(i.cpu().numpy())
        rad.append(r.cpu().numpy())
        n += k
    return c, np.concatenate(idx), np.concatenate(rad), n


def same_bits(x, y):
    x, y = np.asarray(x), np.asarray(y)
    if x.dtype == np.float32:
        x, y = x.view(np.uint32), y.view(np.uint32)
    return x.shape == y.shape and np.array_equal(x, y)


# (d, C, rows, insert batch): every compiled per-thread class count (1, 4, 7,
# 13, 16), ragged last tiles, several tiles per CTA, one-tile batches
SHAPES = [(16, 10, 1000, 1000), (64, 10, 20000, 20000), (128, 100, 30001, 30001), (128, 200, 40000, 16384),
          (96, 250, 3000, 3000), (20, 40, 777, 100), (8, 3, 65, 65), (128, 200, 200, 64)]


@pytest.mark.parametrize("d,C,N,batch", SHAPES)
def test_wide_tile_bit_identical_and_oracle(dev, d, C, N, batch):
    w = synth.WORKLOADS["cifar100"].scaled(d=d, C=C, components=C, N=N, n_queries=512, sphere_radius=4.0)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    a, ia, ra, na = build(dev, W, b, rows, batch, "wide")
    assert a.info()["last_insert_kernel"] == WIDE_TILE
    s, is_, rs, ns = build(dev, W, b, rows, batch, True)
    assert s.info()["last_insert_kernel"] == TILE64
    assert na == ns and same_bits(ia, is_) and same_bits(ra, rs)
    ea, es = a.entries(), s.entries()
    for k in ("keys", "radius", "label", "yG"):
        assert same_bits(ea[k], es[k]), k
    # the probe thresholds (not exported) agree through every probe result
    for path in ("exact", "tensor"):
        a.set_probe_path(path)
        s.set_probe_path(path)
        for x, y in zip(a.probe(T(Q, dev)), s.probe(T(Q, dev))):
            assert same_bits(x.cpu().numpy(), y.cpu().numpy()), path
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    a.close()
    s.close()


# (d, C, rows, insert batch) for the tensor kernel: one and two feature
# buffers, one and two column halves (C <= 32 and C > 32), C = 256 (N = 256,
# eight column chunks), d % 32 == 16, ragged last tiles, fewer tiles than SMs,
# batches smaller than one tile
TC_SHAPES = [(32, 10, 3000, 3000), (64, 10, 20000, 20000), (128, 100, 30001, 30001), (128, 200, 40000, 16384),
             (96, 250, 3000, 3000), (48, 3, 777, 100), (128, 200, 200, 64), (96, 256, 70000, 65536),
             (32, 2, 500, 500)]


@pytest.mark.parametrize("d,C,N,batch", TC_SHAPES)
def test_tensor_bit_identical_and_oracle(dev, d, C, N, batch):
    """The tensor kernel (TF32 screen into TMEM) against the wide-tile kernel:
    every output and stored entry bit for bit, every probe result too (the
    thresholds are not exported), and the oracle."""
    w = synth.WORKLOADS["cifar100"].scaled(d=d, C=C, components=C, N=N, n_queries=512, sphere_radius=4.0)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    a, ia, ra, na = build(dev, W, b, rows, batch, False)
    assert a.info()["last_insert_kernel"] == TENSOR
    assert a.info()["device_errors"] == 0
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    s, is_, rs, ns = build(dev, W, b, rows, batch, "wide")
    if s.info()["last_insert_kernel"] == STREAMED:
        # too large for the wide-tile kernel: the streamed kernel refines with
        # 32 lanes, so only acceptance, indices and y^G agree bit for bit
        assert na == ns and np.array_equal(ia, is_)
        np.testing.assert_array_equal(a.entries()["yG"], s.entries()["yG"])
        a.close()
        s.close()
        return
    assert s.info()["last_insert_kernel"] == WIDE_TILE
    assert na == ns and same_bits(ia, is_) and same_bits(ra, rs)
    ea, es = a.entries(), s.entries()
    for k in ("keys", "radius", "label", "yG"):
        assert same_bits(ea[k], es[k]), k
    for path in ("exact", "tensor"):
        a.set_probe_path(path)
        s.set_probe_path(path)
        for x, y in zip(a.probe(T(Q, dev)), s.probe(T(Q, dev))):
            assert same_bits(x.cpu().numpy(), y.cpu().numpy()), path
    a.close()
    s.close()


def test_tensor_overflow_rows(dev):
    """19 identical head rows: rows whose top two lie in the tied group have
    more candidates than the per-row slots, so the tensor kernel refines
    every class of the row (in the 8-lane order) and the wide-tile kernel its
    one-warp path (32 lanes). Acceptance and indices agree; radii agree with
    the oracle within 1e-5 relative (rows a hair from a boundary go through
    the FP64 pass)."""
    rng = np.random.default_rng(21)
    d, C = 32, 24
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    W[1:20] = W[1]
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    b[1:20] = b[1]
    rows = np.concatenate([3 * W[0] + 0.3 * rng.standard_normal((700, d)),
                           3 * W[1] + 0.3 * rng.standard_normal((700, d)),
                           rng.standard_normal((600, d))]).astype(np.float32)
    a, ia, ra, na = build(dev, W, b, rows, len(rows), False)
    s, is_, rs, ns = build(dev, W, b, rows, len(rows), "wide")
    assert a.info()["last_insert_kernel"] == TENSOR and s.info()["last_insert_kernel"] == WIDE_TILE
    assert na == ns and np.array_equal(ia, is_)
    np.testing.assert_array_equal(a.entries()["yG"], s.entries()["yG"])
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    a.close()
    s.close()


def test_wide_tile_overflow_rows(dev):
    """More candidate classes per row than the per-row slots (19 identical
    head rows): the kernel recomputes those rows' logits and hands them to the
    one-warp refinement; identical to the 64-row-tile kernel."""
    rng = np.random.default_rng(21)
    d, C = 32, 24
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    W[1:20] = W[1]
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    b[1:20] = b[1]
    rows = np.concatenate([3 * W[0] + 0.3 * rng.standard_normal((700, d)),
                           3 * W[1] + 0.3 * rng.standard_normal((700, d)),
                           rng.standard_normal((600, d))]).astype(np.float32)
    a, ia, ra, na = build(dev, W, b, rows, len(rows), "wide")
    s, is_, rs, ns = build(dev, W, b, rows, len(rows), True)
    assert a.info()["last_insert_kernel"] == WIDE_TILE
    assert na == ns and same_bits(ia, is_) and same_bits(ra, rs)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    rep = check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    # near ties go through the FP64 pass on both kernels (a borderline row may
    # go on one only: the kernels refine different candidate sets, whose
    # largest error bound enters the test; the results agree bit for bit)
    assert a.info()["insert_fp64_rows"] > 0 and s.info()["insert_fp64_rows"] > 0
    print("rows re-certified in FP64:", a.info()["insert_fp64_rows"], "of", len(rows), "; in the FP64 band:",
          rep["fp64_band"])
    a.close()
    s.close()


@pytest.mark.parametrize("kernel", ["wide", False])
def test_wide_tile_payload_and_consistency(dev, kernel):
    """Payload labels and the consistency flag go through the same finals
    (wide-tile and tensor kernels against the 64-row-tile kernel)."""
    w = synth.WORKLOADS["cifar10"].scaled(N=6000)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    payload = (np.arange(len(rows)) % w.C).astype(np.int32)
    a, ia, ra, na = build(dev, W, b, rows, 4096, kernel, payload, True)
    assert a.info()["last_insert_kernel"] == (WIDE_TILE if kernel else TENSOR)
    s, is_, rs, ns = build(dev, W, b, rows, 4096, True, payload, True)
    assert na == ns and same_bits(ia, is_) and same_bits(ra, rs)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, payload=payload, require_consistency=True)
    check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    a.close()
    s.close()


def test_kernel_choice(dev):
    """Both radii take the tensor kernel where it applies (d % 16 == 0,
    32 <= d <= 256, 2 <= C <= 256, head resident); the other shapes take the
    wide-tile kernel (d % 4 == 0, head small enough), the 64-row one
    (d % 4 != 0) or the streamed one (large heads)."""
    from paper_2608_13144_gb300.lipcache import LipCache
    cases = [((64, 10), "tight", TENSOR), ((33, 10), "tight", TILE64), ((33, 10), "conservative", TILE64),
             ((256, 200), "conservative", STREAMED), ((128, 300), "conservative", STREAMED),
             ((128, 200), "conservative", TENSOR), ((64, 10), "conservative", TENSOR),
             ((32, 2), "conservative", TENSOR), ((16, 10), "conservative", WIDE_TILE),
             ((40, 10), "conservative", WIDE_TILE), ((128, 200), "tight", TENSOR), ((16, 10), "tight", WIDE_TILE),
             ((96, 256), "conservative", TENSOR), ((128, 256), "conservative", STREAMED)]
    rng = np.random.default_rng(5)
    for (d, C), mode, kernel in cases:
        W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
        b = np.zeros(C, np.float32)
        c = LipCache(d, C, 100, mode, device=dev)
        c.set_head(T(W, dev), T(b, dev))
        c.insert(T(rng.standard_normal((100, d)).astype(np.float32), dev))
        assert c.info()["last_insert_kernel"] == kernel, (d, C, mode)
        c.close()


def _near_ties(W, b, n, rng, k):
    """Rows whose top k logits agree to about 1e-6 relative: random points
    moved onto the set where classes a_1..a_k tie (least-squares step in the
    span of W_{a_i} - W_{a_1}), then perturbed slightly."""
    d = W.shape[1]
    W64, b64 = W.astype(np.float64), b.astype(np.float64)
    out = []
    for _ in range(n):
        z = rng.standard_normal(d) * 2.0
        s = W64 @ z + b64
        top = np.argsort(-s)[:k]
        D = W64[top[1:]] - W64[top[0]]              # (k-1) x d
        g = -(s[top[1:]] - s[top[0]])               # logit differences to cancel
        z = z + D.T @ np.linalg.lstsq(D @ D.T, g, rcond=None)[0]
        z = z + rng.standard_normal(d) * 1e-5 * np.linalg.norm(z) / np.sqrt(d)
        out.append(z)
    return np.asarray(out, dtype=np.float32)


@pytest.mark.parametrize("kernel", ["wide", False])
@pytest.mark.parametrize("d,C", [(16, 10), (64, 40), (128, 100), (128, 200), (96, 250)])
def test_wide_tile_near_ties(dev, d, C, kernel):
    """Rows on two- and three-way logit ties: several candidate classes per
    row, refinement deciding the order, margins near zero (some rows
    rejected). Bit-identical to the 64-row-tile kernel and within
    1e-5 relative of the oracle (after the FP64 pass for near ties)."""
    rng = np.random.default_rng(d * 1000 + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = np.concatenate([_near_ties(W, b, 600, rng, 2), _near_ties(W, b, 600, rng, 3),
                           rng.standard_normal((400, d)).astype(np.float32)])
    a, ia, ra, na = build(dev, W, b, rows, len(rows), kernel)
    s, is_, rs, ns = build(dev, W, b, rows, len(rows), True)
    assert a.info()["last_insert_kernel"] == (TENSOR if not kernel and d >= 32 else WIDE_TILE)
    assert na == ns and same_bits(ia, is_) and same_bits(ra, rs)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows)
    rep = check_insert(ia, ra, na, ref, (W, b, rows, 1.0))
    # near ties go through the FP64 pass on both kernels (a borderline row may
    # go on one only: the kernels refine different candidate sets, whose
    # largest error bound enters the test; the results agree bit for bit)
    assert a.info()["insert_fp64_rows"] > 0 and s.info()["insert_fp64_rows"] > 0
    print("rows re-certified in FP64:", a.info()["insert_fp64_rows"], "of", len(rows), "; in the FP64 band:",
          rep["fp64_band"])
    a.close()
    s.close()


@pytest.mark.parametrize("mode", ["conservative", "tight"])
@pytest.mark.parametrize("d,C", [(64, 40), (128, 200), (96, 250)])
def test_tensor_fp64_pass_in_kernel_and_standalone(dev, mode, d, C):
    """The tensor kernel's own FP64-pass warp (rows handed over through its
    shared-memory queue while the epilogue goes on) and the stand-alone pass
    launched after the kernel re-certify the same listed rows to the same
    bits: near-tie rows, several per tile, more than the queue's 32 slots per
    CTA in a launch."""
    from paper_2608_13144_gb300.lipcache import LipCache
    rng = np.random.default_rng(7 * d + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = np.concatenate([_near_ties(W, b, 1500, rng, 2), _near_ties(W, b, 500, rng, 3),
                           rng.standard_normal((2000, d)).astype(np.float32)])
    rows = rows[rng.permutation(len(rows))]
    out = []
    for flags in (0, DEBUG_INSERT_FIX_STANDALONE):
        c = LipCache(d, C, len(rows), mode, device=dev)
        c.set_head(T(W, dev), T(b, dev))
        c.set_debug(flags)
        i, r, n = c.insert(T(rows, dev))
        inf = c.info()
        assert inf["last_insert_kernel"] == TENSOR
        out.append((i.cpu().numpy(), r.cpu().numpy(), n, inf["insert_fp64_rows"]))
        c.close()
    (ia, ra, na, fa), (ib, rb, nb, fb) = out
    assert fa == fb and fa > 64, (fa, fb)
    assert na == nb and same_bits(ia, ib) and same_bits(ra, rb)


def build_tight(dev, W, b, rows, tile64, kappa=1.0):
    """tile64 as in build(): True, "wide" or False (the library's choice)."""
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], len(rows), "tight", device=dev)
    c.set_radius_scale(kappa)
    c.set_head(T(W, dev), T(b, dev))
    if tile64 == "wide":
        c.set_debug(DEBUG_INSERT_WIDE_TILE)
    elif tile64:
        c.set_debug(DEBUG_INSERT_TILE64)
    i, r, n = c.insert(T(rows, dev))
    return c, i.cpu().numpy(), r.cpu().numpy(), n


@pytest.mark.parametrize("d,C,kappa", [(16, 10, 1.0), (64, 40, 0.8), (128, 100, 1.0), (128, 200, 1.0),
                                       (96, 250, 0.9)])
def test_wide_tile_tight_radius(dev, d, C, kappa):
    """Tight radius (Eq. 29) on the wide-tile kernel: y^G settled by the FP32
    intervals, the minimiser among the classes whose bracket of
    (s_y - s_j) / ||W_y - W_j|| can reach the smallest upper bracket, refined
    with the compensated dot product; rows the intervals cannot settle (ties
    among the top classes) on one warp. Against the oracle and the kernels
    that refine every class in FP64 (64-row or streamed): the same acceptance
    and y^G, radii within 1e-5 relative (FP64-resolution slack at exact
    near ties)."""
    rng = np.random.default_rng(d * 7 + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = np.concatenate([rng.standard_normal((3000, d)).astype(np.float32) * 2,
                           _near_ties(W, b, 300, rng, 2), _near_ties(W, b, 300, rng, 3)])
    a, ia, ra, na = build_tight(dev, W, b, rows, "wide", kappa)
    assert a.info()["last_insert_kernel"] == WIDE_TILE
    s, is_, rs, ns = build_tight(dev, W, b, rows, True, kappa)
    assert s.info()["last_insert_kernel"] in (TILE64, STREAMED)  # FP64 refinement of every class
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=oracle.RADIUS_TIGHT, scale=kappa)
    check_insert(ia, ra, na, ref, ("tight", W, b, rows, kappa))
    assert na == ns and np.array_equal(ia, is_)
    np.testing.assert_array_equal(a.entries()["yG"], s.entries()["yG"])
    m = np.isfinite(rs) & (rs > 0)
    tol = radius_tol(W, b, rows, rs, kappa, tight=True)  # each kernel within it of the exact radius
    assert np.all(np.abs(ra[m].astype(np.float64) - rs[m]) <= 2 * tol[m])
    a.close()
    s.close()


@pytest.mark.parametrize("d,C,kappa", [(32, 10, 1.0), (64, 40, 0.8), (128, 100, 1.0), (128, 200, 1.0),
                                       (96, 250, 0.9), (48, 3, 1.0)])
def test_tensor_tight_radius(dev, d, C, kappa):
    """The tight radius (Eq. 29) on the tensor kernel: y^G settled by the
    screen, the candidates of Eq. 29 from the runner-up's bracket and the
    head's smallest reciprocal pair norm, the same compensated refinement and
    FP64 terms as the wide-tile kernel; rows on ties take the one-warp path.
    Acceptance, indices and y^G as the wide-tile kernel and the oracle; radii
    within 1e-5 relative of both."""
    rng = np.random.default_rng(d * 11 + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = np.concatenate([rng.standard_normal((3000, d)).astype(np.float32) * 2,
                           _near_ties(W, b, 300, rng, 2), _near_ties(W, b, 300, rng, 3)])
    a, ia, ra, na = build_tight(dev, W, b, rows, False, kappa)
    assert a.info()["last_insert_kernel"] == TENSOR and a.info()["device_errors"] == 0
    s, is_, rs, ns = build_tight(dev, W, b, rows, "wide", kappa)
    assert s.info()["last_insert_kernel"] == WIDE_TILE
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=oracle.RADIUS_TIGHT, scale=kappa)
    check_insert(ia, ra, na, ref, ("tight", W, b, rows, kappa))
    assert na == ns and np.array_equal(ia, is_)
    np.testing.assert_array_equal(a.entries()["yG"], s.entries()["yG"])
    m = np.isfinite(rs) & (rs > 0)
    tol = radius_tol(W, b, rows, rs, kappa, tight=True)  # each kernel within it of the exact radius
    assert np.all(np.abs(ra[m].astype(np.float64) - rs[m]) <= 2 * tol[m])
    print("tight radii bit-identical to the wide-tile kernel:", np.mean(ra.view(np.uint32) == rs.view(np.uint32)),
          "rows on the one-warp path:", a.info()["insert_full_rows"])
    a.close()
    s.close()


def test_wide_tile_tight_tied_head_rows(dev):
    """Identical head rows (||W_y - W_j|| = 0, skipped by Eq. 29) and rows won
    by the tied group (several possible y^G: the one-warp row path), on the
    wide-tile and the tensor kernel."""
    rng = np.random.default_rng(21)
    d, C = 32, 24
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    W[1:20] = W[1]
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    b[1:20] = b[1]
    rows = np.concatenate([3 * W[0] + 0.3 * rng.standard_normal((700, d)),
                           3 * W[1] + 0.3 * rng.standard_normal((700, d)),
                           rng.standard_normal((600, d))]).astype(np.float32)
    for kernel, expect in (("wide", WIDE_TILE), (False, TENSOR)):
        a, ia, ra, na = build_tight(dev, W, b, rows, kernel)
        assert a.info()["last_insert_kernel"] == expect
        ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=oracle.RADIUS_TIGHT)
        check_insert(ia, ra, na, ref, ("tight", W, b, rows, 1.0))
        a.close()


@pytest.mark.parametrize("d,C,kernel", [(33, 7, TILE64), (21, 40, TILE64), (256, 200, STREAMED), (128, 300, STREAMED)])
def test_tight_radius_other_kernels(dev, d, C, kernel):
    """The tight radius on the kernels that refine every class in FP64
    (d % 4 != 0; heads too large for shared memory) against the oracle,
    rows on logit ties included."""
    rng = np.random.default_rng(d * 13 + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    rows = np.concatenate([rng.standard_normal((800, d)).astype(np.float32) * 2,
                           _near_ties(W, b, 100, rng, 2), _near_ties(W, b, 100, rng, 3)])
    c, i, r, n = build_tight(dev, W, b, rows, False)
    assert c.info()["last_insert_kernel"] == kernel
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=oracle.RADIUS_TIGHT)
    check_insert(i, r, n, ref)  # FP64 refinement of every class
    c.close()


@pytest.mark.parametrize("mode", ["conservative", "tight"])
@pytest.mark.parametrize("d,C", [(16, 10), (128, 200)])
def test_certify_special_values(dev, mode, d, C):
    """Rows with NaN or infinite features are skipped (a NaN margin fails
    r > 0); zero rows and rows of magnitude 1e-30 or 1e30 are certified like
    any other. Acceptance and indices bit-exact with the oracle, radii within
    1e-5 relative. Probes of the accepted rows inside FP32's range hit
    themselves; the 1e30 row (its |k|^2 overflows FP32, so it has no
    threshold) is never hit, and the zero row ties at FP32 distance 0 with the
    1e-30 row (their squared distance underflows), lowest index first."""
    from paper_2608_13144_gb300.lipcache import LipCache
    rng = np.random.default_rng(d + C)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (0.1 * rng.standard_normal(C)).astype(np.float32)
    base = rng.standard_normal((12, d)).astype(np.float32)
    rows = [base[0], base[1] * 1e-30, base[2] * 1e30, np.zeros(d, np.float32), base[3], base[4]]
    bad = base[5:11].copy()
    bad[0, 3] = np.nan
    bad[1, :] = np.nan
    bad[2, 0] = np.inf
    bad[3, 5] = -np.inf
    rows = np.concatenate([np.stack(rows), bad, base[11:]]).astype(np.float32)
    c = LipCache(d, C, len(rows), mode, device=dev)
    c.set_head(T(W, dev), T(b, dev))
    i, r, n = c.insert(T(rows, dev))
    i, r = i.cpu().numpy(), r.cpu().numpy()
    assert c.info()["last_insert_kernel"] == (TENSOR if d >= 32 else WIDE_TILE)
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=int(mode == "tight"))
    head = ("tight", W, b, rows, 1.0) if mode == "tight" else (W, b, rows, 1.0)
    finite = np.all(np.isfinite(rows), axis=1)
    assert np.all(i[~finite] == -1)
    check_insert(i, r, n, ref, head)
    normal = [k for k in (0, 4, 5, 11) if i[k] >= 0]
    hit, _, dist = c.probe(T(rows[normal], dev))
    np.testing.assert_array_equal(hit.cpu().numpy(), i[normal])
    assert np.all(dist.cpu().numpy() == 0)
    if i[2] >= 0:
        assert c.probe(T(rows[2:3], dev))[0].item() == -1
    if i[1] >= 0 and i[3] >= 0:
        assert c.probe(T(rows[3:4], dev))[0].item() == min(i[1], i[3])
    c.close()
