"""The tensor-core screens' error bound, checked on the CPU by emulating the
TF32 operands (the 13 low mantissa bits dropped) and an FP32 accumulation.

The insert screen (tight and conservative radius) and the probe screen rely
on |a - u.v| <= c ||u|| ||v|| for the value a the TF32 MMA returns, with
c = 2 (2^-9 + 2^-20 + K 2^-22) + 2 gamma_K + 2^-20 for K-long products
(K = d rounded up to 32), and the insert screen on
|fl(a + b) - (u.v + b)| <= E = c wmax ||z|| + 2^-22 Mb. These tests take the
worst the arithmetic allows - truncated operands (maximal when every dropped
bit is 1, products of one sign) and FP32 partial sums in either order - and
check the bound and E. The worst cases reach about a quarter of c, i.e. half
of the undoubled TF32 term: the factor 2 in c is the safety margin, and a
bound built on 2^-10 per product instead of 2^-9 would have none left.

The second half emulates the insert kernel's candidate screens on
adversarial screen errors of up to E: the conservative radius's threshold
l2 - 2E always keeps the true top two, and the tight radius's (Eq. 29)
bracket and union tests keep what gives the oracle's y^G and r*, including
the union test's two corner cases for uncertain rows (a NaN second bound,
and a row that needs that bound). The last part emulates the probe's separable screen with its
directed roundings and the canonical FP32 recheck distance: every pair the
recheck would accept passes fl(a - tau_k) >= kappa_q, with about 60 % of the
slack c |q| |k| left in the worst cases (q near k, every product of one sign,
dropped bits all ones).
"""
import numpy as np
import pytest

U32 = 2.0 ** -24


def gamma32(n):
    return n * U32 / (1 - n * U32)


def c_screen(K):
    return 2 * (2.0 ** -9 + 2.0 ** -20 + K * 2.0 ** -22) + 2 * gamma32(K) + 2.0 ** -20


def tf32(x):
    """FP32 values with the 13 low mantissa bits cleared (TF32 truncation)."""
    b = np.asarray(x, np.float32).view(np.uint32) & np.uint32(0xFFFFE000)
    return b.view(np.float32)


def fp32_dot(u, v, reverse=False):
    """Sequential FP32 sum of the exact products (each product of two TF32
    values is exact in FP32: 11 + 11 significant bits)."""
    p = (u.astype(np.float32) * v.astype(np.float32)).astype(np.float32)
    acc = np.float32(0.0)
    for t in (p[::-1] if reverse else p):
        acc = np.float32(acc + t)
    return float(acc)


def worst_mantissa(rng, n, scale):
    """Values whose dropped 13 bits are all ones (the largest truncation
    error), random signs and exponents within a factor 4 of `scale`."""
    e = rng.integers(-2, 2, n)
    m = (rng.integers(0, 1 << 10, n) << 13) | 0x1FFF
    bits = (np.uint32(127) + e.astype(np.int64) + int(np.floor(np.log2(scale)))).astype(np.uint32) << 23
    vals = (bits | m.astype(np.uint32)).view(np.float32)
    return np.where(rng.random(n) < 0.5, -vals, vals).astype(np.float32)


@pytest.mark.parametrize("d", [32, 64, 128, 256])
def test_tf32_product_within_c_screen(d):
    rng = np.random.default_rng(d)
    K = (d + 31) // 32 * 32
    c = c_screen(K)
    worst = 0.0
    for trial in range(200):
        if trial % 2:
            u = worst_mantissa(rng, d, 1.0)
            v = worst_mantissa(rng, d, 8.0)
            v = np.abs(v) * np.sign(u)  # every product positive: no cancellation of the truncation errors
        else:
            u = rng.standard_normal(d).astype(np.float32)
            v = (rng.standard_normal(d) * 10).astype(np.float32)
        exact = float(np.dot(u.astype(np.float64), v.astype(np.float64)))
        bound = c * float(np.linalg.norm(u.astype(np.float64))) * float(np.linalg.norm(v.astype(np.float64)))
        for rev in (False, True):
            a = fp32_dot(tf32(u), tf32(v), rev)
            err = abs(a - exact)
            assert err <= bound, (d, trial, err, bound)
            worst = max(worst, err / bound)
    # the bound is not vacuous: same-signed worst-case mantissas reach about
    # half of its undoubled value
    assert worst > 0.2, worst


def test_insert_screen_E_covers_bias_rounding():
    """s~ = fl32(a + b) against the exact s = u.v + b, with the kernel's
    E = c wmax hn + 2^-22 Mb (Mb = (1 + c) wmax hn + max |b|)."""
    rng = np.random.default_rng(7)
    d, C = 128, 200
    c = c_screen(128)
    W = (rng.standard_normal((C, d)) / np.sqrt(d)).astype(np.float32)
    b = (rng.standard_normal(C) * 4).astype(np.float32)
    wmax = float(np.linalg.norm(W.astype(np.float64), axis=1).max())
    bmax = float(np.abs(b).max())
    for _ in range(20):
        z = (rng.standard_normal(d) * 3).astype(np.float32)
        hn = float(np.linalg.norm(z.astype(np.float64)))
        Mb = (1 + c) * wmax * hn + bmax
        E = c * wmax * hn + 2.0 ** -22 * Mb
        Wt, zt = tf32(W), tf32(z)
        for j in range(C):
            a = np.float32(fp32_dot(Wt[j], zt))
            s_tilde = float(np.float32(a + b[j]))
            s = float(np.dot(W[j].astype(np.float64), z.astype(np.float64))) + float(b[j])
            assert abs(s_tilde - s) <= E


def test_c_screen_magnitude():
    """c is twice the TF32 product error 2^-9, plus small accumulation terms."""
    assert 2 * 2.0 ** -9 < c_screen(128) < 2 * 2.0 ** -9 * 1.05


# ---------------------------------------------------------------------------
# The tensor insert kernel's candidate screen for the tight radius (Eq. 29),
# emulated in FP64 (its directed roundings only widen the tests): for screen
# values s~ with |s~ - s| <= E, the classes it keeps must contain y^G and the
# minimiser of Eq. 29, so that refining them gives the oracle's y^G and r*.

def pair_tables(W):
    """FP64 pair norms and the kernel's bracket-table bounds: ipn (1/||W_y -
    W_j||, +inf for equal rows, as the bracket tables hold), ipn_min(y) over
    rows that differ from W_y (0 when none), ipn_max(y) over every j != y."""
    C = W.shape[0]
    pn = np.linalg.norm(W[:, None, :] - W[None, :, :], axis=2)
    with np.errstate(divide="ignore"):
        ipn = np.where(pn > 0, 1.0 / np.where(pn > 0, pn, 1.0), np.inf)
    ipn_min = np.zeros(C)
    ipn_max = np.zeros(C)
    for y in range(C):
        others = [j for j in range(C) if j != y]
        nz = [ipn[y, j] for j in others if pn[y, j] > 0]
        ipn_min[y] = min(nz) if nz else 0.0
        ipn_max[y] = max(ipn[y, j] for j in others)
    return pn, ipn, ipn_min, ipn_max


def top2_lowest(v):
    """Top two of v with the lowest index winning ties (the kernel's merges)."""
    order = sorted(range(len(v)), key=lambda c: (-v[c], c))
    return order[0], order[1]


def screen_tight(st, E, ipn, ipn_min, ipn_max):
    """Candidate classes of the tight screen, in the kernel's order of tests."""
    C = len(st)
    y1, y2 = top2_lowest(st)
    l1, l2 = st[y1], st[y2]
    lo1, hi1, lo2, hi2 = l1 - E, l1 + E, l2 - E, l2 + E
    h = st + E
    first = (hi1 - lo2) * ipn[y1, y2]
    with np.errstate(invalid="ignore"):
        if hi2 < lo1:  # y1 is certainly y^G
            crude = (lo1 - h) * ipn_min[y1] <= first
            exact = (lo1 - h) * ipn[y1] <= first
            cand = crude & exact
            cand[y1] = True
            return np.flatnonzero(cand), y1
        second = (hi2 - lo1) * ipn_max[y1]  # NaN (0 x inf) is dropped, as fmaxf does
        U = np.fmax(first, second)
        # any y^G has s >= s_y1 >= lo_1: lo_1 bounds it from below
        imA = ipn_min.min()
        cand = (lo1 - h) * imA <= U
    return np.flatnonzero(cand), None


def refine(s, cand, pn, certain_y):
    """y^G (largest refined candidate, lowest index on ties) and Eq. 29 over
    the candidates (equal rows skipped)."""
    y = certain_y if certain_y is not None else min(cand, key=lambda c: (-s[c], c))
    terms = [(s[y] - s[j]) / pn[y, j] for j in cand if j != y and pn[y, j] > 0]
    return y, min(terms) if terms else np.inf


def oracle_tight(s, pn):
    y = top2_lowest(s)[0]
    terms = [(s[y] - s[j]) / pn[y, j] for j in range(len(s)) if j != y and pn[y, j] > 0]
    return y, min(terms) if terms else np.inf


@pytest.mark.parametrize("seed", range(6))
def test_tight_screen_keeps_the_minimiser(seed):
    rng = np.random.default_rng(100 + seed)
    n_unc = 0
    for trial in range(300):
        C = int(rng.integers(3, 14))
        d = int(rng.integers(2, 7))
        W = rng.standard_normal((C, d))
        b = rng.standard_normal(C) * 0.3
        if trial % 3 == 0:  # duplicated head rows (zero pair norms)
            g, k = sorted(rng.choice(C, 2, replace=False))
            W[k] = W[g]
            if trial % 2:
                b[k] = b[g]
        pn, ipn, ipn_min, ipn_max = pair_tables(W)
        z = rng.standard_normal(d)
        s = W @ z + b
        spread = float(np.ptp(s)) + 1e-3
        E = spread * float(rng.choice([1e-4, 1e-2, 0.1, 0.5]))
        mode = trial % 4
        if mode == 0:
            e = rng.uniform(-E, E, C)
        elif mode == 1:
            e = rng.choice([-E, E], C)
        elif mode == 2:  # push the true argmax down and the rest up
            e = np.full(C, E)
            e[top2_lowest(s)[0]] = -E
        else:
            e = -np.sign(s - s.mean()) * E
        st = s + e
        cand, certain = screen_tight(st, E, ipn, ipn_min, ipn_max)
        n_unc += certain is None
        y_ref, r_ref = oracle_tight(s, pn)
        assert y_ref in cand, (seed, trial)
        y, r = refine(s, cand, pn, certain)
        assert y == y_ref, (seed, trial, y, y_ref)
        assert r == r_ref, (seed, trial, r, r_ref)
    assert n_unc > 20, n_unc  # the union test is exercised


def test_tight_screen_nan_bound_case():
    """Uncertain row with hi_2 = lo_1 exactly and a class g equal to y1 (W and b):
    the second term of U* is 0 x inf = NaN and dropped. g can then be y^G only
    by tying y1, and its Eq. 29 term against y2 has the pair norm ||W_y1 - W_y2||,
    so the first term still bounds r*(g): the screen keeps what Eq. 29 needs."""
    # dyadic values, so every sum below is exact
    W = np.array([[1.0, 0.0], [0.25, 0.75], [0.25, 0.75], [-0.5, 0.5], [1.0, -0.75]])
    b = np.array([0.0, 0.125, 0.125, -0.25, 0.0])
    z = np.array([0.5, 1.0])
    s = W @ z + b  # [0.5, 1, 1, 0, -0.25]: classes 1 and 2 are equal and on top
    g, k, m = 1, 2, 0
    E = 0.25
    st = s - E
    st[k] = s[k] + E  # y1 = 2
    st[m] = s[m] + E
    assert st[g] == st[m]  # g ties y2 = 0 on the screen and loses on the index
    assert np.all(np.abs(st - s) <= E)
    pn, ipn, ipn_min, ipn_max = pair_tables(W)
    y1, y2 = top2_lowest(st)
    assert (y1, y2) == (k, m)
    hi2, lo1 = st[y2] + E, st[y1] - E
    assert hi2 == lo1 and np.isinf(ipn_max[y1])
    cand, certain = screen_tight(st, E, ipn, ipn_min, ipn_max)
    assert certain is None
    y_ref, r_ref = oracle_tight(s, pn)
    assert y_ref == g
    y, r = refine(s, cand, pn, None)
    assert (y, r) == (y_ref, r_ref)


def test_tight_screen_needs_the_second_term():
    """Uncertain row whose true y^G (class 2) is neither screen winner, with the
    Eq. 29 minimiser a far class (3): its term needs U* = (hi_2 - lo_1)
    ipn_max(y1) (here 3.33 against 2 for u_{y2}(y1)); without that term the
    screen drops class 3 and the refined r* (3.33) exceeds the true one (3.125).
    Rows: y1, y2 one apart, class 2 at 0.6 from both, class 3 at 4 from class 2
    (the largest pair norm, so the head's smallest ipn is 1/4); E = 1."""
    h = np.sqrt(0.6 ** 2 - 0.25)
    W = np.array([[-0.5, 0.0], [0.5, 0.0], [0.0, h], [0.0, h - 4.0]])
    s = np.array([-1.0, -1.0, 1.0, -11.5])  # exact logits (b absorbs W z)
    E = 1.0
    st = np.array([0.0, 0.0, 0.0, -12.5])  # every |s~ - s| <= E
    assert np.all(np.abs(st - s) <= E)
    pn, ipn, ipn_min, ipn_max = pair_tables(W)
    assert np.isclose(pn.max(), 4.0) and np.isclose(pn[2, 3], 4.0)
    y_ref, r_ref = oracle_tight(s, pn)
    assert y_ref == 2 and np.isclose(r_ref, 12.5 / 4.0)
    cand, certain = screen_tight(st, E, ipn, ipn_min, ipn_max)
    assert certain is None and 3 in cand
    assert refine(s, cand, pn, None) == (y_ref, r_ref)
    # the first term alone would not keep class 3
    lo = -1.0
    assert (lo - (st[3] + E)) * ipn_min.min() > (2.0 * E) * ipn[0, 1]


def test_tight_screen_lower_end_is_tight():
    """The union test's lower end lo_1 is the best the screen allows: a true
    y^G can sit exactly at lo_1 (its logit equal to s_y1 = lo_1), and then a
    lower end above lo_1 would drop a minimiser the oracle needs. Row: y1 and
    the true y^G tie at lo_1 (y1 read E too high), the minimiser j far below."""
    W = np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 1.0], [-3.0, 0.0]])
    s = np.array([1.0, 1.0, 0.5, -6.0])  # classes 0 and 1 tie on top
    E = 0.5
    st = np.array([1.5, 1.0, 0.5, -5.5])  # |s~ - s| <= E; y1 = 0 with lo_1 = 1.0 = s_0
    assert np.all(np.abs(st - s) <= E)
    pn, ipn, ipn_min, ipn_max = pair_tables(W)
    cand, certain = screen_tight(st, E, ipn, ipn_min, ipn_max)
    y_ref, r_ref = oracle_tight(s, pn)
    assert y_ref in cand
    assert refine(s, cand, pn, certain) == (y_ref, r_ref)
    y1 = top2_lowest(st)[0]
    assert st[y1] - E == s[y_ref]  # the bound is attained


# ---------------------------------------------------------------------------
# The probe's separable screen: a pair is kept iff fl(a - tau_k) >= kappa_q,
# with kappa_q = RD((1 - c) |q|~^2 / 2), tau_k = RD((RD(1 - c) |k|~^2 -
# RU(rr_k / (1 - gamma))) / 2) (|.|~^2 the FP32 norms) and a the TF32 product;
# the recheck accepts iff the canonical FP32 squared distance is below rr_k.
# Every pair the recheck would accept must pass the screen.

def f32_rd(x):
    f = np.float32(x)
    return f if float(f) <= x else np.nextafter(f, np.float32(-np.inf))


def f32_ru(x):
    f = np.float32(x)
    return f if float(f) >= x else np.nextafter(f, np.float32(np.inf))


def fp32_sumsq(x):
    acc = np.float32(0.0)
    for v in x.astype(np.float32):
        acc = np.float32(float(acc) + float(v) * float(v))  # one rounding: a fused multiply-add
    return acc


def dist2_canonical(q, k):
    """32-wide fused multiply-add chains of the rounded differences, chunk sums
    added in order (the recheck's canonical distance)."""
    total = np.float32(0.0)
    for c in range(0, len(q), 32):
        p = np.float32(0.0)
        for j in range(c, c + 32):
            e = np.float32(np.float32(q[j]) - np.float32(k[j]))
            p = np.float32(float(p) + float(e) * float(e))
        total = np.float32(total + p)
    return total


@pytest.mark.parametrize("d", [16, 64, 128, 256])
def test_probe_screen_keeps_every_acceptable_pair(d):
    dpad = (d + 31) // 32 * 32
    c = c_screen(dpad)
    om_c_rd = np.nextafter(np.float32(1.0 - c), np.float32(0.0))
    inv_omg_ru = np.nextafter(np.float32(1.0 / (1.0 - gamma32(dpad // 32 + 33))), np.float32(2.0))
    rng = np.random.default_rng(1000 + d)
    tightest = np.inf
    for trial in range(120):
        q = np.zeros(dpad, np.float32)
        k = np.zeros(dpad, np.float32)
        scale = float(rng.choice([1e-3, 1.0, 37.0]))
        k[:d] = np.abs(worst_mantissa(rng, d, scale))  # every product of one sign
        if trial % 3 == 0:
            q[:d] = k[:d]  # distance zero
        elif trial % 3 == 1:  # a near neighbour, also with dropped bits all ones
            w = np.abs(worst_mantissa(rng, d, scale))
            near = (k[:d] + np.float32(0.01) * (w - k[:d])).astype(np.float32)
            q[:d] = (near.view(np.uint32) | np.uint32(0x1FFF)).view(np.float32)
        else:  # a different norm: the AM-GM step is loose there
            q[:d] = (k[:d] * np.float32(rng.uniform(0.5, 2.0))).astype(np.float32)
        d2 = dist2_canonical(q, k)
        rr = np.nextafter(d2, np.float32(np.inf))  # the pair is accepted just barely
        kn, qn = fp32_sumsq(k), fp32_sumsq(q)
        tau = np.float32(float(f32_rd(float(f32_rd(float(om_c_rd) * float(kn))) -
                                      float(f32_ru(float(rr) * float(inv_omg_ru))))) * 0.5)
        kappa = f32_rd((1.0 - c) * float(qn) * 0.5)
        qk = float(np.linalg.norm(q.astype(np.float64)) * np.linalg.norm(k.astype(np.float64)))
        for rev in (False, True):
            a = np.float32(fp32_dot(tf32(q), tf32(k), rev))
            kept = np.float32(a - tau) >= kappa
            assert d2 < rr and kept, (d, trial, rev)
            tightest = min(tightest, (float(np.float32(a - tau)) - float(kappa)) / (c * qk))
    # not vacuous: the worst case uses a good part of the slack c |q| |k|
    assert 0.0 <= tightest < 0.8, tightest


@pytest.mark.parametrize("seed", range(4))
def test_conservative_screen_keeps_the_top_two(seed):
    """Conservative radius: with l2 the second-largest screen value, the
    candidates s~_c >= T = l2 - 2E hold both classes of the true top two (so
    the refined y^G, runner-up and margin of Eq. 20 are exact), on screen
    errors of up to E in the adversarial directions."""
    rng = np.random.default_rng(300 + seed)
    for trial in range(500):
        C = int(rng.integers(2, 40))
        s = rng.standard_normal(C) * float(rng.choice([0.01, 1.0, 100.0]))
        if trial % 5 == 0:
            s[rng.integers(C)] = s.max()  # a tie at the top
        E = (float(np.ptp(s)) + 1e-9) * float(rng.choice([1e-3, 0.05, 0.3]))
        top = sorted(range(C), key=lambda c: (-s[c], c))[:2]
        e = rng.choice([-E, E], C)
        e[top] = -E  # push the true top two down ...
        e[[c for c in range(C) if c not in top]] = E  # ... and every other class up
        if trial % 2:
            e = rng.uniform(-E, E, C)
        st = s + e
        l2 = sorted(st)[-2]
        cand = np.flatnonzero(st >= l2 - 2 * E)
        assert set(top) <= set(cand.tolist()), (seed, trial)
        # refining the candidates reproduces y^G and the margin of Eq. 20
        y = min(cand, key=lambda c: (-s[c], c))
        runner = max(s[c] for c in cand if c != y)
        ys = top2_lowest(s)[0]
        assert y == ys and runner == max(s[c] for c in range(C) if c != ys)


@pytest.mark.parametrize("d", [32, 128, 256])
def test_insert_screen_E_worst_case(d):
    """E on the worst inputs: head rows and features whose dropped bits are all
    ones, every product of one sign, FP32 sums in either order, biases of
    either sign; the worst error uses a good part of E."""
    rng = np.random.default_rng(40 + d)
    K = (d + 31) // 32 * 32
    c = c_screen(K)
    C = 24
    z = np.abs(worst_mantissa(rng, d, 2.0))
    W = np.abs(np.stack([worst_mantissa(rng, d, float(rng.choice([0.05, 1.0]))) for _ in range(C)]))
    b = (rng.standard_normal(C) * float(np.abs(W @ z).mean())).astype(np.float32)
    wmax = float(np.linalg.norm(W.astype(np.float64), axis=1).max())
    hn = float(np.linalg.norm(z.astype(np.float64)))
    Mb = (1 + c) * wmax * hn + float(np.abs(b).max())
    E = c * wmax * hn + 2.0 ** -22 * Mb
    worst = 0.0
    for j in range(C):
        s = float(np.dot(W[j].astype(np.float64), z.astype(np.float64))) + float(b[j])
        for rev in (False, True):
            a = np.float32(fp32_dot(tf32(W[j]), tf32(z), rev))
            err = abs(float(np.float32(a + b[j])) - s)
            assert err <= E, (d, j, err, E)
            worst = max(worst, err / E)
    assert worst > 0.1, worst


def test_probe_chunk_pretest_never_drops_a_kept_pair():
    """The probe tests each 32-key chunk with fl(max a - min tau) >= kappa before
    the per-pair test fl(a_j - tau_j) >= kappa: rounding to nearest is monotone,
    so a chunk holding a kept pair always passes."""
    rng = np.random.default_rng(77)
    for trial in range(3000):
        scale = float(rng.choice([1e-3, 1.0, 1e4]))
        a = (rng.standard_normal(32) * scale).astype(np.float32)
        tau = (rng.standard_normal(32) * scale).astype(np.float32)
        kept = (a - tau).astype(np.float32)
        kappa = np.float32(kept.max()) if trial % 2 else np.float32(rng.choice(kept))
        if trial % 3 == 0:
            kappa = np.nextafter(kappa, np.float32(-np.inf))
        assert np.any(kept >= kappa)
        assert np.float32(a.max() - tau.min()) >= kappa, trial


# ---------------------------------------------------------------- compensated refinement (Dot2) bound
# The certify kernels refine candidate logits with a compensated dot product
# (Ogita, Rump and Oishi's Dot2: TwoProduct by FMA, TwoSum accumulation, the
# error terms summed in plain FP32) evaluated as L lane chains of n features
# each, a butterfly over the L lanes, then the bias. Its bound, used for the
# certified radius lower bound and for sending rows to the FP64 pass, is
# |hi + lo - exact| <= G (sum |w z| + |b|), G = gamma_D u (n + log2 L + 2),
# D = n + 2 log2 L + 2 (dot2_factor in certify.cu). Emulated here in FP32 with
# round-to-nearest, against exact sums.

def dot2_factor(n, L):
    lg = 0
    while (1 << lg) < L:
        lg += 1
    return gamma32(n + 2 * lg + 2) * U32 * (n + lg + 2) * (1.0 + 1e-3)


def f32(x):
    return np.float32(x)


def two_sum(a, b):
    s = f32(a + b)
    bb = f32(s - a)
    return s, f32(f32(a - f32(s - bb)) + f32(b - bb))


def dot2_lanes(w, z, b, L):
    """The kernels' evaluation order: lane l takes features l, l + L, ...;
    lanes combined by xor butterfly; then the bias and a final TwoSum."""
    d = len(w)
    P = [f32(0)] * L
    Cc = [f32(0)] * L
    for l in range(L):
        p, c = f32(0), f32(0)
        for j in range(l, d, L):
            pr = f32(w[j] * z[j])
            er = f32(float(w[j]) * float(z[j]) - float(pr))  # exact: the FMA's TwoProduct error
            t, q = two_sum(p, pr)
            p = t
            c = f32(c + f32(q + er))
        P[l], Cc[l] = p, c
    o = L // 2
    while o > 0:
        NP, NC = list(P), list(Cc)
        for l in range(L):
            t, q = two_sum(P[l], P[l ^ o])
            NP[l] = t
            NC[l] = f32(f32(Cc[l] + Cc[l ^ o]) + q)
        P, Cc = NP, NC
        o //= 2
    t, q = two_sum(P[0], f32(b))
    hi, lo = two_sum(t, f32(Cc[0] + q))
    return float(hi) + float(lo)  # exact in FP64: lo is at most half an ulp of hi


def exact_dot(w, z, b):
    from fractions import Fraction
    return sum((Fraction(float(x)) * Fraction(float(y)) for x, y in zip(w, z)), Fraction(float(b)))


@pytest.mark.parametrize("d,L", [(128, 8), (256, 8), (48, 8), (128, 32), (64, 1)])
def test_dot2_refinement_bound(d, L):
    from fractions import Fraction
    rng = np.random.default_rng(d * 7 + L)
    G = dot2_factor((d + L - 1) // L, L)
    worst = 0.0
    for trial in range(60):
        kind = trial % 3
        z = rng.standard_normal(d).astype(np.float32) * 3
        w = rng.standard_normal(d).astype(np.float32) / np.sqrt(d)
        if kind == 1:  # heavy cancellation: w nearly orthogonal to z
            w64 = w.astype(np.float64) - (w.astype(np.float64) @ z.astype(np.float64)) / (z @ z) * z.astype(np.float64)
            w = w64.astype(np.float32)
        elif kind == 2:  # features over a wide exponent range
            w = (w * np.exp2(rng.integers(-20, 20, d))).astype(np.float32)
        b = np.float32(0.1 * rng.standard_normal())
        got = dot2_lanes(w, z, b, L)
        ex = exact_dot(w, z, b)
        err = abs(Fraction(got) - ex)
        scale = float(np.sum(np.abs(w.astype(np.float64) * z.astype(np.float64)))) + abs(float(b))
        assert err <= Fraction(G * scale), (d, L, trial, float(err), G * scale)
        worst = max(worst, float(err) / (G * scale))
    assert worst < 1.0


def test_dot2_factor_is_tighter_than_the_sequential_bound():
    # 8-lane groups over d = 128: chains of 16 features; about 1e-12, some
    # hundred times below 2 gamma_{d+40}^2
    g8 = dot2_factor(16, 8)
    assert 1e-12 < g8 < 3e-12
    assert g8 * 50 < 2 * gamma32(168) ** 2
    # one lane over every feature: about (d u)^2
    assert dot2_factor(128, 1) > (128 * U32) ** 2
