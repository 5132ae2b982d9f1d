"""The certify kernels' compensated refinement (Dot2 of Ogita, Rump and
Oishi: TwoProduct and TwoSum per feature, then the bias) computed in two
layouts must give the same bits, emulated here in FP32 on the CPU.

Group layout (every FP32 certify kernel, and the tensor kernel's one-warp
paths): eight lanes share one (row, class) pair; lane s runs the chain over
the features k = s, s + 8, s + 16, ... in ascending order, the eight chains
are combined by a butterfly over the group (xor 4, 2, 1: TwoSum of the two
partial sums, the compensation terms added, then the TwoSum error), and the
bias is added last.

Lane layout (the tensor kernel's candidate list): one lane takes the whole
pair and runs the same eight chains side by side, then combines them in the
butterfly's tree inside the lane: (0,4) (1,5) (2,6) (3,7), then (0,2)
(1,3), then (0,1). For the last few pairs of a list, two lanes share a pair
(lane t: chains 4t..4t+3, the first level across the two lanes) or four do
(lane t: chains t and t+4, the first level in the lane, the others across).

The layouts agree because TwoSum's error term is the exact rounding error of
the sum whichever operand comes first, and FP32 addition is commutative, so
every lane of the group holds the same pair after each level. These tests
check that, and that the group's eight lanes agree, on random, cancelling
and sign-mixed inputs, with d from 16 to 256. The last test checks the
first screening pass's update of the top two s~ of a chunk, two values at a
time, against the one-at-a-time tracker.
"""
import numpy as np
import pytest

f32 = np.float32


def _add(a, b):
    return (a + b).astype(f32)


def _sub(a, b):
    return (a - b).astype(f32)


def _two_sum(a, b):
    s = _add(a, b)
    bb = _sub(s, a)
    e = _add(_sub(a, _sub(s, bb)), _sub(b, bb))
    return s, e


def _two_prod(w, x):
    pr = (w * x).astype(f32)
    # fma(w, x, -pr): the product of two FP32 values is exact in FP64 and its
    # rounding error is an FP32 value, so one rounding of the FP64 difference
    # is the fused result
    er = (w.astype(np.float64) * x.astype(np.float64) - pr.astype(np.float64)).astype(f32)
    return pr, er


def _chains(W, Z):
    """The eight per-residue chains (P, CC) of every pair: W, Z (n, d) FP32."""
    n, d = W.shape
    P = np.zeros((8, n), f32)
    CC = np.zeros((8, n), f32)
    for s in range(8):
        for k in range(s, d, 8):
            pr, er = _two_prod(W[:, k], Z[:, k])
            sm = _add(P[s], pr)
            bb = _sub(sm, P[s])
            q = _add(_sub(P[s], _sub(sm, bb)), _sub(pr, bb))
            P[s] = sm
            CC[s] = _add(CC[s], _add(q, er))
    return P, CC


def _finish(p, cc, bias):
    t, q = _two_sum(p, bias)
    return _two_sum(t, _add(cc, q))


def refine_group(W, Z, bias):
    """Eight lanes, butterfly by shuffles: returns every lane's (hi, lo)."""
    P, CC = _chains(W, Z)
    p, cc = P.copy(), CC.copy()
    for o in (4, 2, 1):
        pn, ccn = np.empty_like(p), np.empty_like(cc)
        for s in range(8):
            t, q = _two_sum(p[s], p[s ^ o])        # own value first, then the partner's
            pn[s] = t
            ccn[s] = _add(_add(cc[s], cc[s ^ o]), q)
        p, cc = pn, ccn
    return [_finish(p[s], cc[s], bias) for s in range(8)]


def refine_lane(W, Z, bias):
    """One lane, the same tree inside the lane."""
    P, CC = _chains(W, Z)
    p, cc = list(P), list(CC)
    for o in (4, 2, 1):
        for s in range(o):
            t, q = _two_sum(p[s], p[s + o])
            cc[s] = _add(_add(cc[s], cc[s + o]), q)
            p[s] = t
    return _finish(p[0], cc[0], bias)


def refine_split(W, Z, bias, K):
    """K lanes per pair: returns every lane's (hi, lo); each lane combines its
    own value first, as the kernel does."""
    P, CC = _chains(W, Z)
    if K == 2:
        # lane t holds chains 4t..4t+3 as local 0..3
        lanes = [[list(P[4 * t:4 * t + 4]), list(CC[4 * t:4 * t + 4])] for t in range(2)]
        new = []
        for t in range(2):
            p, cc = [x.copy() for x in lanes[t][0]], [x.copy() for x in lanes[t][1]]
            for j in range(4):
                s_, q = _two_sum(p[j], lanes[t ^ 1][0][j])
                cc[j] = _add(_add(cc[j], lanes[t ^ 1][1][j]), q)
                p[j] = s_
            for a, b in ((0, 2), (1, 3), (0, 1)):
                s_, q = _two_sum(p[a], p[b])
                cc[a] = _add(_add(cc[a], cc[b]), q)
                p[a] = s_
            new.append(_finish(p[0], cc[0], bias))
        return new
    # K == 4: lane t holds chains t and t + 4; first level in the lane
    vals = []
    for t in range(4):
        s_, q = _two_sum(P[t], P[t + 4])
        vals.append((s_, _add(_add(CC[t], CC[t + 4]), q)))
    for o in (2, 1):
        nv = []
        for t in range(4):
            s_, q = _two_sum(vals[t][0], vals[t ^ o][0])
            nv.append((s_, _add(_add(vals[t][1], vals[t ^ o][1]), q)))
        vals = nv
    return [_finish(v[0], v[1], bias) for v in vals]


def _bits(x):
    return np.asarray(x, f32).view(np.uint32)


def _cases(rng, n, d):
    W = rng.standard_normal((n, d)).astype(f32) / f32(np.sqrt(d))
    Z = (rng.standard_normal((n, d)) * 3.0).astype(f32)
    bias = (rng.standard_normal(n) * 0.1).astype(f32)
    # cancelling pairs: the bias nearly cancels the dot product
    m = n // 4
    dots = (W[:m].astype(np.float64) * Z[:m].astype(np.float64)).sum(1)
    bias[:m] = (-dots).astype(f32)
    # features spanning many binades, exact zeros and negative zeros
    Z[m:2 * m] *= (2.0 ** rng.integers(-30, 30, size=(m, d))).astype(f32)
    Z[2 * m:2 * m + m // 2, ::3] = f32(0.0)
    Z[2 * m + m // 2:3 * m, ::5] = f32(-0.0)
    # halves that cancel term by term: exact dot products of zero
    h = d // 2
    W[3 * m:3 * m + 8, h:] = W[3 * m:3 * m + 8, :h]
    Z[3 * m:3 * m + 8, h:] = -Z[3 * m:3 * m + 8, :h]
    bias[3 * m:3 * m + 8] = f32(0.0)
    return W, Z, bias


@pytest.mark.parametrize("d", [16, 32, 48, 64, 128, 256])
def test_lane_layout_matches_group_layout(d):
    rng = np.random.default_rng(1000 + d)
    W, Z, bias = _cases(rng, 4000, d)
    group = refine_group(W, Z, bias)
    hi, lo = refine_lane(W, Z, bias)
    for s in range(8):  # every lane of the group ends with the same pair
        assert np.array_equal(_bits(group[s][0]), _bits(group[0][0])), s
        assert np.array_equal(group[s][1], group[0][1]), s
    assert np.array_equal(_bits(hi), _bits(group[0][0]))
    assert np.array_equal(hi, group[0][0]) and np.array_equal(lo, group[0][1])


@pytest.mark.parametrize("K", [2, 4])
@pytest.mark.parametrize("d", [16, 48, 128])
def test_split_lanes_match_lane_layout(d, K):
    rng = np.random.default_rng(2000 + d + K)
    W, Z, bias = _cases(rng, 3000, d)
    hi, lo = refine_lane(W, Z, bias)
    for h, l in refine_split(W, Z, bias, K):  # every lane of the K
        assert np.array_equal(_bits(h), _bits(hi))
        assert np.array_equal(_bits(l), _bits(lo))


def test_refinement_is_compensated():
    """The emulation itself is Dot2: hi + lo is within a few units of 2^-48
    of the scale of the exact dot product plus bias (a dropped error term or
    a wrong sign in TwoSum would leave FP32-sized errors)."""
    from fractions import Fraction
    rng = np.random.default_rng(7)
    d = 128
    W, Z, bias = _cases(rng, 400, d)
    hi, lo = refine_lane(W, Z, bias)
    worst = 0.0
    for i in range(0, 400, 7):
        exact = sum(Fraction(float(W[i, k])) * Fraction(float(Z[i, k])) for k in range(d)) + Fraction(float(bias[i]))
        got = Fraction(float(hi[i])) + Fraction(float(lo[i]))
        scale = float(np.abs(W[i].astype(np.float64) * Z[i].astype(np.float64)).sum() + abs(float(bias[i])))
        if scale > 0:
            worst = max(worst, abs(float(got - exact)) / scale)
    assert worst < 2.0 ** -40, worst


def _top2_sequential(vals):
    """The first pass's tracker, one value at a time: t2 = max(t2, min(t1, s)),
    t1 = max(t1, s)."""
    t1 = t2 = -np.inf
    for s_ in vals:
        t2 = max(t2, min(t1, s_))
        t1 = max(t1, s_)
    return t1, t2


def _top2_pairs(vals):
    """The tensor kernel's first pass on a full chunk, two values at a time:
    with hi / lo the larger / smaller of the two, t2 = max(t2, min(t1, hi), lo)
    and t1 = max(t1, hi)."""
    t1 = t2 = -np.inf
    for a, b in zip(vals[0::2], vals[1::2]):
        hi, lo = max(a, b), min(a, b)
        t2 = max(t2, min(t1, hi), lo)
        t1 = max(t1, hi)
    return t1, t2


def test_first_pass_pairs_match_sequential_top_two():
    """The two-at-a-time update keeps the same largest and second-largest
    value (ties counted twice) as the one-at-a-time tracker, on random values,
    heavy ties and infinities."""
    rng = np.random.default_rng(11)
    for trial in range(3000):
        n = 2 * int(rng.integers(1, 17))
        kind = trial % 3
        if kind == 0:
            v = rng.standard_normal(n).astype(np.float32)
        elif kind == 1:
            v = rng.integers(-3, 4, size=n).astype(np.float32)  # many exact ties
        else:
            v = rng.standard_normal(n).astype(np.float32)
            v[rng.random(n) < 0.3] = -np.inf
        vals = [float(x) for x in v]
        assert _top2_pairs(vals) == _top2_sequential(vals), vals
        srt = sorted(vals, reverse=True)
        assert _top2_sequential(vals) == (srt[0], srt[1])
