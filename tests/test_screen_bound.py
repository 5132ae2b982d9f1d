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
