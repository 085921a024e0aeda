"""Pins of the oracle's fp32 Box-Muller pieces: ln(u) and sin/cos(2 pi u)
over every one of their 2^24 inputs against exactly-reduced float64
references, the series coefficients against 50-digit arithmetic, and the
normal values against N(0, 1) (moments, Kolmogorov-Smirnov)."""
import numpy as np
import pytest


def _ulp32(x):
    u = np.spacing(np.abs(x).astype(np.float32)).astype(np.float64)
    return np.maximum(u, 2.0 ** -149)


def test_ln_u24_all_inputs(oracle):
    k = np.arange(1, (1 << 24) + 1, dtype=np.uint32)
    got = oracle.ln_u24(k).astype(np.float64)
    want = np.log(k.astype(np.float64) * 2.0 ** -24)
    err = np.abs(got - want) / _ulp32(want)
    assert err.max() <= 2.0, err.max()
    assert got[-1] == 0.0          # ln(1) is exactly zero


def test_sincos_2pi_u24_all_inputs(oracle):
    sp = pytest.importorskip("scipy.special")
    k = np.arange(0, 1 << 24, dtype=np.uint32)
    sn, cs = oracle.sincos_2pi_u24(k)
    deg = 360.0 * k.astype(np.float64) * 2.0 ** -24     # exact in fp64
    rs, rc = sp.sindg(deg), sp.cosdg(deg)
    assert (np.abs(sn - rs) / _ulp32(rs)).max() <= 2.0
    assert (np.abs(cs - rc) / _ulp32(rc)).max() <= 2.0
    q = 1 << 22                    # quarter turns are exact
    assert (sn[0], cs[0]) == (0.0, 1.0)
    assert (sn[q], cs[q]) == (1.0, 0.0)
    assert (sn[2 * q], cs[2 * q]) == (0.0, -1.0)
    assert (sn[3 * q], cs[3 * q]) == (-1.0, 0.0)


def _rn32(mpmath, x):
    """Correctly rounded fp32 of a 50-digit value."""
    f = np.float32(float(x))
    cands = [np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))]
    return min(cands, key=lambda c: abs(mpmath.mpf(float(c)) - x))


def test_series_coefficients_are_correctly_rounded(oracle):
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 50
    c = oracle.boxmuller_consts()
    ln2 = mpmath.log(2)
    assert c[0] == np.float32(355.0 / 512.0)
    assert c[1] == _rn32(mpmath, ln2 - mpmath.mpf(355) / 512)
    assert c[2] == _rn32(mpmath, mpmath.mpf(1) / 3)
    h = mpmath.pi / 2
    for k in range(5):                       # sin: r^1, r^3, ..., r^9
        j = 2 * k + 1
        assert c[3 + k] == _rn32(mpmath, (-1) ** k * h ** j / mpmath.factorial(j))
    for k in range(6):                       # cos: r^0, r^2, ..., r^10
        j = 2 * k
        assert c[8 + k] == _rn32(mpmath, (-1) ** k * h ** j / mpmath.factorial(j))


def test_ln_table_entries_and_exact_reduction(oracle):
    """Each row: inv_j = round(32768/(128+j))/256, head = -ln(inv_j) rounded
    to a multiple of 2^-9, tail = fp32 of the rest; every mantissa of a
    bucket gives |m*inv_j - 1| < 2^-7 (so one fma is exact)."""
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 50
    t = oracle.ln_table()
    for j in range(129):
        I = int(mpmath.nint(mpmath.mpf(32768) / (128 + j)))
        assert t[j, 0] == np.float32(I / 256.0)
        nl = mpmath.log(mpmath.mpf(256) / I)
        hi = mpmath.nint(nl * 512) / 512
        assert t[j, 1] == np.float32(float(hi))
        assert t[j, 2] == _rn32(mpmath, nl - hi)
        lo_m = max(1.0, 1 + (j - 0.5) / 128)
        hi_m = min(2 - 2.0 ** -23, 1 + (j + 0.5) / 128)
        for m in (lo_m, hi_m):
            assert abs(m * float(t[j, 0]) - 1) < 2.0 ** -7
    assert (t[128, 1], t[128, 2]) == (oracle.boxmuller_consts()[0], oracle.boxmuller_consts()[1])


def test_boxmuller_is_standard_normal(oracle):
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(2024)
    n = 1 << 21
    w0 = rng.integers(0, 1 << 32, size=n, dtype=np.uint64).astype(np.uint32)
    w1 = rng.integers(0, 1 << 32, size=n, dtype=np.uint64).astype(np.uint32)
    z0, z1 = oracle.boxmuller(w0, w1)
    z = np.concatenate([z0, z1]).astype(np.float64)
    m = z.size
    assert abs(z.mean()) < 5 / np.sqrt(m)
    assert abs(z.var() - 1.0) < 5 * np.sqrt(2.0 / m)
    assert abs(stats.skew(z)) < 5 * np.sqrt(6.0 / m)
    assert abs(stats.kurtosis(z)) < 5 * np.sqrt(24.0 / m)
    assert stats.kstest(z, "norm").pvalue > 1e-4
    # the pair is independent: correlation ~ 0
    assert abs(np.corrcoef(z0, z1)[0, 1]) < 5 / np.sqrt(n)
    # radius and angle: z0^2 + z1^2 = -2 ln u1 (up to fp32 rounding)
    u1 = ((w0 >> 8).astype(np.float64) + 1) * 2.0 ** -24
    r2 = z0.astype(np.float64) ** 2 + z1.astype(np.float64) ** 2
    np.testing.assert_allclose(r2, -2 * np.log(u1), rtol=3e-6, atol=1e-6)


def test_boxmuller_extreme_inputs(oracle):
    # u1 = 1 gives rho = 0 (both outputs are signed zeros); the smallest u1
    # gives the largest radius sqrt(-2 ln 2^-24) ~ 5.77
    z0, z1 = oracle.boxmuller(np.array([0xFFFFFFFF, 0], np.uint32),
                              np.array([0, 0], np.uint32))
    assert z0[0] == 0.0 and z1[0] == 0.0
    assert abs(z0[1] - np.sqrt(-2 * np.log(2.0 ** -24))) < 1e-5 and z1[1] == 0.0
