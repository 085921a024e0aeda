"""Pins of the oracle's Eq. 1 sums and cosine for binary64 regions.

The sums of binary64 products are checked against exact rational
arithmetic (fractions.Fraction) over the same index sets, then rounded to
the nearest double; the rounding edges (gradual underflow, ties, overflow)
against values worked out by hand; the cosine against the properties that
fix it: invariance under power-of-two scaling of either vector, agreement
with the plain formula where that one stays in range, and +-1 for parallel
vectors.
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

DBL_MAX = float.fromhex("0x1.fffffffffffffp+1023")
TINY = 2.0 ** -1074


def _bits(x):
    return struct.unpack("<q", struct.pack("<d", x))[0]


def _fraction_sums(r, c):
    """S_rc over pairs with both values finite, S_rr over finite r, S_cc
    over finite c, exactly."""
    s_rc = s_rr = s_cc = Fraction(0)
    for a, b in zip(r.tolist(), c.tolist()):
        fa, fb = math.isfinite(a), math.isfinite(b)
        if fa and fb:
            s_rc += Fraction(a) * Fraction(b)
        if fa:
            s_rr += Fraction(a) * Fraction(a)
        if fb:
            s_cc += Fraction(b) * Fraction(b)
    return s_rc, s_rr, s_cc


def _round(f):
    """A rational rounded to the nearest double, ties to even; infinity
    past the largest finite double's rounding boundary."""
    try:
        return float(f)
    except OverflowError:
        return math.inf if f > 0 else -math.inf


def _sums(o, r, c, threads=1):
    r = np.ascontiguousarray(r, np.float64)
    c = np.ascontiguousarray(c, np.float64)
    return o.eq_sums(r.view(np.uint8), c.view(np.uint8), o.F64, r.size, threads=threads)


def _values(kind, n, rng):
    sign = np.where(rng.random(n) < 0.5, -1.0, 1.0)
    mant = rng.uniform(1.0, 2.0, n)
    if kind == "normal":
        return rng.standard_normal(n)
    if kind == "full_range":
        v = sign * np.ldexp(mant, rng.integers(-1074, 1024, n))
    elif kind == "tiny":
        v = sign * np.ldexp(mant, rng.integers(-1074, -1000, n))
    elif kind == "huge":
        v = sign * np.ldexp(mant, rng.integers(500, 1024, n))
    else:
        raise ValueError(kind)
    v[rng.random(n) < 0.03] = 0.0
    return v


@pytest.mark.parametrize("kind", ["normal", "full_range", "tiny", "huge"])
def test_sums_are_correctly_rounded_exact_sums(oracle, kind):
    rng = np.random.default_rng({"normal": 1, "full_range": 2, "tiny": 3, "huge": 4}[kind])
    n = 300
    r = _values(kind, n, rng)
    # candidates: a few ULP away, an unrelated vector, and one with specials
    cands = [r * (1.0 + rng.integers(-4, 5, n) * 2.0 ** -52), _values(kind, n, rng)]
    sp = r.copy()
    sp[[3, 50, 51]] = [math.inf, math.nan, -math.inf]
    cands.append(sp)
    for c in cands:
        got = _sums(oracle, r, c)
        want = [_round(s) for s in _fraction_sums(r, c)]
        for key, w in zip(("sum_rc", "sum_rr", "sum_cc"), want):
            assert _bits(got[key]) == _bits(w), (kind, key, got[key], w)


def test_reference_specials_leave_its_sums(oracle):
    rng = np.random.default_rng(5)
    r = rng.standard_normal(64)
    c = r.copy()
    r[[1, 9]] = [math.nan, -math.inf]
    c[[9, 20]] = [1.0, math.inf]
    got = _sums(oracle, r, c)
    want = [_round(s) for s in _fraction_sums(r, c)]
    assert [got["sum_rc"], got["sum_rr"], got["sum_cc"]] == want


def test_split_over_threads_is_the_same(oracle):
    rng = np.random.default_rng(6)
    r = _values("full_range", 5000, rng)
    c = _values("full_range", 5000, rng)
    a, b = _sums(oracle, r, c, threads=1), _sums(oracle, r, c, threads=7)
    for key in ("sum_rc", "sum_rr", "sum_cc", "cos"):
        assert _bits(a[key]) == _bits(b[key])


@pytest.mark.parametrize("r,c,want_rc", [
    ([TINY], [TINY], 0.0),                                   # 2^-2148: far below the subnormals
    ([2.0 ** -537], [2.0 ** -537], TINY),                   # exactly the least subnormal
    ([2.0 ** -537], [2.0 ** -538], 0.0),                    # 2^-1075: a tie, to even (zero)
    ([2.0 ** -537, 2.0 ** -550], [2.0 ** -538, 2.0 ** -550], TINY),   # tie + sticky: up
    ([3.0 * 2.0 ** -538], [2.0 ** -538], TINY),             # 0.75 of the least subnormal: up
    ([2.0 ** 512], [DBL_MAX / 2.0 ** 512], DBL_MAX),         # the largest double exactly
    ([2.0 ** 512, 2.0 ** 485], [DBL_MAX / 2.0 ** 512, 2.0 ** 484], DBL_MAX),   # below the midpoint
    ([2.0 ** 512, 2.0 ** 485], [DBL_MAX / 2.0 ** 512, 2.0 ** 485], math.inf),  # the midpoint: to even
    ([2.0 ** 1023], [-(2.0 ** 1023)], -math.inf),
    ([1.0, -1.0], [2.0 ** -1074, 2.0 ** -1074], 0.0),        # exact cancellation
])
def test_rounding_edges_worked_by_hand(oracle, r, c, want_rc):
    got = _sums(oracle, np.array(r), np.array(c))
    assert _bits(got["sum_rc"]) == _bits(want_rc), (got["sum_rc"], want_rc)


def test_squares_overflow_but_the_cosine_does_not(oracle):
    r = np.array([2.0 ** 1023, -(2.0 ** 1000), 3.0 * 2.0 ** 990])
    got = _sums(oracle, r, r)
    assert got["sum_rr"] == math.inf and got["sum_cc"] == math.inf and got["sum_rc"] == math.inf
    assert abs(got["cos"] - 1.0) <= 4 * 2.0 ** -53
    neg = _sums(oracle, r, -r)
    assert neg["sum_rc"] == -math.inf and abs(neg["cos"] + 1.0) <= 4 * 2.0 ** -53


def test_squares_underflow_but_the_cosine_does_not(oracle):
    rng = np.random.default_rng(8)
    r = np.ldexp(rng.uniform(1.0, 2.0, 50), -600)
    c = r * (1.0 + rng.integers(-3, 4, 50) * 2.0 ** -52)
    got = _sums(oracle, r, c)
    assert got["sum_rr"] == 0.0 and got["sum_cc"] == 0.0
    assert 0.9999999 < got["cos"] <= 1.0 + 4 * 2.0 ** -53


@pytest.mark.parametrize("kr,kc", [(900, 0), (-900, 0), (600, -700), (-1000, 1000), (1, 1)])
def test_cosine_is_invariant_under_power_of_two_scaling(oracle, kr, kc):
    rng = np.random.default_rng(9)
    r = rng.standard_normal(400)
    c = r + 1e-3 * rng.standard_normal(400)
    base = _sums(oracle, r, c)["cos"]
    scaled = _sums(oracle, np.ldexp(r, kr), np.ldexp(c, kc))["cos"]
    assert _bits(base) == _bits(scaled), (base, scaled)


@pytest.mark.parametrize("seed", [10, 11, 12])
def test_cosine_is_the_plain_formula_inside_the_double_range(oracle, seed):
    rng = np.random.default_rng(seed)
    r = rng.standard_normal(500) * 1e3
    c = rng.standard_normal(500) * 1e-3 + (r if seed != 12 else 0.0)
    got = _sums(oracle, r, c)
    s_rc, s_rr, s_cc = (_round(s) for s in _fraction_sums(r, c))
    plain = s_rc / (math.sqrt(s_rr) * math.sqrt(s_cc))
    assert _bits(got["cos"]) == _bits(plain)


def test_zero_vectors(oracle):
    z = np.zeros(10)
    one = np.ones(10)
    assert _sums(oracle, z, z)["cos"] == 1.0
    assert _sums(oracle, z, one)["cos"] == 0.0
    assert _sums(oracle, one, z)["cos"] == 0.0
    assert _sums(oracle, np.array([TINY]), np.array([TINY]))["cos"] == 1.0   # sums 2^-2148, not 0


def test_verdict_uses_the_scaled_cosine(oracle):
    r = np.array([2.0 ** 1020, 2.0 ** 1019])
    sums = _sums(oracle, r, r)
    stats = {"mismatches": 0, "max_abs_err": 0.0, "nonfinite_mismatches": 0, "guard_bad_bytes": 0}
    v = oracle.eq_verdict(stats, sums, oracle.F64)
    assert v["eq"] == 1 and v["cos"] == sums["cos"]
