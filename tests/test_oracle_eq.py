"""Pins of the oracle's Eq. 1 aggregate terms (the cosine c_x of a float
region and the verdict eq(K', x) of Eq. 1).

The sums S_rc, S_rr, S_cc are pinned to Python's math.fsum (the correctly
rounded sum of exact doubles, Shewchuk's algorithm) over products formed
from values decoded by torch / numpy, to exact rational arithmetic on tiny
inputs, and to closed forms; the verdict to its four terms one at a time.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

torch = pytest.importorskip("torch")

STORAGE = {"F32": (np.float32, None), "BF16": (np.uint16, torch.bfloat16),
           "F16": (np.float16, None), "F8E4M3": (np.uint8, torch.float8_e4m3fn)}


def _decode(raw, name):
    """Values of a payload decoded outside the oracle (fp64)."""
    np_t, torch_t = STORAGE[name]
    if torch_t is None:
        with np.errstate(invalid="ignore"):
            return raw.view(np_t).astype(np.float64)
    return torch.from_numpy(raw.view(np_t).copy()).view(torch_t).to(torch.float64).numpy()


def _random_bits(name, n, rng):
    size = {"F32": 4, "BF16": 2, "F16": 2, "F8E4M3": 1}[name]
    return rng.integers(0, 256, size=n * size, dtype=np.uint8)


def _fsum_terms(r, c):
    fr, fc = np.isfinite(r), np.isfinite(c)
    both = fr & fc
    return (math.fsum((r[both] * c[both]).tolist()), math.fsum((r[fr] * r[fr]).tolist()),
            math.fsum((c[fc] * c[fc]).tolist()))


def _sums(o, ref, cand, name, n, threads=1):
    s = o.eq_sums(ref, cand, getattr(o, name), n, threads=threads)
    return s["sum_rc"], s["sum_rr"], s["sum_cc"]


def _spread_f32(n, rng, lo=-140, hi=126):
    """fp32 values over the whole exponent range, both signs, with zeros
    and subnormals."""
    mant = rng.uniform(1.0, 2.0, n)
    ex = rng.integers(lo, hi, n)
    v = (np.where(rng.random(n) < 0.5, -1.0, 1.0) * np.ldexp(mant, ex)).astype(np.float32)
    v[rng.random(n) < 0.02] = 0.0
    return v


@pytest.mark.parametrize("name", ["F32", "BF16", "F16", "F8E4M3"])
def test_sums_are_correctly_rounded_exact_sums(oracle, name):
    rng = np.random.default_rng(11)
    n = 20000
    ref = _random_bits(name, n, rng)
    cand = _random_bits(name, n, rng)
    if name == "F32":              # random bits give mostly huge/tiny fp32: use a spread too
        ref[: 4 * n // 2] = _spread_f32(n // 2, rng).view(np.uint8)
        cand[: 4 * n // 2] = _spread_f32(n // 2, rng).view(np.uint8)
    got = _sums(oracle, ref, cand, name, n)
    want = _fsum_terms(_decode(ref, name), _decode(cand, name))
    assert got == want


@pytest.mark.parametrize("name", ["F32", "BF16", "F16", "F8E4M3"])
def test_sums_of_near_values(oracle, name):
    """Candidate = reference with a few low bits changed: the regime of a
    real check, where S_rc, S_rr and S_cc nearly agree."""
    rng = np.random.default_rng(12)
    n = 50000
    if name == "F32":
        ref = rng.standard_normal(n).astype(np.float32).view(np.uint8)
    else:
        t = {"BF16": torch.bfloat16, "F16": torch.float16, "F8E4M3": torch.float8_e4m3fn}[name]
        x = torch.from_numpy(rng.standard_normal(n).astype(np.float32)).to(t)
        ref = x.view(torch.uint8).numpy().copy() if name == "F8E4M3" else \
            x.view(torch.int16).numpy().view(np.uint8).copy()
    size = ref.size // n
    words = ref.view({4: np.uint32, 2: np.uint16, 1: np.uint8}[size]).copy()
    flip = rng.random(n) < 0.3
    words[flip] ^= 1
    cand = words.view(np.uint8)
    got = _sums(oracle, ref, cand, name, n, threads=3)
    assert got == _fsum_terms(_decode(ref, name), _decode(cand, name))


def test_exact_cancellation(oracle):
    """2^120 + 2^-120 - 2^120 = 2^-120 exactly (a running fp64 sum gives 0)."""
    r = np.array([2.0 ** 60, 2.0 ** -60, 2.0 ** 60], np.float32)
    c = np.array([2.0 ** 60, 2.0 ** -60, -(2.0 ** 60)], np.float32)
    rc, rr, cc = _sums(oracle, r.view(np.uint8), c.view(np.uint8), "F32", 3)
    assert rc == 2.0 ** -120
    assert rr == cc == 2.0 ** 121          # the 2^-120 is below half an ulp of 2^121


def test_extreme_magnitudes(oracle):
    """Products at both ends of the range: the largest fp32 squared and the
    smallest subnormal squared, each alone and together."""
    big = np.float32(np.finfo(np.float32).max)
    tiny = np.float32(2.0 ** -149)
    for vals in ([big], [tiny], [big, tiny, -big], [tiny, tiny, tiny]):
        r = np.array(vals, np.float32)
        got = _sums(oracle, r.view(np.uint8), r.view(np.uint8), "F32", len(vals))
        exact = sum(Fraction(float(v)) ** 2 for v in vals)
        assert got[1] == float(exact) == got[2]


def test_bruteforce_rationals(oracle):
    rng = np.random.default_rng(13)
    for trial in range(200):
        n = int(rng.integers(0, 9))
        r = _spread_f32(n, rng, -30, 30)
        c = _spread_f32(n, rng, -30, 30)
        got = _sums(oracle, r.view(np.uint8), c.view(np.uint8), "F32", n)
        fr = [Fraction(float(x)) for x in r]
        fc = [Fraction(float(x)) for x in c]
        want = (float(sum((a * b for a, b in zip(fr, fc)), Fraction(0))),
                float(sum((a * a for a in fr), Fraction(0))),
                float(sum((b * b for b in fc), Fraction(0))))
        assert got == want, trial


def test_closed_forms(oracle):
    ones = np.ones(1000, np.float32).view(np.uint8)
    assert _sums(oracle, ones, ones, "F32", 1000) == (1000.0, 1000.0, 1000.0)
    a = np.array([3, 4], np.float32)
    rc, rr, cc = _sums(oracle, a.view(np.uint8), (-a).view(np.uint8), "F32", 2)
    assert (rc, rr, cc) == (-25.0, 25.0, 25.0)
    assert oracle.eq_cos(rc, rr, cc) == -1.0
    e1, e2 = np.array([1, 0], np.float32), np.array([0, 1], np.float32)
    rc, rr, cc = _sums(oracle, e1.view(np.uint8), e2.view(np.uint8), "F32", 2)
    assert oracle.eq_cos(rc, rr, cc) == 0.0
    z = np.zeros(4, np.float32)
    assert oracle.eq_cos(*_sums(oracle, z.view(np.uint8), z.view(np.uint8), "F32", 4)) == 1.0
    assert oracle.eq_cos(*_sums(oracle, z.view(np.uint8), ones[:16], "F32", 4)) == 0.0
    # the cosine of Eq. 1 in closed form: (1, 1) against (1, 0) is 1/sqrt(2)
    rc, rr, cc = _sums(oracle, np.array([1, 1], np.float32).view(np.uint8),
                       e1.view(np.uint8), "F32", 2)
    assert abs(oracle.eq_cos(rc, rr, cc) - 2 ** -0.5) <= 2 * 2.0 ** -53   # two roundings


def test_nonfinite_terms_are_left_out(oracle):
    """Each sum drops exactly the elements whose own term is not finite."""
    rng = np.random.default_rng(14)
    r = rng.standard_normal(100).astype(np.float32)
    c = r + np.float32(1e-3)
    r2, c2 = r.copy(), c.copy()
    r2[[3, 50]] = np.nan
    c2[[7]] = np.inf
    c2[[50]] = np.nan
    rc, rr, cc = _sums(oracle, r2.view(np.uint8), c2.view(np.uint8), "F32", 100)

    def keep(*drop):
        k = np.ones(100, bool)
        k[list(drop)] = False
        return k
    k = keep(3, 7, 50)
    assert rc == _sums(oracle, r[k].view(np.uint8), c[k].view(np.uint8), "F32", 97)[0]
    k = keep(3, 50)
    assert rr == _sums(oracle, r[k].view(np.uint8), r[k].view(np.uint8), "F32", 98)[1]
    k = keep(7, 50)
    assert cc == _sums(oracle, c[k].view(np.uint8), c[k].view(np.uint8), "F32", 98)[2]
    # matching non-finite positions: all three sums are those of the finite part
    r3, c3 = r.copy(), c.copy()
    r3[[5, 9]] = [np.nan, -np.inf]
    c3[[5, 9]] = [np.nan, -np.inf]
    k = keep(5, 9)
    assert _sums(oracle, r3.view(np.uint8), c3.view(np.uint8), "F32", 100) == \
        _sums(oracle, r[k].view(np.uint8), c[k].view(np.uint8), "F32", 98)


def test_order_and_split_invariance(oracle):
    rng = np.random.default_rng(15)
    n = 3001
    r = _spread_f32(n, rng, -60, 60)
    c = _spread_f32(n, rng, -60, 60)
    whole = oracle.eq_sums_range(r.view(np.uint8), c.view(np.uint8), oracle.F32, 0, n)
    for cut in (0, 1, 1500, n):
        a = oracle.eq_sums_range(r.view(np.uint8), c.view(np.uint8), oracle.F32, 0, cut)
        b = oracle.eq_sums_range(r.view(np.uint8), c.view(np.uint8), oracle.F32, cut, n)
        assert tuple(x + y for x, y in zip(a, b)) == whole
    perm = rng.permutation(n)
    rp, cp = r[perm].copy(), c[perm].copy()
    assert oracle.eq_sums_range(rp.view(np.uint8), cp.view(np.uint8), oracle.F32, 0, n) == whole


def test_integer_regions_have_no_sums(oracle):
    a = np.arange(64, dtype=np.int32).view(np.uint8)
    assert oracle.eq_sums_range(a, a, oracle.I32, 0, 64) == (0, 0, 0)


def _stats(**kw):
    s = {"mismatches": 0, "first_mismatch": (1 << 64) - 1, "max_abs_err": 0.0,
         "max_rel_err": 0.0, "nonfinite_mismatches": 0, "guard_bad_bytes": 0,
         "first_guard_bad": (1 << 64) - 1, "ref_guard_bad_bytes": 0}
    s.update(kw)
    return s


def test_verdict_terms(oracle):
    o = oracle
    all4 = o.EQ_COS | o.EQ_LINF | o.EQ_INT | o.EQ_GUARD
    same = {"sum_rc": 4.0, "sum_rr": 4.0, "sum_cc": 4.0}
    v = o.eq_verdict(_stats(), same, o.F16)
    assert (v["cos"], v["flags"], v["eq"]) == (1.0, all4, 1)
    # L-infinity: tau itself passes, the next double above fails
    assert o.eq_verdict(_stats(max_abs_err=1e-3), same, o.F16)["eq"] == 1
    v = o.eq_verdict(_stats(max_abs_err=float(np.nextafter(1e-3, 1))), same, o.F16)
    assert (v["flags"], v["eq"]) == (all4 & ~o.EQ_LINF, 0)
    # a NaN/Inf-position mismatch fails the L-infinity term
    v = o.eq_verdict(_stats(nonfinite_mismatches=1, mismatches=1), same, o.F32)
    assert v["flags"] == all4 & ~o.EQ_LINF
    # cosine just below theta = 0.9999 fails; exactly theta passes
    rc = 0.9999 * 4.0
    assert o.eq_cos(rc, 4.0, 4.0) == rc / 4.0
    assert o.eq_verdict(_stats(), {"sum_rc": 3.9996, "sum_rr": 4.0, "sum_cc": 4.0},
                        o.F32)["eq"] == int(3.9996 / 4.0 >= 0.9999)
    v = o.eq_verdict(_stats(), {"sum_rc": 3.0, "sum_rr": 4.0, "sum_cc": 4.0}, o.F32)
    assert (v["cos"], v["flags"]) == (0.75, all4 & ~o.EQ_COS)
    # iota: integer buffers bit-exact, candidate guards intact
    v = o.eq_verdict(_stats(mismatches=1, max_abs_err=1.0), {}, o.I32)
    assert math.isnan(v["cos"]) and v["flags"] == all4 & ~o.EQ_INT
    assert o.eq_verdict(_stats(), {}, o.I8)["eq"] == 1
    v = o.eq_verdict(_stats(guard_bad_bytes=1, first_guard_bad=5), same, o.BF16)
    assert v["flags"] == all4 & ~o.EQ_GUARD
    # a float region's tolerance-predicate mismatches do not enter Eq. 1
    assert o.eq_verdict(_stats(mismatches=9, max_abs_err=1e-4), same, o.F32)["eq"] == 1
