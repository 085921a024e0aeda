"""Eq. 1 over a check split into element ranges (host side, no GPU): the
verdict that asmv_eq_from_digits forms from digit vectors summed over the
shards and statistics merged over them equals the oracle's verdict on the
whole region, bit for bit (the three rounded sums, the cosine, the four
terms).  The digit vectors are built here from the oracle's exact integer
sums of each shard, in the library's layout: slot 0 sum r*r, then per
candidate sum r*d and sum d*d (d = c - r) for fp16 and the fp8 formats other
than E4M3, sum r*c and sum c*c otherwise, digit d weighing
2^(32 d + eq_digit_base)."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import distributed as D

FLOATS = ["f32", "bf16", "f16", "f8e4m3", "f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz"]
DIFF_FORM = {"f16", "f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz"}
ONAME = {"f32": "F32", "bf16": "BF16", "f16": "F16", "f8e4m3": "F8E4M3", "f8e5m2": "F8E5M2",
         "f8e4m3fnuz": "F8E4M3FNUZ", "f8e5m2fnuz": "F8E5M2FNUZ", "f64": "F64"}
SIZE = {"f32": 4, "bf16": 2, "f16": 2, "f64": 8}


def to_digits(v, base, rng=None, nd=20):
    """The integer v (value v 2^base) as nd signed int64 digits; with rng,
    a random carry is moved between neighbours (same integer)."""
    d = [(v >> (32 * k)) & 0xFFFFFFFF for k in range(nd - 1)] + [v >> (32 * (nd - 1))]
    if rng is not None:
        for k in range(nd - 1):
            t = int(rng.integers(-3, 4))
            d[k] += t << 32
            d[k + 1] -= t
    return np.array(d, np.int64)


def shard_digits(o, ref, cands, dt, i0, i1, rng=None, nd=None):
    """Digit vectors (1 + 2k, nd) of elements [i0, i1) of one region; nd
    defaults to the digits its dtype needs (20, or 136 for binary64)."""
    code = getattr(o, ONAME[dt])
    base = asmv.eq_digit_base(dt)
    nd = nd or (asmv.EQ64_DIGITS if dt == "f64" else asmv.EQ_DIGITS)
    if dt == "f64":
        assert base == o.EQ64_BASE
        vals = []
        for c in cands:
            rc, rr, cc = o.eq64_sums_range(ref, c, i0, i1)
            vals += [rc, cc]
        return np.stack([to_digits(v, base, rng, nd) for v in [rr] + vals])
    shift = base - o.EQ_BASE
    out = []
    s_rr = None
    per = []
    for c in cands:
        rc, rr, cc = o.eq_sums_range(ref, c, code, i0, i1)
        s_rr = rr
        per.append((rc, cc))
    vals = [s_rr]
    for rc, cc in per:
        if dt in DIFF_FORM:
            vals += [rc - s_rr, cc - 2 * rc + s_rr]
        else:
            vals += [rc, cc]
    for v in vals:
        assert v % (1 << shift) == 0
        out.append(to_digits(v >> shift, base, rng, nd))
    return np.stack(out)


def full_stats(o, ref, cand, dt, i0, i1, tol):
    st = o.compare_range(ref, cand, getattr(o, ONAME[dt]), i0, i1, tol[0], tol[1])
    out = D.empty_stats()
    for f in ("mismatches", "first_mismatch", "max_abs_err", "max_rel_err", "nonfinite_mismatches"):
        out[f] = st[f]
    return out


def _payloads(o, dt, n, k, rng):
    size = SIZE.get(dt, 1)
    code = getattr(o, ONAME[dt])
    ref = np.zeros(n * size, np.uint8)
    o.fill_payload(ref, code, o.NORMAL, 0, n, 3, 0.0, 2.0, 17)
    cands = []
    for j in range(k):
        c = ref.copy()
        pos = rng.integers(0, n * size, 40 * (j + 1))
        c[pos] ^= rng.integers(1, 4, pos.size).astype(np.uint8)
        cands.append(c)
    return ref, cands


@pytest.mark.parametrize("dt", FLOATS)
def test_sharded_verdict_equals_whole(oracle, dt):
    rng = np.random.default_rng(7)
    n, k = 5003, 2
    ref, cands = _payloads(oracle, dt, n, k, rng)
    tol = (1e-2, 1e-2)
    cuts = [0, 1601, 1602, n]                       # three shards, one of a single element
    dig = sum(shard_digits(oracle, ref, cands, dt, a, b, rng) for a, b in zip(cuts, cuts[1:]))
    stats = []
    for c in cands:
        m = D.empty_stats()
        for a, b in zip(cuts, cuts[1:]):
            m = D.merge_stats(m, D.to_region_coordinates(full_stats(oracle, ref, c, dt, a, b, tol), a, 0))
        stats.append([m])
    got = asmv.eq_from_digits([dt], stats, dig[None, :, :])
    for j, c in enumerate(cands):
        whole = full_stats(oracle, ref, c, dt, 0, n, tol)
        assert stats[j][0] == whole
        sums = oracle.eq_sums(ref, c, getattr(oracle, ONAME[dt]), n)
        want = oracle.eq_verdict(whole, sums, getattr(oracle, ONAME[dt]))
        for f in ("sum_rc", "sum_rr", "sum_cc", "flags", "eq"):
            assert got[j][0][f] == want[f], (dt, j, f)
        assert got[j][0]["cos"] == want["cos"] or (np.isnan(got[j][0]["cos"]) and np.isnan(want["cos"]))


def _f64_payloads(kind, n, k, rng):
    sign = np.where(rng.random(n) < 0.5, -1.0, 1.0)
    mant = rng.uniform(1.0, 2.0, n)
    lo, hi = {"normal": (-8, 3), "full_range": (-1074, 1024), "huge": (900, 1024),
              "tiny": (-1074, -1000)}[kind]
    r = sign * np.ldexp(mant, rng.integers(lo, hi, n))
    r[rng.random(n) < 0.02] = 0.0
    r[[5, 6]] = [np.nan, np.inf]
    cands = []
    for j in range(k):
        c = r.copy()
        bits = c.view(np.uint64)
        flip = rng.random(n) < 0.3
        bits[flip] ^= np.uint64(1 + j)
        c[rng.choice(n, 2, replace=False)] *= -0.5
        if j == 1:
            c[9] = -np.inf
        cands.append(c.view(np.uint8))
    return r.view(np.uint8), cands


def _bits(x):
    return np.float64(x).view(np.uint64)


@pytest.mark.parametrize("kind", ["normal", "full_range", "huge", "tiny"])
def test_sharded_binary64_verdict_equals_whole(oracle, kind):
    """Binary64: the exact sums (rounded with gradual underflow and
    overflow to infinity) and the scaled cosine, from digit vectors summed
    over three shards, equal the oracle's on the whole region bit for bit."""
    rng = np.random.default_rng(21)
    n, k = 3001, 2
    ref, cands = _f64_payloads(kind, n, k, rng)
    tol = (1e-9, 1e-9)
    cuts = [0, 1000, 1001, n]
    dig = sum(shard_digits(oracle, ref, cands, "f64", a, b, rng) for a, b in zip(cuts, cuts[1:]))
    stats = []
    for c in cands:
        m = D.empty_stats()
        for a, b in zip(cuts, cuts[1:]):
            m = D.merge_stats(m, D.to_region_coordinates(full_stats(oracle, ref, c, "f64", a, b, tol), a, 0))
        stats.append([m])
    got = asmv.eq_from_digits(["f64"], stats, D.normalize_digits(dig)[None, :, :])
    for j, c in enumerate(cands):
        whole = full_stats(oracle, ref, c, "f64", 0, n, tol)
        want = oracle.eq_verdict(whole, oracle.eq_sums(ref, c, oracle.F64, n), oracle.F64)
        for f in ("sum_rc", "sum_rr", "sum_cc", "cos"):
            assert _bits(got[j][0][f]) == _bits(want[f]), (kind, j, f, got[j][0][f], want[f])
        assert (got[j][0]["flags"], got[j][0]["eq"]) == (want["flags"], want["eq"])


def test_mixed_table_pads_every_region_to_binary64_digits(oracle):
    rng = np.random.default_rng(22)
    n = 777
    ref64, c64 = _f64_payloads("normal", n, 1, rng)
    ref32, c32 = _payloads(oracle, "f32", n, 1, rng)
    tol = (1e-6, 1e-6)
    nd = asmv.digits_per_slot(["f32", "f64"])
    assert nd == asmv.EQ64_DIGITS and asmv.digits_per_slot(["f32", "i8"]) == asmv.EQ_DIGITS
    dig = np.stack([shard_digits(oracle, ref32, c32, "f32", 0, n, nd=nd),
                    shard_digits(oracle, ref64, c64, "f64", 0, n, nd=nd)])
    stats = [[full_stats(oracle, ref32, c32[0], "f32", 0, n, tol),
              full_stats(oracle, ref64, c64[0], "f64", 0, n, tol)]]
    got = asmv.eq_from_digits(["f32", "f64"], stats, dig)[0]
    for g, (dt, r, c) in zip(got, (("f32", ref32, c32[0]), ("f64", ref64, c64[0]))):
        code = getattr(oracle, ONAME[dt])
        want = oracle.eq_verdict(full_stats(oracle, r, c, dt, 0, n, tol),
                                 oracle.eq_sums(r, c, code, n), code)
        for f in ("sum_rc", "sum_rr", "sum_cc", "cos", "flags", "eq"):
            assert _bits(g[f]) == _bits(want[f]), (dt, f)
    bad = dig.copy()
    bad[0, 1, 40] = 1                      # an f32 digit beyond its 20
    with pytest.raises(asmv.AsmvError):
        asmv.eq_from_digits(["f32", "f64"], stats, bad)
    neg = dig.copy()
    neg[1, 0, :] = 0
    neg[1, 0, 0] = -1                      # a negative sum of squares
    with pytest.raises(asmv.AsmvError):
        asmv.eq_from_digits(["f32", "f64"], stats, neg)
    assert asmv.eq_digit_base("f64") == oracle.EQ64_BASE


def test_normalized_digits_keep_the_integer():
    rng = np.random.default_rng(3)
    for _ in range(200):
        v = int(rng.integers(-2 ** 62, 2 ** 62)) << int(rng.integers(0, 500))
        d = to_digits(v, 0, rng)
        nd = D.normalize_digits(d)
        assert sum(int(x) << (32 * i) for i, x in enumerate(nd)) == v
        assert all(0 <= int(x) < 2 ** 32 for x in nd[:-1])


def test_integer_regions_and_rejections():
    st = [[D.empty_stats()]]
    dig = np.zeros((1, 3, asmv.EQ_DIGITS), np.int64)
    e = asmv.eq_from_digits(["i32"], st, dig)[0][0]
    assert e["flags"] == 15 and e["eq"] == 1 and np.isnan(e["cos"])
    st[0][0]["mismatches"] = 1
    assert asmv.eq_from_digits(["i32"], st, dig)[0][0]["flags"] == 11
    for bad in (lambda: asmv.eq_from_digits(["f32"], [[D.empty_stats()]], dig, theta=float("nan")),
                lambda: asmv.eq_from_digits(["f32"], [[D.empty_stats()]], dig, tau=-1.0)):
        with pytest.raises(asmv.AsmvError) as ex:
            bad()
        assert ex.value.status == asmv.EINVAL
    huge = dig.copy()
    huge[0, 0, 5] = huge[0, 1, 5] = 2 ** 62              # S_rr + 2 sum r d leaves int64
    with pytest.raises(asmv.AsmvError):
        asmv.eq_from_digits(["f16"], [[D.empty_stats()]], huge)
    with pytest.raises(asmv.AsmvError):
        asmv.eq_digit_base("i8")
