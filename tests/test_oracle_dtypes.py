"""Pins of the oracle on the further stored formats: OCP FP8 E5M2, the fnuz
FP8 formats E4M3FNUZ and E5M2FNUZ, binary64, int16 and int64.  Decoders by
exhaustive or random enumeration against torch / numpy; encoders against
torch's round-to-nearest-even conversions inside the range, every halfway
point of each grid, and closed forms for saturation and zero; the fill
mappings and the comparison statistics through the same independent
conversions and exact integer arithmetic."""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

FP8 = {"F8E5M2": (torch.float8_e5m2, 57344.0), "F8E4M3FNUZ": (torch.float8_e4m3fnuz, 240.0),
       "F8E5M2FNUZ": (torch.float8_e5m2fnuz, 57344.0)}


def _same_f64(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return bool(((a.view(np.uint64) == b.view(np.uint64)) | (np.isnan(a) & np.isnan(b))).all())


def _all_bytes():
    return np.arange(256, dtype=np.uint32).astype(np.uint8)


def _torch_decode(raw, tdt):
    return torch.from_numpy(raw.copy()).view(tdt).double().numpy()


@pytest.mark.parametrize("name", sorted(FP8))
def test_decode_fp8_exhaustive(oracle, name):
    tdt, mx = FP8[name]
    b = _all_bytes()
    got = oracle.decode(b, getattr(oracle, name))
    assert _same_f64(got, _torch_decode(b, tdt))
    fin = got[np.isfinite(got)]
    assert fin.max() == mx and fin.min() == -mx


def test_fp8_landmarks(oracle):
    e5 = oracle.decode(_all_bytes(), oracle.F8E5M2)
    assert e5[0x7C] == np.inf and e5[0xFC] == -np.inf and np.isnan(e5).sum() == 6
    assert e5[0x01] == 2.0 ** -16 and e5[0x7B] == 57344.0
    for name, least in (("F8E4M3FNUZ", 2.0 ** -10), ("F8E5M2FNUZ", 2.0 ** -17)):
        v = oracle.decode(_all_bytes(), getattr(oracle, name))
        assert np.isnan(v).sum() == 1 and np.isnan(v[0x80]) and np.isfinite(v[0x7F])
        assert v[0x01] == least and not np.signbit(v[0x00])


def test_decode_wide_types(oracle):
    rng = np.random.default_rng(3)
    bits = rng.integers(0, 1 << 63, size=50000, dtype=np.uint64) * np.uint64(2) + \
        rng.integers(0, 2, size=50000, dtype=np.uint64)
    specials = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, 1.7976931348623157e308])
    f64 = np.concatenate([bits.view(np.float64), specials])
    assert _same_f64(oracle.decode(f64.view(np.uint8), oracle.F64), f64)
    i16 = np.arange(-32768, 32768, dtype=np.int16)
    assert _same_f64(oracle.decode(i16.view(np.uint8), oracle.I16), i16.astype(np.float64))
    i64 = np.array([0, 1, -1, 2**53, -2**53, 2**62, -2**63, 2**63 - 1], np.int64)
    assert _same_f64(oracle.decode(i64.view(np.uint8), oracle.I64), i64.astype(np.float64))


def _grid_and_mids(oracle, code):
    g = oracle.decode(_all_bytes(), code)
    g = np.unique(g[np.isfinite(g)])
    mids = (g[1:] + g[:-1]) / 2                  # exact in fp64 and in fp32
    return g, mids


@pytest.mark.parametrize("name", sorted(FP8))
def test_encode_fp8_rne(oracle, name):
    tdt, mx = FP8[name]
    code = getattr(oracle, name)
    g, mids = _grid_and_mids(oracle, code)
    rng = np.random.default_rng(11)
    x = np.concatenate([
        rng.uniform(-mx, mx, 1 << 18),
        rng.standard_normal(1 << 18) * np.exp2(rng.uniform(-20, 16, 1 << 18)),
        g, mids, np.nextafter(mids, np.inf), np.nextafter(mids, -np.inf)]).astype(np.float32)
    x = x[np.abs(x) <= mx]
    got = oracle.encode(x, code)
    want = torch.from_numpy(x.copy()).to(tdt).view(torch.uint8).numpy()
    if name != "F8E5M2":                         # fnuz: no negative zero
        want = np.where(want == 0x80, 0, want)
    np.testing.assert_array_equal(got, want)
    # every halfway point goes to the neighbour with an even mantissa
    enc = oracle.encode(mids.astype(np.float32), code)
    lo_enc = oracle.encode(g[:-1].astype(np.float32), code)
    hi_enc = oracle.encode(g[1:].astype(np.float32), code)
    mag = enc & 0x7F                             # zero's sign follows the midpoint's
    assert ((mag == lo_enc & 0x7F) | (mag == hi_enc & 0x7F)).all() and ((enc & 1) == 0).all()


@pytest.mark.parametrize("name", sorted(FP8))
def test_encode_fp8_saturation_zero_nan(oracle, name):
    tdt, mx = FP8[name]
    code = getattr(oracle, name)
    top = oracle.encode(np.array([mx], np.float32), code)[0]
    big = np.array([mx * 1.1, 1e30, np.inf, -mx * 1.1, -np.inf], np.float32)
    np.testing.assert_array_equal(oracle.encode(big, code), [top] * 3 + [top | 0x80] * 2)
    tiny = np.array([-0.0, -1e-30, 1e-30], np.float32)
    z = oracle.encode(tiny, code)
    if name == "F8E5M2":
        np.testing.assert_array_equal(z, [0x80, 0x80, 0x00])
        assert oracle.encode(np.array([np.nan], np.float32), code)[0] & 0x7F == 0x7F
    else:
        np.testing.assert_array_equal(z, [0, 0, 0])
        assert oracle.encode(np.array([np.nan], np.float32), code)[0] == 0x80


def test_encode_f64_is_exact_widening(oracle):
    rng = np.random.default_rng(12)
    x = rng.integers(0, 1 << 32, size=100000, dtype=np.uint64).astype(np.uint32).view(np.float32)
    x = x[~np.isnan(x)]
    got = oracle.encode(x, oracle.F64).view(np.float64)
    assert _same_f64(got, x.astype(np.float64))


@pytest.mark.parametrize("name", ["F8E5M2", "F8E4M3FNUZ", "F8E5M2FNUZ", "F64"])
def test_fill_float_mappings(oracle, torch_philox, name):
    """binary64 takes word (i mod 4) of block i div 4 (UNIFORM) and the pairs
    of words (0, 1), (2, 3) (NORMAL); the 8-bit formats take byte (i mod 4)
    of word (i mod 16) div 4 of block i div 16 (UNIFORM, f = b 2^-8) and the
    8 + 8 pair of half (i mod 4) div 2 of that word (NORMAL)."""
    code = getattr(oracle, name)
    n = 4099
    size = oracle.DTYPE_SIZE[code]
    per = 16 // size if size == 1 else 4
    p = np.zeros(n * size, np.uint8)
    oracle.fill_payload(p, code, oracle.UNIFORM, 0, n, 5, -3.0, 5.0, 21)
    w = torch_philox(21, 5, np.arange((n + per - 1) // per)).reshape(-1)
    if size == 1:
        f = np.stack([(w >> (8 * q)) & 0xFF for q in range(4)], axis=1).reshape(-1)[:n]
        f = f.astype(np.float32) * np.float32(2.0 ** -8)
    else:
        f = (w[:n] >> 8).astype(np.float32) * np.float32(2.0 ** -24)
    v = np.float32(-3.0) + f * np.float32(8.0)
    want = oracle.encode(v, code)
    np.testing.assert_array_equal(p, want)
    q = np.zeros(n * size, np.uint8)
    oracle.fill_payload(q, code, oracle.NORMAL, 0, n, 6, 0.5, 2.0, 22)
    w = torch_philox(22, 6, np.arange((n + per - 1) // per))
    if size == 1:
        h = np.stack([w & 0xFFFF, w >> 16], axis=2).reshape(-1)
        v0, v1 = oracle.normal8(h, 0.5, 2.0)
        vz = np.stack([v0, v1], axis=1).reshape(-1)[:n]
    else:
        z0a, z1a = oracle.boxmuller(w[:, 0], w[:, 1])
        z0b, z1b = oracle.boxmuller(w[:, 2], w[:, 3])
        z = np.stack([z0a, z1a, z0b, z1b], axis=1).reshape(-1)[:n]
        vz = np.float32(0.5) + np.float32(2.0) * z
    np.testing.assert_array_equal(q, oracle.encode(vz, code))
    if name != "F64":
        tdt = FP8[name][0]
        inr = np.abs(v) <= FP8[name][1]
        t = torch.from_numpy(v[inr].copy()).to(tdt).view(torch.uint8).numpy()
        np.testing.assert_array_equal(p[inr], t)


@pytest.mark.parametrize("name,lo,hi", [("I16", -32768, 32768), ("I16", -5, 1000),
                                        ("I64", -(2 ** 53), 2 ** 53 - 2 ** 32 + 7),
                                        ("I64", 0, 1 << 32)])
def test_fill_int_range(oracle, torch_philox, name, lo, hi):
    code = getattr(oracle, name)
    n = 1001
    size = oracle.DTYPE_SIZE[code]
    p = np.zeros(n * size, np.uint8)
    span = min(hi - lo, 1 << 32)
    oracle.fill_payload(p, code, oracle.INT_RANGE, 0, n, 9, float(lo), float(lo + span), 4)
    w = torch_philox(4, 9, np.arange((n + 3) // 4)).reshape(-1)[:n].astype(object)
    want = [lo + ((int(x) * span) >> 32) for x in w]
    got = p.view(np.int16 if name == "I16" else np.int64).tolist()
    assert got == want


def _cmp(oracle, r, c, code, atol=0.0, rtol=0.0):
    return oracle.compare_range(np.ascontiguousarray(r).view(np.uint8),
                                np.ascontiguousarray(c).view(np.uint8), code, 0, len(r), atol, rtol)


def test_int64_statistics_are_exact(oracle):
    r = np.array([2 ** 62, 5, -2 ** 63, 2 ** 53 + 1, 0, 7], np.int64)
    c = np.array([-2 ** 62, 5, 2 ** 63 - 1, 2 ** 53 + 3, 3, 7], np.int64)
    st = _cmp(oracle, r, c, oracle.I64)
    assert st["mismatches"] == 4 and st["first_mismatch"] == 0
    diffs = [abs(int(a) - int(b)) for a, b in zip(r, c)]
    assert st["max_abs_err"] == float(max(diffs)) == 2.0 ** 64      # |c - r| = 2^64 - 1, rounded
    assert st["max_rel_err"] == math.inf                           # r = 0, c = 3
    # operands beyond 2^53: the difference is formed exactly before rounding
    st = _cmp(oracle, np.array([2 ** 53 + 1], np.int64), np.array([2 ** 53 + 3], np.int64), oracle.I64)
    assert st["max_abs_err"] == 2.0 and st["max_rel_err"] == 2.0 / 2.0 ** 53
    st = _cmp(oracle, r[:4], c[:4], oracle.I64)
    assert st["max_rel_err"] == max(float(d) / abs(float(a)) for d, a in zip(diffs[:4], r[:4])
                                    if a != 0)


@pytest.mark.parametrize("name", ["F8E5M2", "F8E4M3FNUZ", "F8E5M2FNUZ", "F64"])
def test_float_predicate_matches_torch_isclose(oracle, name):
    code = getattr(oracle, name)
    rng = np.random.default_rng(31)
    n = 20000
    if name == "F64":
        r = rng.standard_normal(n) * np.exp2(rng.integers(-30, 30, n))
        c = r * (1 + rng.standard_normal(n) * 1e-3)
        c[::97] = r[::97]
        r[5], c[5] = np.nan, np.nan
        r[6], c[6] = np.inf, np.inf
        r[7], c[7] = 1.0, np.inf
        rr, cc = r, c
        rawr, rawc = r.view(np.uint8), c.view(np.uint8)
    else:
        rawr = rng.integers(0, 256, n, dtype=np.uint8)
        rawc = rawr.copy()
        flip = rng.random(n) < 0.5
        rawc[flip] ^= rng.integers(1, 8, flip.sum(), dtype=np.uint8)
        tdt = FP8[name][0]
        rr, cc = _torch_decode(rawr, tdt), _torch_decode(rawc, tdt)
    for atol, rtol in ((1e-5, 1e-3), (0.0, 0.1), (0.5, 0.0)):
        st = oracle.compare_range(rawr, rawc, code, 0, n, atol, rtol)
        tr, tc = torch.from_numpy(np.asarray(rr, np.float64)), torch.from_numpy(np.asarray(cc, np.float64))
        ok = torch.isclose(tc, tr, rtol=rtol, atol=atol, equal_nan=True).numpy()
        assert st["mismatches"] == int((~ok).sum())
