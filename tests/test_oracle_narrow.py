"""Pins of the oracle's fill for the 16-bit and 8-bit float formats (reading
R12 of the oracle: one Philox block per 16-byte chunk; Box-Muller on a
16-bit radius index and a 16-bit angle index per 32-bit word for the 16-bit
formats, on an 8-bit radius index and an 8-bit angle index per 16 bits for
the 8-bit formats).

What fixes each part, independently of the oracle's own code:
- every table entry equals the correctly rounded fp32 value of its closed
  form, evaluated with 40-digit arithmetic;
- the 16-bit radius, over all 2^16 inputs, against float64
  sqrt(-2 ln((k + 1/2) 2^-16)): the chord over a cell of relative width
  1/16 is within 2^-13 of the curve, so that is the bound;
- the 16-bit angle, over all 2^16 inputs, in polar form against float64
  theta = 2 pi (a + 1/2) / 65536: a first-order rotation by |delta| <=
  pi / 256 scales by sqrt(1 + delta^2) <= 1 + 2^-13.7 and turns by
  delta - atan(delta) <= delta^3 / 3 < 2^-20.5;
- which bits feed which quantity, and the element order, from Philox words
  of PyTorch's engine run as a black box, against the float64 polar closed
  form of each element;
- the distributions: moments and Kolmogorov-Smirnov against N(0, 1), the
  tail reach in closed form, and the exact KS distance of the 8 + 8 law.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _rn32(mpmath, x):
    f = np.float32(float(x))
    cands = [np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))]
    return min(cands, key=lambda c: abs(mpmath.mpf(float(c)) - x))


def test_narrow_tables_are_correctly_rounded(oracle):
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 40
    t = oracle.narrow_tables()
    half = mpmath.mpf(1) / 2
    for E in range(32):
        d = 1 if E >= 16 else 0
        e = E - 16 * d
        for i in range(16):
            m0 = 1 + mpmath.mpf(i) / 16
            m1 = m0 + mpmath.mpf(1) / 16

            def g(m):
                y = m * mpmath.mpf(2) ** (e - 17)
                return mpmath.sqrt(-2 * mpmath.log(1 - y if d else y))
            S = 16 * (g(m1) - g(m0))
            assert t["A"][16 * E + i] == _rn32(mpmath, S * mpmath.mpf(2) ** (-E)), (E, i)
            assert t["B"][16 * E + i] == _rn32(mpmath, g(m0) - S * m0), (E, i)
    for j in range(256):
        phi = 2 * mpmath.pi * (j + half) / 256
        assert t["sin"][j] == _rn32(mpmath, mpmath.sin(phi))
        assert t["cos"][j] == _rn32(mpmath, mpmath.cos(phi))
        assert t["r8"][j] == _rn32(mpmath, mpmath.sqrt(-2 * mpmath.log((j + half) / 256)))
    assert t["c16"] == _rn32(mpmath, 2 * mpmath.pi / 65536)


def test_radius16_all_inputs(oracle):
    k = np.arange(1 << 16, dtype=np.uint32)
    got = oracle.radius16(k).astype(np.float64)
    want = np.sqrt(-2.0 * np.log((k + 0.5) * 2.0 ** -16))
    rel = np.abs(got - want) / want
    assert rel.max() <= 2.0 ** -13, rel.max()
    # the ends: the largest radius sqrt(2 * 17 ln 2) and the smallest
    assert abs(got[0] - np.sqrt(34 * np.log(2.0))) <= 2.0 ** -13 * got[0]
    assert abs(got[-1] - np.sqrt(-2 * np.log1p(-2.0 ** -17))) <= 2.0 ** -13 * got[-1]
    # the halves meet: u just below and just above 1/2
    assert abs(got[32767] - got[32768]) < 1e-4


def test_angle16_all_inputs(oracle):
    a = np.arange(1 << 16, dtype=np.uint32)
    sn, cs = oracle.angle16(a)
    sn, cs = sn.astype(np.float64), cs.astype(np.float64)
    theta = 2 * np.pi * (a + 0.5) / 65536
    scale = np.hypot(sn, cs)
    turn = np.angle(np.exp(1j * (np.arctan2(sn, cs) - theta)))
    assert np.abs(scale - 1).max() <= 2.0 ** -13.6, np.abs(scale - 1).max()
    assert np.abs(turn).max() <= 2.0 ** -20, np.abs(turn).max()
    assert (scale >= 1 - 2.0 ** -23).all()         # a rotation by delta never shrinks


def _f16_ulp(x):
    return np.spacing(np.abs(x).astype(np.float16)).astype(np.float64)


@pytest.mark.parametrize("dt,tdt", [("F16", torch.float16), ("BF16", torch.bfloat16)])
def test_normal16_bits_and_element_order(oracle, torch_philox, dt, tdt):
    code = getattr(oracle, dt)
    n = 8 * 3000 + 6                                  # a ragged last chunk
    p = np.zeros(2 * n, np.uint8)
    oracle.fill_payload(p, code, oracle.NORMAL, 0, n, 12, 0.0, 1.0, 2024)
    got = torch.from_numpy(p.view(np.int16).copy()).view(tdt).to(torch.float64).numpy()
    w = torch_philox(2024, 12, np.arange((n + 7) // 8)).reshape(-1)     # word q of block b
    k = (w & 0xFFFF).astype(np.float64)
    a = (w >> 16).astype(np.float64)
    rho = np.sqrt(-2 * np.log((k + 0.5) * 2.0 ** -16))
    th = 2 * np.pi * (a + 0.5) / 65536
    want = np.stack([rho * np.cos(th), rho * np.sin(th)], axis=1).reshape(-1)[:n]
    rho_e = np.repeat(rho, 2)[:n]
    ulp = _f16_ulp(want) if code == oracle.F16 else np.abs(
        torch.from_numpy(want).to(torch.bfloat16).to(torch.float64).numpy()) * 2.0 ** -7 + 2.0 ** -133
    err = np.abs(got - want)
    assert (err <= 2.0 ** -12.3 * rho_e + ulp).all(), err.max()


def test_normal8_bits_and_element_order(oracle, torch_philox):
    n = 16 * 2000 + 9
    p = np.zeros(n, np.uint8)
    oracle.fill_payload(p, oracle.F8E4M3, oracle.NORMAL, 0, n, 3, 0.0, 1.0, 55)
    got = torch.from_numpy(p.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    w = torch_philox(55, 3, np.arange((n + 15) // 16)).reshape(-1)
    halves = np.stack([w & 0xFFFF, w >> 16], axis=1).reshape(-1)    # low half first
    k = (halves & 0xFF).astype(np.float64)
    a = (halves >> 8).astype(np.float64)
    rho = np.sqrt(-2 * np.log((k + 0.5) / 256))
    th = 2 * np.pi * (a + 0.5) / 256
    z = np.stack([rho * np.cos(th), rho * np.sin(th)], axis=1).reshape(-1)[:n]
    # RNE of the exact value, except where fp32 rounding decides a near-tie
    want = torch.from_numpy(z).to(torch.float8_e4m3fn).to(torch.float64).numpy()
    diff = got != want
    near = np.abs(np.abs(z) - np.abs(got + want) / 2) <= 4e-7 * np.abs(z) + 1e-30
    assert (~diff | near).all()
    assert diff.mean() < 1e-3


def test_normal16_is_standard_normal(oracle):
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(77)
    w = rng.integers(0, 1 << 32, size=1 << 21, dtype=np.uint64).astype(np.uint32)
    v0, v1 = oracle.normal16(w)
    z = np.concatenate([v0, v1]).astype(np.float64)
    m = z.size
    assert abs(z.mean()) < 5 / np.sqrt(m)
    assert abs(z.var() - 1.0) < 5 * np.sqrt(2.0 / m)
    assert abs(stats.skew(z)) < 5 * np.sqrt(6.0 / m)
    assert abs(stats.kurtosis(z)) < 5 * np.sqrt(24.0 / m)
    assert stats.kstest(z, "norm").pvalue > 1e-4
    assert abs(np.corrcoef(v0, v1)[0, 1]) < 5 / np.sqrt(w.size)
    # mean and std enter as rs = rho*std, v = rs*cos + mean
    u0, u1 = oracle.normal16(w[:4096], 0.75, 3.0)
    r0, _ = oracle.normal16(w[:4096])
    np.testing.assert_allclose(u0, 0.75 + 3.0 * r0.astype(np.float64), rtol=0, atol=1e-5)


def test_normal8_law(oracle):
    """All 2^16 inputs of an 8-bit pair: the exact KS distance of the law to
    N(0, 1), its tail reach sqrt(-2 ln(1/512)) cos(pi/256) (the largest
    radius at the angle nearest an axis) and its symmetry."""
    special = pytest.importorskip("scipy.special")
    h = np.arange(1 << 16, dtype=np.uint32)
    v0, v1 = oracle.normal8(h)
    z = np.sort(np.concatenate([v0, v1]).astype(np.float64))
    n = z.size
    phi = special.ndtr(z)
    ks = max(np.max(np.arange(1, n + 1) / n - phi), np.max(phi - np.arange(n) / n))
    assert ks < 2.0 ** -9.3, ks
    assert abs(np.abs(z).max() - np.sqrt(-2 * np.log(1 / 512)) * np.cos(np.pi / 256)) < 1e-6
    np.testing.assert_array_equal(z, -z[::-1])              # the angles are symmetric
    assert abs(z.var() - 1.0) < 2e-3


@pytest.mark.parametrize("dt,tdt,lo,hi", [("BF16", torch.bfloat16, -1.0, 1.0),
                                          ("F16", torch.float16, -1.0, 1.0),
                                          ("F8E4M3", torch.float8_e4m3fn, 0.0, 1.0),
                                          ("F8E5M2", torch.float8_e5m2, -1.0, 1.0)])
def test_uniform_narrow_is_rne_of_the_exact_fraction(oracle, torch_philox, dt, tdt, lo, hi):
    code = getattr(oracle, dt)
    sz = oracle.DTYPE_SIZE[code]
    per = 16 // sz                                         # elements per block
    n = per * 500 + per // 2 + 1
    p = np.zeros(n * sz, np.uint8)
    oracle.fill_payload(p, code, oracle.UNIFORM, 0, n, 6, lo, hi, 31)
    w = torch_philox(31, 6, np.arange((n + per - 1) // per)).reshape(-1)
    bits = 8 * sz
    parts = np.stack([(w >> (bits * q)) & ((1 << bits) - 1) for q in range(32 // bits)],
                     axis=1).reshape(-1)[:n].astype(np.float64)
    v = lo + (hi - lo) * parts * 2.0 ** -bits              # exact in fp32 for these ranges
    want = torch.from_numpy(v.astype(np.float32)).to(tdt)
    want = want.view(torch.uint8 if sz == 1 else torch.int16).numpy().view(np.uint8)
    np.testing.assert_array_equal(p, want)
