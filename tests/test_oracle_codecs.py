"""Pins of the oracle's exact decoders (stored format -> fp64) and its
round-to-nearest-even encoders (fp32 -> bf16 / fp16 / OCP fp8 E4M3), by
exhaustive enumeration against numpy's and torch's own conversions."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _all_u16():
    return np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)


def _same_f64(a, b):
    """Bitwise equality with NaN == NaN (any payload)."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    both_nan = np.isnan(a) & np.isnan(b)
    same = (a.view(np.uint64) == b.view(np.uint64)) | both_nan
    return bool(same.all())


def test_decode_f16_exhaustive(oracle):
    h = _all_u16()
    got = oracle.decode(h.view(np.uint8), oracle.F16)
    want = h.view(np.float16).astype(np.float64)
    assert _same_f64(got, want)


def test_decode_bf16_exhaustive(oracle):
    h = _all_u16()
    got = oracle.decode(h.view(np.uint8), oracle.BF16)
    want = torch.from_numpy(h.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    assert _same_f64(got, want)


def test_decode_f8e4m3_exhaustive(oracle):
    b = np.arange(256, dtype=np.uint32).astype(np.uint8)
    got = oracle.decode(b, oracle.F8E4M3)
    want = torch.from_numpy(b.copy()).view(torch.float8_e4m3fn).double().numpy()
    assert _same_f64(got, want)
    # the format's landmarks: max 448, least subnormal 2^-9, NaN only at S.1111.111
    assert got[0x7E] == 448.0 and got[0x01] == 2.0 ** -9
    assert np.isnan(got[0x7F]) and np.isnan(got[0xFF]) and np.isnan(got).sum() == 2


def test_decode_ints(oracle):
    b = np.arange(256, dtype=np.uint32).astype(np.uint8)
    assert _same_f64(oracle.decode(b, oracle.I8), b.view(np.int8).astype(np.float64))
    assert _same_f64(oracle.decode(b, oracle.U8), b.astype(np.float64))
    v = np.array([0, 1, -1, 2**31 - 1, -2**31, 123456789], np.int32)
    assert _same_f64(oracle.decode(v.view(np.uint8), oracle.I32), v.astype(np.float64))


def _fp32_sweep(seed=5):
    """Random bit patterns over every exponent, every halfway point of the
    16-bit grids, and their neighbours."""
    rng = np.random.default_rng(seed)
    rnd = rng.integers(0, 1 << 32, size=1 << 21, dtype=np.uint64).astype(np.uint32)
    hi = (np.arange(1 << 16, dtype=np.uint32) << 16)
    ties_bf16 = hi | 0x8000                        # exactly halfway between bf16 neighbours
    f16_grid = _all_u16().view(np.float16).astype(np.float32)
    f16_grid = f16_grid[np.isfinite(f16_grid)]
    nxt = np.nextafter(f16_grid, np.float32(np.inf))
    # midpoints of consecutive fp16 values are exact in fp32
    srt = np.sort(np.unique(f16_grid.astype(np.float64)))
    mids = ((srt[1:] + srt[:-1]) / 2).astype(np.float32)
    pats = [rnd, hi, ties_bf16, ties_bf16 - 1, ties_bf16 + 1,
            f16_grid.view(np.uint32), nxt.view(np.uint32), mids.view(np.uint32),
            np.nextafter(mids, np.float32(np.inf)).view(np.uint32),
            np.nextafter(mids, np.float32(-np.inf)).view(np.uint32)]
    return np.concatenate(pats).view(np.float32)


def test_encode_bf16_rne(oracle):
    x = _fp32_sweep()
    fin = ~np.isnan(x)
    got = oracle.encode(x[fin], oracle.BF16).view(np.uint16)
    want = torch.from_numpy(x[fin].copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)


def test_encode_f16_rne(oracle):
    x = _fp32_sweep()
    fin = ~np.isnan(x)
    got = oracle.encode(x[fin], oracle.F16).view(np.uint16)
    with np.errstate(over="ignore"):
        want = x[fin].astype(np.float16).view(np.uint16)
    np.testing.assert_array_equal(got, want)


def test_encode_f8e4m3_rne_and_saturation(oracle):
    rng = np.random.default_rng(9)
    grid = oracle.decode(np.arange(256, dtype=np.uint32).astype(np.uint8), oracle.F8E4M3)
    grid = np.unique(grid[np.isfinite(grid)])
    mids = (grid[1:] + grid[:-1]) / 2
    x = np.concatenate([
        rng.uniform(-460, 460, 1 << 20),
        rng.standard_normal(1 << 20) * np.exp2(rng.uniform(-12, 8, 1 << 20)),
        grid, mids, np.nextafter(mids, np.inf), np.nextafter(mids, -np.inf),
    ]).astype(np.float32)
    inr = np.abs(x) < 448.0
    got = oracle.encode(x[inr], oracle.F8E4M3)
    want = torch.from_numpy(x[inr].copy()).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    np.testing.assert_array_equal(got, want)
    # finite overflow and infinities saturate to +-448 (0x7E / 0xFE); NaN -> S.1111.111
    big = np.array([448, 449, 463.9, 464, 465, 1e6, np.inf, -448, -500, -np.inf], np.float32)
    np.testing.assert_array_equal(oracle.encode(big, oracle.F8E4M3),
                                  [0x7E] * 7 + [0xFE] * 3)
    assert oracle.encode(np.array([np.nan], np.float32), oracle.F8E4M3)[0] & 0x7F == 0x7F
