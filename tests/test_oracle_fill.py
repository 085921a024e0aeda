"""Pins of the oracle's Tier 1 guarded fill (AsmEvo Sec. 3.4, Tier 1: seeded
deterministic inputs, allocations with canary guard regions).

Philox words come from PyTorch's engine run as a black box, so each test
checks the oracle's element mapping against an independent generator and a
closed form of the distribution."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _payload(o, dtype, n):
    return np.zeros(n * o.DTYPE_SIZE[dtype], np.uint8)


def test_raw_bytes_are_the_block_stream(oracle, torch_philox):
    n = 1000                                   # 62.5 blocks: a ragged tail
    p = _payload(oracle, oracle.U8, n)
    oracle.fill_payload(p, oracle.U8, oracle.RAW, 0, n, 7, 0, 0, 99)
    blocks = torch_philox(99, 7, np.arange(63))
    want = blocks.astype("<u4").view(np.uint8).reshape(-1)[:n]
    np.testing.assert_array_equal(p, want)
    # the same bytes for any element width: RAW is a byte stream
    q = _payload(oracle, oracle.I32, n // 4)
    oracle.fill_payload(q, oracle.I32, oracle.RAW, 0, n // 4, 7, 0, 0, 99)
    np.testing.assert_array_equal(q, want[:n // 4 * 4])


def test_int_range_power_of_two_is_a_shift(oracle, torch_philox):
    n = 4096
    p = _payload(oracle, oracle.I32, n)
    oracle.fill_payload(p, oracle.I32, oracle.INT_RANGE, 0, n, 0, 0, 131072, 3)
    w = torch_philox(3, 0, np.arange(n // 4)).reshape(-1)
    # (w * 2^17) >> 32 == w >> 15, and lo = 0
    np.testing.assert_array_equal(p.view(np.int32), (w >> 15).astype(np.int32))


def test_int_range_offset_and_span(oracle, torch_philox):
    n = 4000
    p = _payload(oracle, oracle.I8, n)
    oracle.fill_payload(p, oracle.I8, oracle.INT_RANGE, 0, n, 5, -100, 100, 11)
    w = torch_philox(11, 5, np.arange(n // 4)).reshape(-1).astype(np.uint64)
    want = (-100 + ((w * 200) >> 32).astype(np.int64)).astype(np.int8)
    np.testing.assert_array_equal(p.view(np.int8), want)
    v = p.view(np.int8)
    assert v.min() >= -100 and v.max() < 100


def test_uniform_minus_one_one_is_exact(oracle, torch_philox):
    n = 8192
    p = _payload(oracle, oracle.F32, n)
    oracle.fill_payload(p, oracle.F32, oracle.UNIFORM, 0, n, 0, -1.0, 1.0, 1)
    w = torch_philox(1, 0, np.arange(n // 4)).reshape(-1)
    # -1 + 2 * (w >> 8) 2^-24 is exact in fp32
    want = -1.0 + (w >> 8).astype(np.float64) * 2.0 ** -23
    np.testing.assert_array_equal(p.view(np.float32).astype(np.float64), want)


@pytest.mark.parametrize("dt,tdt", [("BF16", torch.bfloat16), ("F16", torch.float16),
                                    ("F8E4M3", torch.float8_e4m3fn)])
def test_uniform_low_precision_is_rne_of_fp32(oracle, torch_philox, dt, tdt):
    """16-bit formats take half (i mod 2) of word (i mod 8) div 2 of block
    i div 8 as f = h 2^-16, 8-bit formats byte (i mod 4) of word (i mod 16)
    div 4 of block i div 16 as f = b 2^-8; v = lo + f*(hi - lo) in fp32."""
    code = getattr(oracle, dt)
    sz = oracle.DTYPE_SIZE[code]
    per, bits = 16 // sz, 8 * sz
    n = 4096
    p = _payload(oracle, code, n)
    oracle.fill_payload(p, code, oracle.UNIFORM, 0, n, 2, -3.0, 5.0, 8)
    w = torch_philox(8, 2, np.arange(n // per)).reshape(-1)
    k = np.stack([(w >> (bits * q)) & ((1 << bits) - 1) for q in range(32 // bits)], axis=1)
    f = k.reshape(-1).astype(np.float32) * np.float32(2.0 ** -bits)
    v = np.float32(-3.0) + f * np.float32(8.0)        # fp32 mul then add, as stated
    want = torch.from_numpy(v).to(tdt).view(torch.uint8 if sz == 1 else torch.int16)
    np.testing.assert_array_equal(p, want.numpy().view(np.uint8))


def test_normal_element_mapping(oracle, torch_philox):
    """fp32: block i div 4 gives two pairs, words (0, 1) and (2, 3); the
    16-bit and 8-bit formats are pinned in test_oracle_narrow."""
    n = 1002                                  # odd pairs at the tail
    p = _payload(oracle, oracle.F32, n)
    oracle.fill_payload(p, oracle.F32, oracle.NORMAL, 0, n, 4, 0.25, 0.5, 77)
    w = torch_philox(77, 4, np.arange((n + 3) // 4))
    z0a, z1a = oracle.boxmuller(w[:, 0], w[:, 1])     # pair from words 0,1
    z0b, z1b = oracle.boxmuller(w[:, 2], w[:, 3])     # pair from words 2,3
    z = np.stack([z0a, z1a, z0b, z1b], axis=1).reshape(-1)[:n]
    v = np.float32(0.25) + np.float32(0.5) * z
    np.testing.assert_array_equal(p, v.view(np.uint8))


CASES = [("F32", "UNIFORM", -2.0, 3.0), ("F32", "NORMAL", 0.0, 1.0),
         ("BF16", "NORMAL", 1.0, 2.0), ("F16", "UNIFORM", 0.0, 1.0),
         ("F8E4M3", "NORMAL", 0.0, 1.0), ("I32", "INT_RANGE", -5, 1000),
         ("I8", "RAW", 0, 0), ("U8", "INT_RANGE", 0, 256), ("F16", "RAW", 0, 0)]


@pytest.mark.parametrize("dt,dist,p0,p1", CASES)
def test_fill_is_position_addressed(oracle, dt, dist, p0, p1):
    """Filling [0, n) in one call or in arbitrary pieces gives the same
    bytes: every element depends only on (seed, region, index)."""
    code, dcode = getattr(oracle, dt), getattr(oracle, dist)
    n = 777
    whole = _payload(oracle, code, n)
    oracle.fill_payload(whole, code, dcode, 0, n, 9, p0, p1, 1234)
    rng = np.random.default_rng(1)
    cuts = np.sort(rng.choice(np.arange(1, n), 6, replace=False))
    pieces = _payload(oracle, code, n)
    for a, b in zip([0, *cuts], [*cuts, n]):
        oracle.fill_payload(pieces, code, dcode, int(a), int(b), 9, p0, p1, 1234)
    np.testing.assert_array_equal(whole, pieces)
    # different seed or region id changes the stream
    other = _payload(oracle, code, n)
    oracle.fill_payload(other, code, dcode, 0, n, 10, p0, p1, 1234)
    sz = oracle.DTYPE_SIZE[code]
    differ = (other.reshape(-1, sz) != whole.reshape(-1, sz)).any(axis=1)
    assert differ.mean() > 0.5


def test_guards_and_payload_boundaries(oracle):
    glo, ghi, n = 37, 1001, 333
    alloc = np.full(glo + 4 * n + ghi + 16, 0x11, np.uint8)
    oracle.fill_region(alloc, n, oracle.I32, oracle.RAW, glo, ghi, 0, 0xA5, 0, 0, 5)
    assert (alloc[:glo] == 0xA5).all()
    assert (alloc[glo + 4 * n:glo + 4 * n + ghi] == 0xA5).all()
    assert (alloc[glo + 4 * n + ghi:] == 0x11).all()       # nothing past the allocation
    assert oracle.guard_check(alloc, 4 * n, glo, ghi, 0xA5) == (0, oracle.U64_NONE)


def test_none_writes_only_guards(oracle):
    alloc = np.full(64 + 40 + 64, 0x33, np.uint8)
    oracle.fill_region(alloc, 10, oracle.F32, oracle.NONE, 64, 64, 0, 0x5A, 0, 0, 1)
    assert (alloc[64:104] == 0x33).all() and (alloc[:64] == 0x5A).all()


def test_guard_check_closed_forms(oracle):
    glo, ghi, nb = 256, 256, 1000
    alloc = np.full(glo + nb + ghi, 0xA5, np.uint8)
    alloc[glo:glo + nb] = 0                      # payload content is irrelevant
    assert oracle.guard_check(alloc, nb, glo, ghi, 0xA5) == (0, oracle.U64_NONE)
    k = glo + nb + 17
    alloc[k] = 0x5A
    assert oracle.guard_check(alloc, nb, glo, ghi, 0xA5) == (1, k)
    alloc[3] = 0
    assert oracle.guard_check(alloc, nb, glo, ghi, 0xA5) == (2, 3)   # low side first
    alloc[:] = 0
    assert oracle.guard_check(alloc, nb, glo, ghi, 0xA5) == (glo + ghi, 0)


def test_rejects_inapplicable_distributions(oracle):
    p = np.zeros(64, np.uint8)
    with pytest.raises(ValueError):
        oracle.fill_payload(p, oracle.F32, oracle.INT_RANGE, 0, 4, 0, 0, 10, 1)
    with pytest.raises(ValueError):
        oracle.fill_payload(p, oracle.I32, oracle.NORMAL, 0, 4, 0, 0, 1, 1)
