"""GPU parity of the compare screens that work in the stored 16-bit format
(fp16, bf16, and every fp8 format through its fp16 value), with all
candidates of a batched launch sharing the reference's bounds:

- every pair of fp8 bit patterns (256 x 256), eight candidates per launch;
- every 16-bit reference pattern against eight perturbations of it (one
  to 64 units in the last place, a sign flip, random bits, the format's
  specials), so that every exponent, subnormal, zero, infinity and NaN of
  the reference meets differences on both sides of the tolerance bound;
- tolerances that make the bracket's lower end zero (atol = rtol = 0),
  its upper end overflow (rtol = 4, atol near the format's maximum), pure
  relative and pure absolute tolerances.

Each candidate's statistics are compared with the oracle bit for bit."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import assert_stats_equal, oracle_region_stats, to_device, torch_cuda

pytestmark = pytest.mark.gpu

FP8 = ["f8e4m3", "f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz"]
TOLS = [(0.0, 0.0), (1e-3, 1e-2), (0.0, 0.125), (1.0, 0.0), (60000.0, 4.0), (2.0 ** -20, 2.0 ** -9)]


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _run(ctx, oracle, dtype, R, Cs, tol):
    n = len(R) // W.DTYPE_SIZE[dtype]
    reg = W.Region("x", dtype, n, "raw", 0, 0, 0, 0, 0xA5, 0)
    reg.offset = 0
    dref = to_device(R)
    dcs = [to_device(C) for C in Cs]
    tl = {dtype: tol}
    got = ctx.compare_batched([asmv.make_region(dref.data_ptr(), n, dtype)],
                              [[asmv.make_region(d.data_ptr(), n, dtype)] for d in dcs], tl)
    for j, C in enumerate(Cs):
        want = oracle_region_stats(oracle, R, reg, C, reg, tl)
        assert_stats_equal(got[j][0], want, "%s tol %r cand %d" % (dtype, tol, j))
    return got


@pytest.mark.parametrize("dtype", FP8)
@pytest.mark.parametrize("tol", TOLS)
def test_every_fp8_pair(ctx, oracle, dtype, tol):
    """All 65536 (reference, candidate) byte pairs, in eight orders (one
    per candidate) so that every pair also meets its neighbours in a chunk."""
    a = np.arange(256, dtype=np.uint8)
    R = np.repeat(a, 256)
    base = np.tile(a, 256)
    rng = np.random.default_rng(256 + FP8.index(dtype))
    Cs = [base]
    for j in range(1, 8):
        # rotate the candidate bytes within each reference's block of 256
        Cs.append(np.tile(np.roll(a, 37 * j), 256) if j < 4 else
                  rng.permutation(256).astype(np.uint8)[base])
    _run(ctx, oracle, dtype, R, [np.ascontiguousarray(c) for c in Cs], tol)


def _specials(dtype):
    if dtype == "f16":
        return [0x0000, 0x8000, 0x7C00, 0xFC00, 0x7E00, 0xFE01, 0x7BFF, 0xFBFF, 0x0001, 0x8001, 0x0400]
    return [0x0000, 0x8000, 0x7F80, 0xFF80, 0x7FC0, 0xFFC1, 0x7F7F, 0xFF7F, 0x0001, 0x8001, 0x0080]


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("tol", TOLS)
def test_every_16bit_reference(ctx, oracle, dtype, tol):
    """Each of the 65536 16-bit patterns as a reference (twice, in two
    orders), against candidates moved 1, 2, 3, 8 and 64 units in the last
    place (either way), sign-flipped, random, or a special value."""
    rng = np.random.default_rng(16 + (dtype == "bf16"))
    r16 = np.concatenate([np.arange(65536, dtype=np.uint16),
                          rng.permutation(65536).astype(np.uint16)])
    n = len(r16)
    sp = np.array(_specials(dtype), np.uint16)
    Cs = []
    for j, k in enumerate([1, 2, 3, 8, 64]):
        sgn = np.where(rng.random(n) < 0.5, -1, 1)
        Cs.append((r16.astype(np.int64) + sgn * k).astype(np.uint16))   # wraps across signs
    Cs.append(r16 ^ np.uint16(0x8000))
    Cs.append(rng.integers(0, 65536, n).astype(np.uint16))
    Cs.append(np.where(rng.random(n) < 0.5, sp[rng.integers(0, len(sp), n)],
                       r16 ^ rng.integers(0, 16, n).astype(np.uint16)))
    R = r16.view(np.uint8).copy()
    _run(ctx, oracle, dtype, R, [c.view(np.uint8).copy() for c in Cs], tol)


@pytest.mark.parametrize("dtype", ["f16", "bf16", "f8e4m3", "f32"])
def test_single_candidate_matches_batched(ctx, oracle, dtype):
    """The one-candidate launch (its own kernel instance and tile size) and
    the batched launch agree with each other and with the oracle on the
    same dense differences."""
    import torch
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16,
           "f8e4m3": torch.float8_e4m3fn}[dtype]
    st = {"f32": torch.int32, "bf16": torch.int16, "f16": torch.int16, "f8e4m3": torch.uint8}[dtype]
    rng = np.random.default_rng(5)
    n = 3 * 16384 + 123
    r = torch.from_numpy(rng.standard_normal(n)).to(tdt)
    noise = {"f32": 2e-3, "bf16": 2e-2, "f16": 2e-3, "f8e4m3": 0.1}[dtype]
    c = torch.from_numpy(r.double().numpy() * (1 + rng.normal(0, noise, n))).to(tdt)
    R = r.view(st).numpy().view(np.uint8).copy()
    C = c.view(st).numpy().view(np.uint8).copy()
    reg = W.Region("x", dtype, n, "raw", 0, 0, 0, 0, 0xA5, 0)
    reg.offset = 0
    tol = {dtype: (1e-4, 1e-3)}
    dref, dc = to_device(R), to_device(C)
    one = ctx.compare([asmv.make_region(dref.data_ptr(), n, dtype)],
                      [asmv.make_region(dc.data_ptr(), n, dtype)], tol)[0]
    many = ctx.compare_batched([asmv.make_region(dref.data_ptr(), n, dtype)],
                               [[asmv.make_region(dc.data_ptr(), n, dtype)]] * 3, tol)
    want = oracle_region_stats(oracle, R, reg, C, reg, tol)
    assert_stats_equal(one, want, "single")
    for j in range(3):
        assert_stats_equal(many[j][0], want, "batched %d" % j)
    assert want["mismatches"] > 0
