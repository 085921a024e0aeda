"""GPU parity on the further stored formats (FP8 E5M2, E4M3FNUZ, E5M2FNUZ,
binary64, int16, int64): the guarded fill byte for byte, the comparison
field by field (bit patterns over the whole code space, special values, the
fnuz NaN and top values, int64 differences beyond 2^53), and Eq. 1's exact
sums for the fp8 formats (binary64: test_gpu_eq64.py), all against the
oracle on the same bytes."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from oracle.oracle import CODE_OF_DTYPE as ORACLE_DTYPE

from ._gpu import (assert_stats_equal, oracle_fill_arena, oracle_region_stats, to_device,
                   to_host, torch_cuda)

pytestmark = pytest.mark.gpu

TILE = 16 * 1024
NEW_FLOATS = ("f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz", "f64")
NEW_INTS = ("i16", "i64")


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _layout(regs, skew=None):
    off = 0
    for i, r in enumerate(regs):
        off = (off + 255) // 256 * 256 + (skew or {}).get(i, 0)
        r.offset = off
        off += r.alloc_bytes
    return off + 64


FILL = [(dt, "uniform", -3.0, 5.0) for dt in NEW_FLOATS] + \
       [(dt, "normal", 0.5, 2.0) for dt in NEW_FLOATS] + \
       [("f8e4m3fnuz", "uniform", -300.0, 300.0), ("f8e5m2fnuz", "uniform", -70000.0, 70000.0),
        ("f8e5m2", "normal", 0.0, 30000.0)] + \
       [(dt, "raw", 0, 0) for dt in NEW_FLOATS + NEW_INTS] + \
       [("i16", "int_range", -32768, 32768), ("i16", "int_range", -7, 1000),
        ("i64", "int_range", -(2 ** 53), -(2 ** 53) + 2 ** 32), ("i64", "int_range", 5, 6)]


def test_fill_new_dtypes(ctx, oracle):
    torch = torch_cuda()
    rng = np.random.default_rng(1)
    regs = []
    for i, (dt, dist, p0, p1) in enumerate(FILL):
        nb = int(rng.choice([17, 4099, TILE + 5, 3 * TILE + 16]))
        n = max(1, nb // W.DTYPE_SIZE[dt])
        regs.append(W.Region("r%d" % i, dt, n, dist, p0, p1, int(rng.choice([0, 5, 256])),
                             int(rng.choice([0, 16, 4096])), int(rng.integers(0, 256)), i))
    nbytes = _layout(regs, skew={3: 2, 7: 8, 11: 1})
    dev = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    ctx.fill(asmv.regions_in_arena(regs, dev.data_ptr()), seed=77)
    want = oracle_fill_arena(oracle, regs, nbytes, 77)
    got = to_host(dev)
    for r in regs:
        a, b = r.offset, r.offset + r.alloc_bytes
        np.testing.assert_array_equal(got[a:b], want[a:b], err_msg="%s %s" % (r.dtype, r.dist))


def _words(arena, r):
    view = {1: np.uint8, 2: np.uint16, 8: np.uint64}[W.DTYPE_SIZE[r.dtype]]
    return arena[r.payload_offset:r.payload_offset + r.payload_bytes].view(view)


def _table(dts, seed, n_elems=3 * TILE // 8 + 37):
    rng = np.random.default_rng(seed)
    regs = [W.Region("r%d" % i, dt, n_elems + int(rng.integers(0, 9)), "raw", 0, 0, 64, 64, 0xA5, i)
            for i, dt in enumerate(dts)]
    return regs, _layout(regs, skew={1: 2})


def _candidates(ref, regs, rng, k):
    out = []
    for j in range(k):
        c = ref.copy()
        for r in regs:
            w = _words(c, r)
            flip = rng.random(w.size) < (0.3 if j % 2 else 0.02)
            w[flip] ^= w.dtype.type(1 + j)
            if W.DTYPE_SIZE[r.dtype] == 8:
                big = rng.random(w.size) < 0.01
                w[big] ^= w.dtype.type(1 << 55)
        out.append(c)
    return out


def test_compare_new_dtypes(ctx, oracle):
    dts = NEW_FLOATS + NEW_INTS
    regs, nbytes = _table(dts, 2)
    rng = np.random.default_rng(3)
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=5)           # RAW: the whole code space
    for r in regs:                                                   # special values at fixed places
        w = _words(ref, r)
        if r.dtype == "f64":
            w[:6] = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 1e308]).view(np.uint64)
        elif r.dtype.startswith("f8"):
            w[:8] = [0x00, 0x80, 0x7F, 0xFF, 0x7C, 0xFC, 0x01, 0x81]
        elif r.dtype == "i64":
            w[:4] = np.array([2 ** 63 - 1, -2 ** 63, 2 ** 53 + 1, 0], np.int64).view(np.uint64)
    cands = _candidates(ref, regs, rng, 3)
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    for tol in (W.DEFAULT_TOL, {dt: (0.5, 0.1) for dt in NEW_FLOATS},
                {dt: (0.0, 0.0) for dt in NEW_FLOATS}):
        got = ctx.compare_batched(asmv.regions_in_arena(regs, dref.data_ptr()),
                                  [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc], tol)
        for j, c in enumerate(cands):
            for i, r in enumerate(regs):
                want = oracle_region_stats(oracle, ref, r, c, r, tol, threads=4)
                assert_stats_equal(got[j][i], want, "%s cand %d" % (r.dtype, j))


def test_fnuz_and_e5m2_code_space(ctx, oracle):
    """Every (reference, candidate) pair of byte values once, per fp8 format."""
    a = np.repeat(np.arange(256, dtype=np.uint8), 256)
    b = np.tile(np.arange(256, dtype=np.uint8), 256)
    for dt in ("f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz"):
        r = W.Region("x", dt, 65536, "raw", 0, 0, 0, 0, 0xA5, 0)
        nbytes = _layout([r])
        ref = np.zeros(nbytes, np.uint8)
        cand = np.zeros(nbytes, np.uint8)
        ref[r.payload_offset:r.payload_offset + 65536] = a
        cand[r.payload_offset:r.payload_offset + 65536] = b
        dref, dc = to_device(ref), to_device(cand)
        for tol in ((1e-5, 0.25), (0.0, 0.0), (1.0, 0.0)):
            got = ctx.compare(asmv.regions_in_arena([r], dref.data_ptr()),
                              asmv.regions_in_arena([r], dc.data_ptr()), {dt: tol})
            want = oracle_region_stats(oracle, ref, r, cand, r, {dt: tol})
            assert_stats_equal(got[0], want, "%s %s" % (dt, tol))


def test_eq_sums_new_fp8(ctx, oracle):
    dts = ("f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz")
    regs, nbytes = _table(dts, 4, n_elems=3 * TILE + 99)
    for r in regs:
        r.dist, r.p0, r.p1 = "normal", 0.0, 3.0
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=8)
    rng = np.random.default_rng(5)
    cands = _candidates(ref, regs, rng, 3)
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    stats, eqs = ctx.compare_eq(asmv.regions_in_arena(regs, dref.data_ptr()),
                                [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc],
                                W.DEFAULT_TOL)
    for j, c in enumerate(cands):
        for i, r in enumerate(regs):
            st = oracle_region_stats(oracle, ref, r, c, r, W.DEFAULT_TOL)
            a = r.payload_offset
            sums = oracle.eq_sums(ref[a:a + r.payload_bytes], c[a:a + r.payload_bytes],
                                  ORACLE_DTYPE[r.dtype], r.n_elems)
            want = oracle.eq_verdict(st, sums, ORACLE_DTYPE[r.dtype])
            assert_stats_equal(eqs[j][i], want, "%s cand %d" % (r.dtype, j))


def test_restore_wide_types(ctx, oracle):
    torch = torch_cuda()
    regs, nbytes = _table(("f64", "i64", "i16"), 6)
    rng = np.random.default_rng(7)
    arena_h = rng.integers(0, 256, nbytes, dtype=np.uint8)
    snap_h = rng.integers(0, 256, nbytes, dtype=np.uint8)
    arena, snap = to_device(arena_h), to_device(snap_h)
    src = [snap.data_ptr() + r.payload_offset for r in regs]
    ctx.restore(asmv.regions_in_arena(regs, arena.data_ptr()), src)
    want = arena_h.copy()
    for r in regs:
        oracle.restore_region(want[r.offset:r.offset + r.alloc_bytes], r.payload_bytes, r.guard_lo,
                              r.guard_hi, r.canary,
                              snap_h[r.payload_offset:r.payload_offset + r.payload_bytes])
    np.testing.assert_array_equal(to_host(arena), want)
    torch.cuda.synchronize()


def test_strided_view_compare(ctx, oracle):
    """A non-contiguous fp16 view (a slice of a transposed tensor) checked
    as one region per contiguous run; each run's statistics equal the
    oracle's on the same bytes."""
    torch = torch_cuda()
    g = torch.Generator(device="cpu").manual_seed(3)
    host = torch.randn(64, 48, 40, generator=g).to(torch.float16)
    cand = host.clone()
    cand.view(-1)[::97] += 0.01
    dref, dcand = host.cuda(), cand.cuda()
    view_r = dref.transpose(0, 1)[5:40, ::2, 3:29]
    view_c = dcand.transpose(0, 1)[5:40, ::2, 3:29]
    regs_r = asmv.strided_regions(view_r.data_ptr(), view_r.shape, view_r.stride(), "f16")
    regs_c = asmv.strided_regions(view_c.data_ptr(), view_c.shape, view_c.stride(), "f16")
    assert len(regs_r) == 35 * 32
    got = ctx.compare(regs_r, regs_c, W.DEFAULT_TOL)
    hr, hc = host.numpy().view(np.uint8).ravel(), cand.numpy().view(np.uint8).ravel()
    base_r = dref.data_ptr()
    t = W.DEFAULT_TOL["f16"]
    total = 0
    for r, s in zip(regs_r, got):
        off = r.alloc - base_r
        want = oracle.compare_region(hr[off:], 0, 0, 0xA5, hc[off:], 0, 0, 0xA5, r.n_elems,
                                     ORACLE_DTYPE["f16"], t.atol, t.rtol)
        assert_stats_equal(s, want)
        total += want["mismatches"]
    assert total > 0
