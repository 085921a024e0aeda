"""GPU parity of Eq. 1 on binary64 regions: the exact sums (rounded with
gradual underflow and overflow to infinity) and the scaled cosine, against
the oracle on the same bytes -- values over the whole binary64 range,
special values, ragged and unaligned payloads, empty regions, binary64
regions beside other formats, two launch groups of candidates, and a check
split over shards through the digit-vector calls."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from oracle.oracle import CODE_OF_DTYPE as ORACLE_DTYPE

from ._gpu import assert_stats_equal, oracle_region_stats, to_device, torch_cuda

pytestmark = pytest.mark.gpu

TILE64 = 2048                      # binary64 values per tile of the kernel
TOL = {"f64": (1e-9, 1e-9), "f32": (1e-5, 1e-5), "f16": (1e-5, 1e-3)}


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _layout(regs, skew):
    off = 0
    for i, r in enumerate(regs):
        off = (off + 255) // 256 * 256 + skew.get(i, 0)
        r.offset = off
        off += r.alloc_bytes
    return off + 64


def _values(kind, n, rng):
    sign = np.where(rng.random(n) < 0.5, -1.0, 1.0)
    mant = rng.uniform(1.0, 2.0, n)
    if kind == "normal":
        v = rng.standard_normal(n)
    elif kind == "full_range":
        v = sign * np.ldexp(mant, rng.integers(-1074, 1024, n))
    elif kind == "tiny":
        v = sign * np.ldexp(mant, rng.integers(-1074, -1000, n))
    elif kind == "huge":
        v = sign * np.ldexp(mant, rng.integers(900, 1024, n))
    else:
        v = sign * np.ldexp(mant, rng.integers(-40, 40, n))
    v[rng.random(n) < 0.02] = 0.0
    return v


def _put(arena, r, v):
    a = r.payload_offset
    arena[a:a + r.payload_bytes] = np.ascontiguousarray(v, np.float64).view(np.uint8)


def _get(arena, r):
    a = r.payload_offset
    return arena[a:a + r.payload_bytes].copy().view(np.float64)


def _candidate(ref, regs, rng, j):
    """The reference with ULP noise, a few large moves, and (odd j) NaN/Inf
    at new positions; even j keep the reference's specials."""
    cand = ref.copy()
    for r in regs:
        if r.n_elems == 0:
            continue
        if r.dtype != "f64":
            w = cand[r.payload_offset:r.payload_offset + r.payload_bytes]
            w[rng.random(w.size) < 0.1] ^= np.uint8(1)
            continue
        v = _get(cand, r)
        bits = v.view(np.uint64)
        flip = rng.random(v.size) < 0.3
        bits[flip] ^= np.uint64(1 + j % 5)
        big = rng.choice(v.size, size=min(v.size, 2), replace=False)
        with np.errstate(invalid="ignore"):                # a NaN may be among them
            v[big] = -0.5 * v[big]
        if j % 2 == 1:
            v[rng.choice(v.size, size=1)] = [np.nan, np.inf, -np.inf][j % 3]
        _put(cand, r, v)
    return cand


def _table(seed, sizes, kinds, extra=()):
    rng = np.random.default_rng(seed)
    regs = []
    for i, n in enumerate(sizes):
        regs.append(W.Region("d%d" % i, "f64", n, "raw", 0, 0, int(rng.choice([0, 8, 64])),
                             int(rng.choice([0, 24, 256])), 0xA5, i))
    for i, (dt, n) in enumerate(extra):
        regs.append(W.Region("x%d" % i, dt, n, "raw", 0, 0, 64, 64, 0x5A, 100 + i))
    # an unaligned binary64 payload (3 bytes off) and one off by 8 bytes
    size = _layout(regs, {1: 3, 2: 8})
    ref = rng.integers(0, 256, size, dtype=np.uint8)
    for r in regs:                 # guard bands hold the canary
        ref[r.offset:r.offset + r.guard_lo] = r.canary
        e = r.offset + r.guard_lo + r.payload_bytes
        ref[e:e + r.guard_hi] = r.canary
    for i, r in enumerate(regs):
        if r.dtype == "f64":
            v = _values(kinds[i % len(kinds)], r.n_elems, rng)
            if r.n_elems > 10 and i % 2 == 0:
                v[[1, 7]] = [np.nan, -np.inf]
            _put(ref, r, v)
        else:
            dt = np.float32 if r.dtype == "f32" else np.float16
            a = r.payload_offset
            ref[a:a + r.payload_bytes] = rng.standard_normal(r.n_elems).astype(dt).view(np.uint8)
    return regs, ref, rng


def _check(ctx, oracle, regs, ref, cands):
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    stats, eqs = ctx.compare_eq(asmv.regions_in_arena(regs, dref.data_ptr()),
                                [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc], TOL)
    for j, c in enumerate(cands):
        for i, r in enumerate(regs):
            st = oracle_region_stats(oracle, ref, r, c, r, TOL)
            assert_stats_equal(stats[j][i], st, "stats cand %d %s" % (j, r.name))
            a = r.payload_offset
            code = ORACLE_DTYPE[r.dtype]
            sums = oracle.eq_sums(ref[a:a + r.payload_bytes], c[a:a + r.payload_bytes], code,
                                  r.n_elems)
            want = oracle.eq_verdict(st, sums, code)
            assert_stats_equal(eqs[j][i], want, "eq cand %d %s" % (j, r.name))
    return eqs


@pytest.mark.parametrize("k", [1, 3, 9])
def test_eq64_matches_oracle(ctx, oracle, k):
    sizes = [1, 7, TILE64, TILE64 + 1, 3 * TILE64 + 5, 0, 20000]
    regs, ref, rng = _table(10 + k, sizes, ["normal", "full_range", "tiny", "huge", "moderate"])
    cands = [_candidate(ref, regs, rng, j) for j in range(k)]
    cands[0] = ref.copy() if k > 1 else cands[0]          # one candidate equal to the reference
    _check(ctx, oracle, regs, ref, cands)


def test_eq64_beside_other_formats(ctx, oracle):
    regs, ref, rng = _table(31, [5000, 3 * TILE64 + 17], ["normal", "full_range"],
                            extra=(("f32", 9000), ("f16", 4 * 8192 + 3)))
    cands = [_candidate(ref, regs, rng, j) for j in range(2)]
    _check(ctx, oracle, regs, ref, cands)


def test_eq64_squares_beyond_the_double_range(ctx, oracle):
    """Outputs near the ends of the binary64 range: the sums round to
    infinity or to zero, the cosine stays that of the vectors."""
    regs, ref, rng = _table(41, [4 * TILE64 + 9, 3000], ["huge", "tiny"])
    cands = [ref.copy(), _candidate(ref, regs, rng, 2)]
    eqs = _check(ctx, oracle, regs, ref, cands)
    assert eqs[0][0]["sum_rr"] == float("inf") and eqs[0][0]["cos"] > 0.9999
    assert eqs[0][1]["sum_rr"] == 0.0 and eqs[0][1]["cos"] > 0.9999


def test_eq64_many_regions(ctx, oracle):
    """Many small binary64 regions: a CTA crosses region boundaries and
    flushes each region's digits separately."""
    rng = np.random.default_rng(51)
    sizes = [int(x) for x in rng.integers(0, 700, 300)]
    regs, ref, rng = _table(52, sizes, ["normal", "moderate", "full_range"])
    cands = [_candidate(ref, regs, rng, j) for j in range(2)]
    _check(ctx, oracle, regs, ref, cands)


def test_eq64_split_over_shards_equals_whole(ctx, oracle):
    """Binary64 regions (and an fp32 and an fp16 region beside them, so
    every region takes 136 digits per sum) split into three element ranges:
    the digit vectors of asmv_compare_eq_digits summed over the shards and
    the merged statistics give, through asmv_eq_from_digits, exactly the
    result of asmv_compare_eq on the whole regions."""
    from paper_2608_20711_gb300 import distributed as D
    regs, ref, rng = _table(61, [3 * TILE64 + 77, 9000, 5], ["normal", "huge", "full_range"],
                            extra=(("f32", 7000), ("f16", 3 * 8192 + 1)))
    cands = [_candidate(ref, regs, rng, j) for j in range(3)]
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    rr = asmv.regions_in_arena(regs, dref.data_ptr())
    cc = [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc]
    whole_stats, whole_eq = ctx.compare_eq(rr, cc, TOL)
    world, digits = 3, 0
    stats = [[D.empty_stats() for _ in regs] for _ in cands]
    for rank in range(world):
        sr, firsts, shifts = [], [], []
        for i, r in enumerate(rr):
            s, first, shift = D.shard_region(r, W.DTYPE_SIZE[regs[i].dtype], rank, world)
            sr.append(s)
            firsts.append(first)
            shifts.append(shift)
        sc = [[D.shard_region(r, W.DTYPE_SIZE[regs[i].dtype], rank, world)[0] for i, r in enumerate(c)]
              for c in cc]
        st, dig = ctx.compare_eq_digits(sr, sc, TOL)
        assert dig.shape == (len(regs), 1 + 2 * len(cands), asmv.EQ64_DIGITS)
        digits = digits + D.normalize_digits(dig)
        for j in range(len(cands)):
            for i in range(len(regs)):
                stats[j][i] = D.merge_stats(stats[j][i],
                                            D.to_region_coordinates(st[j][i], firsts[i], shifts[i]))
    got = asmv.eq_from_digits([r.dtype for r in regs], stats, digits)
    for j in range(len(cands)):
        for i, r in enumerate(regs):
            where = "cand %d region %s (%s)" % (j, r.name, r.dtype)
            assert_stats_equal(stats[j][i], whole_stats[j][i], where)
            assert_stats_equal(got[j][i], whole_eq[j][i], where)
