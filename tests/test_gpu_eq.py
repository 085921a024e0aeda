"""GPU parity of Eq. 1 as a whole (asmv_compare_eq): the exact sums S_rc,
S_rr, S_cc of every float region, the cosine formed from them and the
four-term verdict, bit for bit against the oracle on the same bytes.

Inputs cover every float dtype over several tiles with a ragged tail,
candidates from one to eleven (two launch groups), values at the window
edges and outside it (the atomic path), zeros, subnormals, NaN and Inf at
matching and at mismatching positions, unaligned payloads, mixed tables
with integer regions and damaged guards, and the full-size fp16 output of
the batched GEMM workload."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from oracle.oracle import CODE_OF_DTYPE as ORACLE_DTYPE

from ._gpu import (assert_stats_equal, oracle_fill_arena, oracle_region_stats, to_device,
                   torch_cuda)

pytestmark = pytest.mark.gpu

TILE = 16 * 1024
FLOATS = ("f32", "bf16", "f16", "f8e4m3")


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _layout(regs, align=256, skew=None):
    off = 0
    for i, r in enumerate(regs):
        off = (off + align - 1) // align * align + (skew or {}).get(i, 0)
        r.offset = off
        off += r.alloc_bytes
    return off + 64


def _payload_words(arena, r):
    sz = W.DTYPE_SIZE[r.dtype]
    view = {4: np.uint32, 2: np.uint16, 1: np.uint8}[sz]
    return arena[r.payload_offset:r.payload_offset + r.payload_bytes].view(view)


def _plant_specials(arena, r, rng, frac=0.002):
    """Zeros, subnormals, extreme magnitudes, NaN and Inf in a payload."""
    w = _payload_words(arena, r)
    n = w.size
    if n == 0:
        return
    pick = lambda k: rng.choice(n, size=min(n, k), replace=False)
    k = max(1, int(n * frac))
    if r.dtype == "f32":
        specials = [0x00000000, 0x80000000, 0x00000001, 0x807FFFFF, 0x7F7FFFFF, 0xFF7FFFFF,
                    0x0DA24260, 0x72A00000, 0x7FC00000, 0x7F800000, 0xFF800000]
    elif r.dtype == "bf16":
        specials = [0x0000, 0x8000, 0x0001, 0x807F, 0x7F7F, 0xFF7F, 0x1DA2, 0x72A0,
                    0x7FC0, 0x7F80, 0xFF80]
    elif r.dtype == "f16":
        specials = [0x0000, 0x8000, 0x0001, 0x83FF, 0x7BFF, 0xFBFF, 0x7E00, 0x7C00, 0xFC00]
    else:
        specials = [0x00, 0x80, 0x01, 0x87, 0x7E, 0xFE, 0x7F, 0xFF]
    w[pick(k)] = rng.choice(np.array(specials, dtype=w.dtype), size=min(n, k))


def _perturb(cand, ref, r, rng, j):
    """Candidate j: the reference with low-bit noise, a few large moves,
    NaN/Inf copied at the same positions, and (odd j) some mismatched
    non-finite values."""
    wc, wr = _payload_words(cand, r), _payload_words(ref, r)
    n = wc.size
    if n == 0:
        return
    flip = rng.random(n) < 0.2
    wc[flip] ^= wc.dtype.type(1 + (j % 3))
    big = rng.choice(n, size=min(n, 3), replace=False)
    wc[big] ^= wc.dtype.type(1 << (8 * wc.itemsize - 3))
    if j % 2 == 1:
        wc[rng.choice(n, size=1)] = {4: 0x7FC00000, 2: 0x7E00 if r.dtype == "f16" else 0x7FC0,
                                     1: 0x7F}[wc.itemsize]
    # keep the reference's planted specials in about half of the candidates
    if j % 3 == 0:
        same = rng.random(n) < 0.5
        wc[same] = wr[same]


def _oracle_eq(oracle, ref, cand, r, tol, theta, tau, threads):
    st = oracle_region_stats(oracle, ref, r, cand, r, tol, threads=threads)
    code = ORACLE_DTYPE[r.dtype]
    if r.dtype in FLOATS:
        a = r.payload_offset
        sums = oracle.eq_sums(ref[a:a + r.payload_bytes], cand[a:a + r.payload_bytes], code,
                              r.n_elems, threads=threads)
    else:
        sums = {}
    return st, oracle.eq_verdict(st, sums, code, theta, tau)


def _check(ctx, oracle, regs, ref, cands, tol, theta=asmv.THETA, tau=asmv.TAU):
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    stats, eqs = ctx.compare_eq(asmv.regions_in_arena(regs, dref.data_ptr()),
                                [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc],
                                tol, theta, tau)
    th = oracle.host_threads()
    for j, c in enumerate(cands):
        for i, r in enumerate(regs):
            st, want = _oracle_eq(oracle, ref, c, r, tol, theta, tau, th)
            where = "cand %d region %s (%s)" % (j, r.name, r.dtype)
            assert_stats_equal(stats[j][i], st, where)
            assert_stats_equal(eqs[j][i], want, where)
    return stats, eqs


def _table(seed, dtypes=FLOATS, skew=None):
    rng = np.random.default_rng(seed)
    regs = []
    for rid, dt in enumerate(dtypes):
        sz = W.DTYPE_SIZE[dt]
        n = (3 * TILE + 4099) // sz + int(rng.integers(0, 40))
        dist = "normal" if dt in FLOATS else "int_range"
        p0, p1 = {"i32": (0, 1000), "i8": (-100, 100), "u8": (0, 256)}.get(dt, (0.0, 1.0))
        regs.append(W.Region("r%d" % rid, dt, n, dist, p0, p1, 64, 64, 0xA5, rid))
    return regs, _layout(regs, skew=skew)


@pytest.mark.parametrize("k", [1, 3, 11])
def test_eq_matches_oracle(ctx, oracle, k):
    regs, nbytes = _table(100 + k)
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=7 + k)
    rng = np.random.default_rng(k)
    for r in regs:
        _plant_specials(ref, r, rng)
    cands = []
    for j in range(k):
        c = ref.copy()
        for r in regs:
            _perturb(c, ref, r, rng, j)
        cands.append(c)
    _check(ctx, oracle, regs, ref, cands, W.DEFAULT_TOL)


def test_eq_out_of_window_values(ctx, oracle):
    """bf16 and fp32 values far from 1 (products outside the register
    window, added by the atomic path), mixed with ordinary ones."""
    regs, nbytes = _table(5, dtypes=("f32", "bf16"))
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=3)
    rng = np.random.default_rng(9)
    for r in regs:
        w = _payload_words(ref, r)
        sel = rng.random(w.size) < 0.3
        if r.dtype == "f32":
            ex = rng.integers(1, 255, sel.sum()).astype(np.uint32)
            w[sel] = (w[sel] & np.uint32(0x807FFFFF)) | (ex << np.uint32(23))
        else:
            ex = rng.integers(1, 255, sel.sum()).astype(np.uint16)
            w[sel] = (w[sel] & np.uint16(0x807F)) | (ex << np.uint16(7))
    cands = []
    for j in range(2):
        c = ref.copy()
        for r in regs:
            _perturb(c, ref, r, rng, 2 * j)     # no non-finite mismatches
        cands.append(c)
    _check(ctx, oracle, regs, ref, cands, W.DEFAULT_TOL)


def test_eq_unaligned_and_mixed_table(ctx, oracle):
    dts = ("f16", "i32", "f32", "u8", "bf16", "i8", "f8e4m3")
    regs, nbytes = _table(6, dtypes=dts, skew={0: 2, 2: 4, 4: 6, 6: 1})
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=11)
    rng = np.random.default_rng(11)
    good = ref.copy()
    bad = ref.copy()
    for r in regs:
        _perturb(bad, ref, r, rng, 2)
    bad[regs[3].offset + 1] ^= 0xFF                 # one damaged low-guard byte of the u8 region
    stats, eqs = _check(ctx, oracle, regs, ref, [good, bad], W.DEFAULT_TOL)
    assert all(e["eq"] == 1 for e in eqs[0])
    assert eqs[1][3]["flags"] & asmv.EQ_GUARD == 0
    assert eqs[1][1]["flags"] & asmv.EQ_INT == 0      # int32 payload changed


def test_eq_thresholds_decide(ctx, oracle):
    """theta and tau are passed through: the same pair passes loose
    thresholds and fails tight ones."""
    regs, nbytes = _table(8, dtypes=("f16",))
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=13)
    c = ref.copy()
    w = _payload_words(c, regs[0])
    w[::7] ^= np.uint16(0x40)                        # moves of about 2^-4 relative
    for theta, tau in ((0.9, 1.0), (0.9999999, 1.0), (0.9, 1e-6)):
        _, eqs = _check(ctx, oracle, regs, ref, [c], W.DEFAULT_TOL, theta, tau)
    assert eqs[0][0]["eq"] == 0 and eqs[0][0]["flags"] & asmv.EQ_LINF == 0


def test_eq_identical_and_empty(ctx, oracle):
    regs, nbytes = _table(9)
    regs.append(W.Region("empty", "f32", 0, "uniform", 0.0, 1.0, 16, 16, 0x11, 99))
    nbytes = _layout(regs)
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=17)
    _, eqs = _check(ctx, oracle, regs, ref, [ref.copy()], W.DEFAULT_TOL)
    for e in eqs[0]:
        assert e["eq"] == 1 and e["sum_rc"] == e["sum_rr"] == e["sum_cc"]
    assert eqs[0][-1]["cos"] == 1.0 and eqs[0][-1]["sum_rr"] == 0.0


def test_eq_rejects_bad_arguments(ctx):
    torch = torch_cuda()
    buf = torch.zeros(1 << 16, dtype=torch.uint8, device="cuda")
    reg = [asmv.make_region(buf.data_ptr(), 100, "f32")]
    for theta, tau in ((float("nan"), 1e-3), (0.9, -1.0), (0.9, float("inf"))):
        with pytest.raises(asmv.AsmvError) as e:
            ctx.compare_eq(reg, [reg], W.DEFAULT_TOL, theta, tau)
        assert e.value.status == asmv.EINVAL
    with pytest.raises(asmv.AsmvError):
        ctx.compare_eq(reg, [], W.DEFAULT_TOL)


def test_eq_batched_gemm_full(ctx, oracle):
    """The fp16 [32768, 32768] output against 8 candidates with 0..8 ULP
    noise (the bench's comparison), every Eq. 1 term against the oracle."""
    torch = torch_cuda()
    wl = W.batched_gemm()
    r = wl.regions[0]
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    dref = to_device(ref)
    cands = []
    for j in range(wl.n_cands):
        c = dref.clone()
        W.perturb_uniform_ulps(c, r, seed=wl.seed * 100 + j, magnitude=wl.ulp_magnitudes[j])
        cands.append(c)
    torch.cuda.synchronize()
    stats, eqs = ctx.compare_eq(asmv.regions_in_arena(wl.regions, dref.data_ptr()),
                                [asmv.regions_in_arena(wl.regions, c.data_ptr()) for c in cands],
                                wl.tol)
    th = oracle.host_threads()
    for j, c in enumerate(cands):
        ch = c.cpu().numpy()
        st, want = _oracle_eq(oracle, ref, ch, r, wl.tol, asmv.THETA, asmv.TAU, th)
        assert_stats_equal(stats[j][0], st, "candidate %d" % j)
        assert_stats_equal(eqs[j][0], want, "candidate %d" % j)
        del ch


def test_eq_split_over_shards_equals_whole(ctx, oracle):
    """A check split into element ranges (as processes of a multi-GPU run
    would take them): the digit vectors of asmv_compare_eq_digits summed
    over three shards and the merged statistics give, through
    asmv_eq_from_digits, exactly the result of asmv_compare_eq on the whole
    regions -- every float dtype, a mixed table, three candidates."""
    from paper_2608_20711_gb300 import distributed as D
    dts = ("f32", "bf16", "f16", "f8e4m3", "f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz", "i32", "u8")
    rng = np.random.default_rng(13)
    regs = []
    for rid, dt in enumerate(dts):
        n = (3 * TILE + 4099) // W.DTYPE_SIZE[dt] + int(rng.integers(0, 40))
        dist, p0, p1 = {"i32": ("int_range", 0, 1000), "u8": ("raw", 0, 0)}.get(dt, ("normal", 0.0, 1.0))
        regs.append(W.Region("r%d" % rid, dt, n, dist, p0, p1, 64, 64, 0xA5, rid))
    nbytes = _layout(regs)
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=12)
    for r in regs:
        if r.dtype in W.FLOAT_DTYPES:
            _plant_specials(ref, r, rng)
    cands = []
    for j in range(3):
        c = ref.copy()
        for r in regs:
            if W.DTYPE_SIZE[r.dtype] in (1, 2, 4):
                _perturb(c, ref, r, rng, j)
        cands.append(c)
    dref = to_device(ref)
    dc = [to_device(c) for c in cands]
    rr = asmv.regions_in_arena(regs, dref.data_ptr())
    cc = [asmv.regions_in_arena(regs, d.data_ptr()) for d in dc]
    whole_stats, whole_eq = ctx.compare_eq(rr, cc, W.DEFAULT_TOL)
    world = 3
    digits = 0
    stats = [[D.empty_stats() for _ in regs] for _ in cands]
    for rank in range(world):
        sr, firsts, shifts = [], [], []
        for r in rr:
            s, first, shift = D.shard_region(r, W.DTYPE_SIZE[regs[len(sr)].dtype], rank, world)
            sr.append(s)
            firsts.append(first)
            shifts.append(shift)
        sc = []
        for c in cc:
            sc.append([D.shard_region(r, W.DTYPE_SIZE[regs[i].dtype], rank, world)[0]
                       for i, r in enumerate(c)])
        st, dig = ctx.compare_eq_digits(sr, sc, W.DEFAULT_TOL)
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
