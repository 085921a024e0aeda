"""Pins of the oracle's equivalence check (AsmEvo Sec. 3.2 Eq. 1, restated
per element; Sec. 3.4 Tier 2: floats within tolerance, integers, opaque
bytes and guards bit-exact).

Expected values come from torch.isclose (the library predicate), from
closed forms, from the ground truth of a construction, or from invariants;
none is produced by the oracle itself."""
import zlib

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_20711_gb300 import workloads as W  # noqa: E402

TDT = {"F32": torch.float32, "BF16": torch.bfloat16, "F16": torch.float16,
       "F8E4M3": torch.float8_e4m3fn}
STORE = {"F32": torch.int32, "BF16": torch.int16, "F16": torch.int16,
         "F8E4M3": torch.uint8}


def _raw(t, name):
    return t.view(STORE[name]).numpy().view(np.uint8).copy()


def _cmp(o, ref, cand, code, atol, rtol):
    n = ref.size // o.DTYPE_SIZE[code]
    return o.compare_range(ref, cand, code, 0, n, atol, rtol)


def _special_values(name):
    v = [0.0, -0.0, 1.0, -1.0, float("inf"), float("-inf"), float("nan"), 1e-3, 2.5, -7.0]
    if name == "F8E4M3":
        v = [x for x in v if not np.isinf(x)]
    return v


@pytest.mark.parametrize("name", ["F32", "BF16", "F16", "F8E4M3"])
@pytest.mark.parametrize("atol,rtol", [(1e-5, 1e-5), (1e-2, 1.6e-2), (0.0, 1e-3), (1e-3, 0.0)])
def test_predicate_matches_torch_isclose(oracle, name, atol, rtol):
    code = getattr(oracle, name)
    rng = np.random.default_rng(zlib.crc32(repr((name, atol, rtol)).encode()))
    n = 1 << 16
    r64 = rng.standard_normal(n) * np.exp2(rng.integers(-8, 8, n))
    # candidates: exact copies, near the tolerance boundary, far, and specials
    bound = atol + rtol * np.abs(r64)
    c64 = r64 + rng.choice([-1, 1], n) * bound * rng.choice([0.0, 0.5, 0.999, 1.0, 1.001, 3.0], n)
    sv = _special_values(name)
    k = 4096
    r64[:k] = rng.choice(sv, k)
    c64[:k] = rng.choice(sv, k)
    rt = torch.from_numpy(r64).to(TDT[name])
    ct = torch.from_numpy(c64).to(TDT[name])
    got = _cmp(oracle, _raw(rt, name), _raw(ct, name), code, atol, rtol)
    close = torch.isclose(ct.double(), rt.double(), rtol=rtol, atol=atol, equal_nan=True).numpy()
    bad = np.flatnonzero(~close)
    assert got["mismatches"] == bad.size
    assert got["first_mismatch"] == (bad[0] if bad.size else oracle.U64_NONE)
    # NaN/Inf-position mismatches: a non-finite on either side that isclose rejects
    rd, cd = rt.double().numpy(), ct.double().numpy()
    nonfin = ~(np.isfinite(rd) & np.isfinite(cd))
    assert got["nonfinite_mismatches"] == int((nonfin & ~close).sum())
    # maxima over finite pairs (numpy's own abs/divide in fp64)
    fin = ~nonfin
    d = np.abs(cd[fin] - rd[fin])
    assert got["max_abs_err"] == d.max()
    with np.errstate(divide="ignore", invalid="ignore"):
        rel = np.where(rd[fin] != 0, d / np.abs(rd[fin]), np.where(d == 0, 0.0, np.inf))
    assert got["max_rel_err"] == rel.max()


@pytest.mark.parametrize("code", range(7))
def test_identical_buffers_have_zero_stats(oracle, code):
    """compare(x, x): random bit patterns, NaN and Inf included."""
    n = 5000
    x = np.zeros(n * oracle.DTYPE_SIZE[code], np.uint8)
    oracle.fill_payload(x, code, oracle.RAW, 0, n, 3, 0, 0, 42)
    got = _cmp(oracle, x, x.copy(), code, 1e-5, 1e-5)
    assert got == {"mismatches": 0, "first_mismatch": oracle.U64_NONE, "max_abs_err": 0.0,
                   "max_rel_err": 0.0, "nonfinite_mismatches": 0}


def test_closed_forms_fp32(oracle):
    def one(r, c, atol=0.0, rtol=0.0):
        R = np.array([r], np.float32).view(np.uint8)
        C = np.array([c], np.float32).view(np.uint8)
        return _cmp(oracle, R, C, oracle.F32, atol, rtol)
    s = one(1.0, 1.0 + 2.0 ** -23)
    assert (s["max_abs_err"], s["max_rel_err"], s["mismatches"]) == (2.0 ** -23, 2.0 ** -23, 1)
    s = one(1.0, 1.0 + 2.0 ** -23, atol=2.0 ** -23)            # equality with the bound passes
    assert s["mismatches"] == 0
    s = one(1.0, 1.0 + 2.0 ** -23, rtol=2.0 ** -23)
    assert s["mismatches"] == 0
    s = one(2.0 ** -126, 2.0 ** -126 + 2.0 ** -149)             # subnormal step
    assert (s["max_abs_err"], s["max_rel_err"]) == (2.0 ** -149, 2.0 ** -23)
    s = one(0.0, -0.0)
    assert (s["mismatches"], s["max_abs_err"], s["max_rel_err"]) == (0, 0.0, 0.0)
    s = one(0.0, 1e-30, atol=1.0)                               # within atol, rel undefined
    assert s["mismatches"] == 0 and s["max_rel_err"] == np.inf
    s = one(3e38, -3e38, atol=1.0)                              # overflows fp32, not fp64
    assert s["max_abs_err"] == 2 * float(np.float32(3e38)) and s["mismatches"] == 1
    s = one(float("nan"), 1.0)
    assert (s["mismatches"], s["nonfinite_mismatches"], s["max_abs_err"]) == (1, 1, 0.0)
    s = one(float("inf"), float("inf"))
    assert s["mismatches"] == 0
    s = one(float("inf"), float("-inf"))
    assert (s["mismatches"], s["nonfinite_mismatches"]) == (1, 1)


def test_closed_forms_f16_extremes(oracle):
    R = np.array([65504.0, 2.0 ** -24, 1.0], np.float16).view(np.uint8)
    C = np.array([-65504.0, -2.0 ** -24, 1.0], np.float16).view(np.uint8)
    s = _cmp(oracle, R, C, oracle.F16, 0.0, 0.0)
    assert s["max_abs_err"] == 131008.0 and s["max_rel_err"] == 2.0
    assert (s["mismatches"], s["first_mismatch"]) == (2, 0)


def test_integers_closed_forms(oracle):
    r = np.array([0, 5, -7, 2 ** 31 - 1, -2 ** 31], np.int32)
    c = r.copy()
    c[1] ^= 1 << 3                                    # 5 -> 13: |d| = 8, rel 8/5
    c[4] ^= np.int32(-2 ** 31)                       # sign bit flip: |d| = 2^31
    s = _cmp(oracle, r.view(np.uint8), c.view(np.uint8), oracle.I32, 1e9, 1e9)
    assert (s["mismatches"], s["first_mismatch"]) == (2, 1)   # tolerances never apply to ints
    assert s["max_abs_err"] == 2.0 ** 31 and s["max_rel_err"] == 8 / 5
    r8 = np.array([0, 200, 7], np.uint8)
    c8 = np.array([1, 200, 7], np.uint8)
    s = _cmp(oracle, r8, c8, oracle.U8, 0, 0)
    assert (s["mismatches"], s["max_abs_err"], s["max_rel_err"]) == (1, 1.0, np.inf)
    s = _cmp(oracle, r8, c8, oracle.I8, 0, 0)      # same bytes as signed: 200 -> -56
    assert s["mismatches"] == 1


def test_brute_force_single_element_perturbations(oracle):
    """Every position of a small fp16 array, replaced in turn by each value
    of a set: exactly that element decides every statistic."""
    ref = np.array([0.5, -1.0, 3.0, 0.0, 1e-4, -0.25, 7.5, 100.0, -2.0, 0.125, 1.0, -0.0],
                   np.float16)
    repl = np.array([0.5001, -1.0, 3.002, 1e-3, np.nan, np.inf, -0.0, 1e-7, 65504, -3.0],
                    np.float16)
    atol, rtol = 1e-3, 1e-3
    for i in range(ref.size):
        for v in repl:
            cand = ref.copy()
            cand[i] = v
            got = _cmp(oracle, ref.view(np.uint8), cand.view(np.uint8), oracle.F16, atol, rtol)
            rt, ct = torch.from_numpy(ref.astype(np.float64)), torch.from_numpy(cand.astype(np.float64))
            close = torch.isclose(ct, rt, rtol=rtol, atol=atol, equal_nan=True).numpy()
            assert close[np.arange(ref.size) != i].all()
            want_mis = 0 if close[i] else 1
            assert got["mismatches"] == want_mis
            assert got["first_mismatch"] == (i if want_mis else oracle.U64_NONE)
            r, c = float(ref[i]), float(v)
            if np.isfinite(c):
                d = abs(c - r)
                assert got["max_abs_err"] == d
                assert got["max_rel_err"] == (d / abs(r) if r != 0 else (0.0 if d == 0 else np.inf))
                assert got["nonfinite_mismatches"] == 0
            else:
                assert got["max_abs_err"] == 0.0 and got["nonfinite_mismatches"] == 1


@pytest.mark.parametrize("code", [0, 1, 2, 3, 4, 5, 6])
def test_range_split_and_merge_invariance(oracle, code):
    n = 20000
    sz = oracle.DTYPE_SIZE[code]
    ref = np.zeros(n * sz, np.uint8)
    oracle.fill_payload(ref, code, oracle.RAW, 0, n, 1, 0, 0, 5)
    cand = ref.copy()
    rng = np.random.default_rng(code)
    cand[rng.choice(ref.size, 300, replace=False)] ^= 0x10
    whole = _cmp(oracle, ref, cand, code, 1e-3, 1e-3)
    cuts = [0, *np.sort(rng.choice(np.arange(1, n), 9, replace=False)), n]
    parts = [oracle.compare_range(ref, cand, code, int(a), int(b), 1e-3, 1e-3)
             for a, b in zip(cuts[:-1], cuts[1:])]
    rng.shuffle(parts)
    assert oracle.merge_partials(parts) == whole
    assert whole["mismatches"] > 0


def _host_fill(o, wl, threads=4):
    code = {n: getattr(o, n.upper()) for n in W.DTYPES}
    dist = {n: getattr(o, n.upper()) for n in W.DISTS}
    arena = np.zeros(wl.arena_bytes, np.uint8)
    for r in wl.regions:
        o.fill_region(arena[r.offset:r.offset + r.alloc_bytes], r.n_elems, code[r.dtype],
                      dist[r.dist], r.guard_lo, r.guard_hi, r.region_id, r.canary,
                      r.p0, r.p1, wl.seed, threads=threads)
    return arena, code


def _region_stats(o, wl, ref, cand, r, code):
    t = wl.tol.get(r.dtype, W.Tolerance(0.0, 0.0))
    return o.compare_region(ref[r.offset:], r.guard_lo, r.guard_hi, r.canary,
                            cand[r.offset:], r.guard_lo, r.guard_hi, r.canary,
                            r.n_elems, code[r.dtype], t.atol, t.rtol)


def test_fp32_workload_ground_truth(oracle):
    """37 seeded perturbations (20 inside tolerance, 15 outside, one NaN,
    one +Inf) and one overwritten guard byte: the counts are known from the
    construction."""
    wl = W.fp32_single()
    ref, code = _host_fill(oracle, wl)
    cand_t = torch.from_numpy(ref.copy())
    truth = W.perturb_fp32_single(cand_t, wl)
    cand = cand_t.numpy()
    s = _region_stats(oracle, wl, ref, cand, wl.regions[0], code)
    assert s["mismatches"] == truth["mismatches"] == 17
    assert s["nonfinite_mismatches"] == 2
    assert s["first_mismatch"] == truth["first_mismatch"]
    assert (s["guard_bad_bytes"], s["first_guard_bad"]) == (1, truth["first_guard_bad"])
    assert s["ref_guard_bad_bytes"] == 0
    # the values are U[-1,1): 15 out-of-tolerance moves of >= 2*bound set the max
    assert 2e-5 < s["max_abs_err"] < 0.01


def test_int_workload_ground_truth(oracle):
    """One flipped bit per region: exactly one mismatch at that index with
    |delta| = 2^bit (the sign bit of two's complement included)."""
    wl = W.int_exact(scale=16)
    ref, code = _host_fill(oracle, wl)
    cand_t = torch.from_numpy(ref.copy())
    rng = np.random.default_rng(3)
    flips = [W.flip_bit(cand_t, r, rng) for r in wl.regions]
    cand = cand_t.numpy()
    for r, (i, bit) in zip(wl.regions, flips):
        s = _region_stats(oracle, wl, ref, cand, r, code)
        assert (s["mismatches"], s["first_mismatch"]) == (1, i)
        assert s["max_abs_err"] == 2.0 ** bit
        assert s["guard_bad_bytes"] == 0 and s["nonfinite_mismatches"] == 0


def test_region_order_does_not_matter(oracle):
    wl = W.snapshot(n_regions=24, total_bytes=1 << 20, seed=11)
    ref, code = _host_fill(oracle, wl)
    cand_t = torch.from_numpy(ref.copy())
    rng = np.random.default_rng(0)
    for r in wl.regions:
        W.perturb_sparse(cand_t, r, rng, rate=1e-2)
    cand = cand_t.numpy()
    a = [_region_stats(oracle, wl, ref, cand, r, code) for r in wl.regions]
    perm = rng.permutation(len(wl.regions))
    b = {int(k): _region_stats(oracle, wl, ref, cand, wl.regions[k], code) for k in perm}
    assert all(a[k] == b[k] for k in range(len(a)))
    assert sum(x["mismatches"] for x in a) > 0
