"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle,
element by element and field by field, on seeded inputs that span several
tiles, ragged tails, unaligned payloads, empty and one-element regions and
guard bands longer than one guard segment."""
import zlib

import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import (assert_stats_equal, device_arena, oracle_fill_arena, oracle_region_stats,
                   to_device, to_host, torch_cuda)

pytestmark = pytest.mark.gpu

TILE = 16 * 1024


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _place(regs, align=256, skew=None):
    """Lay out allocations; `skew` maps region index -> extra byte offset
    (to make payloads unaligned)."""
    off = 0
    for i, r in enumerate(regs):
        off = (off + align - 1) // align * align + (skew or {}).get(i, 0)
        r.offset = off
        off += r.alloc_bytes
    return off + 64


FILL_CASES = [
    ("f32", "uniform", -1.0, 1.0), ("f32", "normal", 0.0, 1.0), ("bf16", "normal", 0.5, 2.0),
    ("bf16", "uniform", -3.0, 5.0), ("f16", "normal", 0.0, 0.5), ("f16", "uniform", 0.0, 1.0),
    ("f8e4m3", "normal", 0.0, 1.0), ("f8e4m3", "uniform", -600.0, 600.0),
    ("i32", "int_range", 0, 131072), ("i32", "int_range", -2 ** 31, 2 ** 31),
    ("i8", "int_range", -100, 100), ("u8", "int_range", 0, 256), ("i8", "raw", 0, 0),
    ("u8", "raw", 0, 0), ("f32", "raw", 0, 0), ("f16", "raw", 0, 0), ("i32", "raw", 0, 0),
    ("f32", "none", 0, 0),
    # widths and scales whose products are inexact: the multiply and the add round separately
    ("f32", "uniform", -2.0, 3.0), ("f32", "normal", 0.3, 1.7), ("f64", "uniform", -2.0, 3.0),
    ("f64", "normal", 0.3, 1.7), ("f16", "uniform", -2.0, 3.0), ("bf16", "normal", 0.3, 1.7),
    ("f8e4m3", "normal", 0.3, 1.7),
]


def _fill_table(seed):
    rng = np.random.default_rng(seed)
    regs = []
    sizes_bytes = [1, 7, 16, 17, 1000, 4099, TILE + 5, 3 * TILE, 100 * 1024 + 3]
    rid = 0
    for dt, dist, p0, p1 in FILL_CASES:
        for nb in rng.choice(sizes_bytes, 3, replace=False):
            n = max(1, int(nb) // W.DTYPE_SIZE[dt])
            glo, ghi = [int(x) for x in rng.choice([0, 5, 256, 4096, 5000], 2)]
            regs.append(W.Region("r%d" % rid, dt, n, dist, p0, p1, glo, ghi,
                                 int(rng.integers(0, 256)), rid))
            rid += 1
    regs.append(W.Region("empty", "f32", 0, "uniform", 0.0, 1.0, 32, 32, 0x11, rid))
    return regs


@pytest.mark.parametrize("seed", [1, 2])
def test_fill_bytes_match_oracle(ctx, oracle, seed):
    regs = _fill_table(seed)
    skew = {i: (i * 3) % 16 for i in range(0, len(regs), 4)}   # unaligned payloads too
    size = _place(regs, skew=skew)
    dev = device_arena(size, 0x3C)
    ctx.fill(asmv.regions_in_arena(regs, dev.data_ptr()), seed=1234 + seed)
    got = to_host(dev)
    want = oracle_fill_arena(oracle, regs, size, 1234 + seed,
                             base=np.full(size, 0x3C, np.uint8))
    if not np.array_equal(got, want):
        bad = np.flatnonzero(got != want)
        reg = [r.name for r in regs if r.offset <= bad[0] < r.offset + r.alloc_bytes]
        pytest.fail("%d bytes differ, first at %d (%s)" % (bad.size, bad[0], reg))


def test_fill_normal_large_region(ctx, oracle):
    """A multi-tile NORMAL bf16 region: every byte."""
    regs = [W.Region("O", "bf16", 3 * 1024 * 1024 + 3, "normal", 0.0, 1.0, 4096, 4096, 0xA5, 0)]
    size = _place(regs)
    dev = device_arena(size)
    ctx.fill(asmv.regions_in_arena(regs, dev.data_ptr()), seed=2)
    want = oracle_fill_arena(oracle, regs, size, 2)
    np.testing.assert_array_equal(to_host(dev), want)


def test_guard_check_matches_oracle(ctx, oracle):
    torch = torch_cuda()
    regs = _fill_table(7)
    size = _place(regs, skew={3: 1, 9: 7})
    dev = device_arena(size)
    ctx.fill(asmv.regions_in_arena(regs, dev.data_ptr()), seed=9)
    rng = np.random.default_rng(7)
    # damage guards (and some payload bytes, which must not count) of our own arena
    for r in regs[::3]:
        if r.guard_lo:
            dev[r.offset + int(rng.integers(0, r.guard_lo))] ^= 0xFF
        if r.guard_hi:
            k = r.guard_lo + r.payload_bytes + int(rng.integers(0, r.guard_hi))
            dev[r.offset + k] ^= 0x01
        if r.payload_bytes:
            dev[r.payload_offset] ^= 0x80
    torch.cuda.synchronize()
    got = ctx.guard_check(asmv.regions_in_arena(regs, dev.data_ptr()))
    host = to_host(dev)
    for r, g in zip(regs, got):
        bad, first = oracle.guard_check(host[r.offset:], r.payload_bytes, r.guard_lo, r.guard_hi,
                                        r.canary)
        assert (g["guard_bad_bytes"], g["first_guard_bad"]) == (bad, first), r.name
        assert g["mismatches"] == 0 and g["first_mismatch"] == asmv.U64_NONE


# ----------------------------------------------------------------- compare
CMP_DTYPES = ["f32", "bf16", "f16", "f8e4m3", "i32", "i8", "u8"]
TOL = {"f32": (1e-5, 1e-5), "bf16": (1e-2, 1.6e-2), "f16": (1e-5, 1e-3),
       "f8e4m3": (1e-5, 0.125)}


def _cmp_table(seed, n_regions=40):
    rng = np.random.default_rng(seed)
    regs = []
    for i in range(n_regions):
        dt = CMP_DTYPES[i % len(CMP_DTYPES)]
        nb = int(rng.choice([0, 1, 16, 33, 999, 4100, TILE, 2 * TILE + 7, 200 * 1024 + 1]))
        n = nb // W.DTYPE_SIZE[dt] if nb else 0
        if nb and n == 0:
            n = 1
        dist = "normal" if dt in W.FLOAT_DTYPES else "raw"
        regs.append(W.Region("c%d" % i, dt, n, dist, 0.0, 1.0, int(rng.choice([0, 256, 4100])),
                             int(rng.choice([0, 64, 4096])), 0xA5, i))
    return regs


def _perturb_host(ref_arena, regs, seed, dense=False):
    """Candidate arena: sparse and dense ULP moves, NaN/Inf/zero swaps,
    integer bit flips, guard damage."""
    import torch
    cand = torch.from_numpy(ref_arena.copy())
    rng = np.random.default_rng(seed)
    for r in regs:
        if r.n_elems == 0:
            continue
        if dense and r.dtype in W.FLOAT_DTYPES:
            W.perturb_uniform_ulps(cand, r, int(rng.integers(1 << 30)), int(rng.integers(1, 9)))
        else:
            W.perturb_sparse(cand, r, rng, rate=0.02)
        if r.dtype in W.FLOAT_DTYPES and r.n_elems > 8:
            view, tdt = W._elem_view(cand, r)
            pos = rng.choice(r.n_elems, 4, replace=False)
            specials = {"f32": [0x7FC00000, 0x7F800000, 0xFF800000, 0x80000000],
                        "bf16": [0x7FC0, 0x7F80, 0xFF80, 0x8000],
                        "f16": [0x7E00, 0x7C00, 0xFC00, 0x8000],
                        "f8e4m3": [0x7F, 0xFF, 0x80, 0x00]}[r.dtype]
            for p, v in zip(pos, specials):
                view[int(p)] = W._to_storage(torch.tensor([v]), tdt, r.dtype)[0]
        if r.guard_hi and rng.random() < 0.3:
            W.corrupt_guard(cand, r, rng, "hi")
        if r.guard_lo and rng.random() < 0.2:
            W.corrupt_guard(cand, r, rng, "lo")
    return cand.numpy()


@pytest.mark.parametrize("seed,dense", [(11, False), (12, True), (13, True)])
def test_compare_matches_oracle(ctx, oracle, seed, dense):
    regs = _cmp_table(seed)
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, seed)
    cand = _perturb_host(ref, regs, seed + 100, dense=dense)
    ref[regs[5].offset] ^= 0x40 if regs[5].guard_lo else 0     # a damaged reference guard
    dref, dcand = to_device(ref), to_device(cand)
    got = ctx.compare(asmv.regions_in_arena(regs, dref.data_ptr()),
                      asmv.regions_in_arena(regs, dcand.data_ptr()), TOL)
    for r, g in zip(regs, got):
        want = oracle_region_stats(oracle, ref, r, cand, r, TOL)
        assert_stats_equal(g, want, r.name + "/" + r.dtype)


def test_compare_unaligned_and_different_layouts(ctx, oracle):
    """Reference and candidate at different misalignments (byte path)."""
    regs = _cmp_table(21, n_regions=21)
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, 21)
    cand_regs = [W.Region(**{**r.__dict__}) for r in regs]
    for i, r in enumerate(cand_regs):
        r.guard_lo = r.guard_lo + (i % 5)                      # shifts the payload
    csize = _place(cand_regs, skew={i: i % 3 for i in range(len(cand_regs))})
    cand = np.zeros(csize, np.uint8)
    pert = _perturb_host(ref, regs, 5)
    for r, c in zip(regs, cand_regs):
        cand[c.offset:c.offset + c.guard_lo] = c.canary
        cand[c.payload_offset:c.payload_offset + c.payload_bytes] = \
            pert[r.payload_offset:r.payload_offset + r.payload_bytes]
        cand[c.payload_offset + c.payload_bytes:c.offset + c.alloc_bytes] = c.canary
    dref, dcand = to_device(ref), to_device(cand)
    got = ctx.compare(asmv.regions_in_arena(regs, dref.data_ptr()),
                      asmv.regions_in_arena(cand_regs, dcand.data_ptr()), TOL)
    for r, c, g in zip(regs, cand_regs, got):
        want = oracle_region_stats(oracle, ref, r, cand, c, TOL)
        assert_stats_equal(g, want, r.name)


def _boundary_pairs(dtype, atol, rtol, n, rng):
    """Reference values of every magnitude and candidates placed at,
    just inside and just outside atol + rtol*|r| (after rounding to the
    dtype), plus overflowing and subnormal differences."""
    import torch
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16,
           "f8e4m3": torch.float8_e4m3fn}[dtype]
    lim = {"f32": 120, "bf16": 120, "f16": 14, "f8e4m3": 7}[dtype]
    r = rng.standard_normal(n) * np.exp2(rng.integers(-lim, lim, n).astype(np.float64))
    r = torch.from_numpy(r).to(tdt).double().numpy()
    bound = atol + rtol * np.abs(r)
    f = rng.choice([1.0, 1.0 - 2 ** -20, 1.0 + 2 ** -20, 1 - 2 ** -10, 1 + 2 ** -10, 0.5, 2.0], n)
    c = r + rng.choice([-1.0, 1.0], n) * bound * f
    if dtype == "f32":
        big = rng.random(n) < 0.01
        r[big] = 3.0e38 * np.sign(rng.standard_normal(big.sum()))
        c[big] = -r[big]
    rt = torch.from_numpy(r).to(tdt)
    ct = torch.from_numpy(c).to(tdt)
    st = {"f32": torch.int32, "bf16": torch.int16, "f16": torch.int16,
          "f8e4m3": torch.uint8}[dtype]
    return (rt.view(st).numpy().view(np.uint8).copy(), ct.view(st).numpy().view(np.uint8).copy())


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16", "f8e4m3"])
@pytest.mark.parametrize("atol,rtol", [(1e-5, 1e-5), (0.0, 1e-3), (1e-3, 0.0), (0.0, 0.0),
                                       (1e-30, 2.0 ** -10), (float("inf"), 0.0)])
def test_compare_screen_boundaries(ctx, oracle, dtype, atol, rtol):
    """Candidates at the tolerance boundary exercise every branch of the
    fp32 screen; the decisions and maxima must equal the fp64 oracle."""
    rng = np.random.default_rng(zlib.crc32(repr((dtype, atol, rtol)).encode()))
    n = 50000
    R, C = _boundary_pairs(dtype, atol, rtol, n, rng)
    reg = W.Region("b", dtype, n, "raw", 0, 0, 0, 0, 0xA5, 0)
    reg.offset = 0
    dref, dcand = to_device(R), to_device(C)
    tol = {dtype: (atol, rtol)}
    got = ctx.compare([asmv.make_region(dref.data_ptr(), n, dtype)],
                      [asmv.make_region(dcand.data_ptr(), n, dtype)], tol)[0]
    want = oracle_region_stats(oracle, R, reg, C, reg, tol)
    assert_stats_equal(got, want, dtype)


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16", "f8e4m3"])
def test_compare_subnormal_differences(ctx, oracle, dtype):
    """Pairs around the smallest normal value whose differences are
    subnormal: a flush to zero anywhere would lose them."""
    import torch
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16,
           "f8e4m3": torch.float8_e4m3fn}[dtype]
    st = {"f32": torch.int32, "bf16": torch.int16, "f16": torch.int16,
          "f8e4m3": torch.uint8}[dtype]
    mn = float(torch.finfo(tdt).tiny)
    rng = np.random.default_rng(17)
    n = 4096
    r = mn * rng.uniform(1.0, 2.0, n) * rng.choice([-1, 1], n)
    c = r * (1.0 + rng.uniform(-0.3, 0.3, n))
    c[::7] = r[::7]                                   # some equal pairs
    c[3::11] = 0.5 * r[3::11]                         # subnormal values themselves
    R = torch.from_numpy(r).to(tdt).view(st).numpy().view(np.uint8).copy()
    C = torch.from_numpy(c).to(tdt).view(st).numpy().view(np.uint8).copy()
    reg = W.Region("s", dtype, n, "raw", 0, 0, 0, 0, 0xA5, 0)
    reg.offset = 0
    dref, dcand = to_device(R), to_device(C)
    for tol in [{dtype: (0.0, 0.0)}, {dtype: (0.0, 1e-3)}]:
        got = ctx.compare([asmv.make_region(dref.data_ptr(), n, dtype)],
                          [asmv.make_region(dcand.data_ptr(), n, dtype)], tol)[0]
        want = oracle_region_stats(oracle, R, reg, C, reg, tol)
        assert_stats_equal(got, want, dtype)
        assert want["mismatches"] > n // 2


@pytest.mark.parametrize("k", [1, 8])
def test_partial_tiles_of_every_shape(ctx, oracle, k):
    """Region sizes that leave the last tile of each region at every
    fraction of a tile, for the single (15 KiB tiles) and the batched
    (7.5 KiB tiles) launch; dense differences keep the exact-path queue busy."""
    rng = np.random.default_rng(100 + k)
    regs = []
    tile = 15360 if k == 1 else 7680
    for i, frac in enumerate(np.linspace(0.02, 0.98, 23)):
        dt = ["f16", "bf16", "f32", "f8e4m3", "i8"][i % 5]
        nb = tile * int(rng.integers(1, 4)) + int(frac * tile) + int(rng.integers(0, 16))
        n = max(1, nb // W.DTYPE_SIZE[dt])
        dist = "normal" if dt in W.FLOAT_DTYPES else "raw"
        regs.append(W.Region("p%d" % i, dt, n, dist, 0.0, 1.0, 256, 256, 0xA5, i))
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, 77)
    cands = [_perturb_host(ref, regs, 300 + j, dense=True) for j in range(k)]
    dref = to_device(ref)
    dcs = [to_device(c) for c in cands]
    rr = asmv.regions_in_arena(regs, dref.data_ptr())
    if k == 1:
        got = [ctx.compare(rr, asmv.regions_in_arena(regs, dcs[0].data_ptr()), TOL)]
    else:
        got = ctx.compare_batched(rr, [asmv.regions_in_arena(regs, d.data_ptr()) for d in dcs], TOL)
    for j in range(k):
        for r, g in zip(regs, got[j]):
            want = oracle_region_stats(oracle, ref, r, cands[j], r, TOL)
            assert_stats_equal(g, want, "cand %d %s" % (j, r.name))


@pytest.mark.parametrize("k", [2, 5, 6, 7, 8, 11])
def test_batched_matches_oracle(ctx, oracle, k):
    regs = _cmp_table(31, n_regions=14)
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, 31)
    cands = [_perturb_host(ref, regs, 200 + j, dense=(j % 2 == 0)) for j in range(k)]
    dref = to_device(ref)
    dcs = [to_device(c) for c in cands]
    got = ctx.compare_batched(asmv.regions_in_arena(regs, dref.data_ptr()),
                              [asmv.regions_in_arena(regs, d.data_ptr()) for d in dcs], TOL)
    for j in range(k):
        for r, g in zip(regs, got[j]):
            want = oracle_region_stats(oracle, ref, r, cands[j], r, TOL)
            assert_stats_equal(g, want, "cand %d %s" % (j, r.name))


def test_identical_candidate_is_clean(ctx):
    regs = _cmp_table(41)
    size = _place(regs)
    dev = device_arena(size)
    rr = asmv.regions_in_arena(regs, dev.data_ptr())
    ctx.fill(rr, seed=5)
    for g in ctx.compare(rr, rr, TOL):
        assert g == {"mismatches": 0, "first_mismatch": asmv.U64_NONE, "max_abs_err": 0.0,
                     "max_rel_err": 0.0, "nonfinite_mismatches": 0, "guard_bad_bytes": 0,
                     "first_guard_bad": asmv.U64_NONE, "ref_guard_bad_bytes": 0}


def test_rejects_host_memory_and_bad_tables(ctx):
    host = np.zeros(4096, np.uint8)
    bad = [asmv.make_region(host.ctypes.data, 16, "f32")]
    with pytest.raises(asmv.AsmvError) as e:
        ctx.guard_check(bad)
    assert e.value.status == asmv.EINVAL
    dev = device_arena(4096)
    ok = [asmv.make_region(dev.data_ptr(), 16, "f32", "uniform", 0, 0, 0, 0xA5, 0.0, 1.0)]
    overlap = ok + [asmv.make_region(dev.data_ptr() + 32, 16, "f32", "raw")]
    with pytest.raises(asmv.AsmvError):
        ctx.fill(overlap, seed=1)
    with pytest.raises(asmv.AsmvError):
        ctx.compare(ok, [asmv.make_region(dev.data_ptr(), 16, "f16")], TOL)
    with pytest.raises(asmv.AsmvError):
        ctx.compare(ok, ok, {"f32": (-1.0, 0.0)})
    assert ctx.compare([], [], TOL) == []


def test_radius_sqrt_matches_ieee_on_its_whole_domain(tmp_path):
    """The fill's Box-Muller radius uses its own correctly rounded square
    root; it must equal the IEEE square root on all 2^24 possible inputs."""
    import os
    import subprocess
    torch_cuda()
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    exe = str(tmp_path / "radius_sqrt_check")
    subprocess.check_call(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                           "-I", os.path.join(root, "paper_2608_20711_gb300", "csrc"), "-o", exe,
                           os.path.join(root, "tests", "helpers", "radius_sqrt_check.cu")])
    out = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stdout + out.stderr
    assert "differing 0 " in out.stdout


def test_sm_limit_changes_no_result(ctx, oracle):
    """A context whose launches are bounded to a few SMs fills the same bytes
    and finds the same statistics (the grids are persistent, their size only
    spreads the tiles differently)."""
    regs = _cmp_table(51, n_regions=6)
    size = _place(regs)
    ref = oracle_fill_arena(oracle, regs, size, 51)
    cand = _perturb_host(ref, regs, 52, dense=True)
    dref, dcand = to_device(ref), to_device(cand)
    rr = asmv.regions_in_arena(regs, dref.data_ptr())
    cr = asmv.regions_in_arena(regs, dcand.data_ptr())
    full = ctx.compare(rr, cr, TOL)
    dev = device_arena(size, 0x3C)
    try:
        ctx.set_sm_limit(5)
        small = ctx.compare(rr, cr, TOL)
        ctx.fill(asmv.regions_in_arena(regs, dev.data_ptr()), seed=51)
    finally:
        ctx.set_sm_limit(0)
    got = to_host(dev)
    want = oracle_fill_arena(oracle, regs, size, 51, base=np.full(size, 0x3C, np.uint8))
    assert np.array_equal(got, want)
    for r, a, b in zip(regs, full, small):
        assert_stats_equal(b, a, r.name)
        assert_stats_equal(a, oracle_region_stats(oracle, ref, r, cand, r, TOL), r.name)
