"""Host-side checks of the C ABI (no GPU needed): the library loads and
exports every function include/asmv.h declares, the ctypes layouts match
the header's, the host-only calls behave as documented (table validation,
status strings, the exact-sum rounding of Eq. 1), and with no GPU a
context cannot be created: nothing falls back to the CPU."""
import ctypes
import os
import random
import re
from fractions import Fraction

import pytest

from paper_2608_20711_gb300 import asmv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "asmv.h")


def _lib():
    from paper_2608_20711_gb300 import build
    build.build()                      # rebuilds only when a source is newer than the library
    return asmv.lib()


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return set(re.findall(r"\b(asmv_\w+)\s*\(", text)) - {"asmv_ctx"}


def test_every_declared_function_is_exported():
    L = _lib()
    declared = _declared_functions()
    assert declared == set(asmv.ABI_FUNCTIONS)
    for name in declared:
        assert hasattr(L, name), name


def test_layouts_and_version():
    text = open(HEADER).read()
    assert ctypes.sizeof(asmv.Region) == 56
    assert ctypes.sizeof(asmv.Stats) == 64
    assert ctypes.sizeof(asmv.EqResult) == 40
    ver = int(re.search(r"#define ASMV_ABI_VERSION (\d+)", text).group(1))
    assert _lib().asmv_abi_version() == ver
    assert int(re.search(r"#define ASMV_WAIT_ROUNDS (\d+)u", text).group(1)) == asmv.WAIT_ROUNDS
    assert _lib().asmv_ctx_set_wait_rounds(None, 0) == asmv.EINVAL
    for name, code in (("ASMV_EQ_COS", asmv.EQ_COS), ("ASMV_EQ_LINF", asmv.EQ_LINF),
                       ("ASMV_EQ_INT", asmv.EQ_INT), ("ASMV_EQ_GUARD", asmv.EQ_GUARD)):
        assert int(re.search(r"#define %s +(\d+)u" % name, text).group(1)) == code


def test_status_strings():
    _lib()
    for st in (asmv.OK, asmv.EINVAL, asmv.ECUDA, asmv.ETIMEOUT, asmv.ENOMEM):
        assert asmv.strerror(st)
    assert asmv.strerror(asmv.OK) != asmv.strerror(asmv.EINVAL)


def test_region_table_validation():
    _lib()
    ok = dict(alloc=1 << 20, n_elems=100, dtype="f32", dist="uniform", p0=-1.0, p1=1.0,
              guard_lo=64, guard_hi=64)
    assert asmv.check_regions([ok], for_fill=True) == asmv.OK
    bad = [dict(ok, dtype=13), dict(ok, dist=7), dict(ok, dist="int_range", p0=0, p1=5),
           dict(ok, p0=2.0, p1=1.0), dict(ok, n_elems=1 << 62), dict(ok, alloc=0)]
    for b in bad:
        assert asmv.check_regions([b], for_fill=True) == asmv.EINVAL, b
    # overlap is a fill error, not a compare error
    two = [ok, dict(ok, alloc=ok["alloc"] + 100)]
    assert asmv.check_regions(two, for_fill=True) == asmv.EINVAL
    assert asmv.check_regions(two, for_fill=False) == asmv.OK
    assert asmv.check_regions([], for_fill=True) == asmv.OK


def test_fill_order_groups_regions_by_kind():
    """The tile order of asmv_fill: a permutation of the table, grouped by
    (distribution, dtype) with RAW of any dtype one kind, table order kept
    within a kind; rejected tables leave the output untouched."""
    _lib()
    rng = random.Random(9)
    kinds = [("raw", "i8", 0, 0), ("raw", "i32", 0, 0), ("raw", "f16", 0, 0),
             ("normal", "f16", 0.0, 1.0), ("normal", "f32", 0.0, 1.0), ("normal", "bf16", 0.0, 1.0),
             ("uniform", "f16", -1.0, 1.0), ("int_range", "i32", 0, 100), ("none", "f32", 0, 0)]
    regs, addr = [], 1 << 24
    for i in range(300):
        dist, dt, p0, p1 = rng.choice(kinds)
        regs.append(dict(alloc=addr, n_elems=rng.randrange(0, 5000), dtype=dt, dist=dist, p0=p0, p1=p1,
                         guard_lo=64, guard_hi=64, region_id=i))
        addr += 64 + 4 * 5000 + 64 + 256
    order = asmv.fill_order(regs)
    assert sorted(order) == list(range(len(regs)))

    def kind(i):
        r = asmv.make_region(**regs[i])
        return (r.dist, 0 if r.dist == asmv.DIST_RAW else r.dtype)
    keys = [kind(i) for i in order]
    assert keys == sorted(keys)
    for k in set(keys):                  # stable: table order within a kind
        idx = [i for i in order if kind(i) == k]
        assert idx == sorted(idx)
    assert kind(order[0])[0] == asmv.DIST_RAW        # RAW first, every dtype together
    assert asmv.fill_order([]) == []
    with pytest.raises(asmv.AsmvError):
        asmv.fill_order([regs[0], dict(regs[0], alloc=regs[0]["alloc"] + 8)])   # overlapping


def _exact(digits, base):
    v = sum(int(d) << (32 * k) for k, d in enumerate(digits))
    return float(Fraction(v) * Fraction(2) ** base) if base >= 0 else v / (1 << -base)


def _digits_of(v, nd, rng):
    """A (non-normalised) digit vector of the integer v."""
    d = []
    for k in range(nd - 1):
        lo = v & 0xFFFFFFFF
        if rng.random() < 0.5 and k < nd - 2:          # move a random multiple up a digit
            extra = rng.randrange(-(1 << 20), 1 << 20)
            lo += extra << 32
        d.append(lo)
        v = (v - lo) >> 32
    d.append(v)
    assert all(-(1 << 63) <= x < (1 << 63) for x in d)
    return d


def test_exact_to_double_random_and_ties():
    _lib()
    rng = random.Random(5)
    nd, base = 20, -318
    cases = [0, 1, -1, 1 << 300, -(1 << 300) + 1]
    for _ in range(400):
        bits = rng.randrange(1, 600)
        cases.append(rng.choice([-1, 1]) * rng.getrandbits(bits))
    # exact ties: (2^53 + odd/even) * 2^s + half, with and without sticky bits
    for s in (0, 7, 100, 400):
        for m in ((1 << 53) + 1, (1 << 53) + 2, (1 << 54) - 1):
            half = 1 << s
            for extra in (0, 1):
                v = (m << (s + 1)) + half + (extra if s > 0 else 0)
                cases += [v, -v]
    for v in cases:
        d = _digits_of(v, nd, rng)
        assert asmv.exact_to_double(d, base) == _exact(d, base), v


def test_exact_to_double_rejects_bad_arguments():
    _lib()
    with pytest.raises(asmv.AsmvError):
        asmv.exact_to_double([], -318)
    with pytest.raises(asmv.AsmvError):
        asmv.exact_to_double([1] * 65, 0)
    with pytest.raises(asmv.AsmvError):
        asmv.exact_to_double([1], 1200)        # beyond the double range


def test_no_gpu_means_no_context():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    _lib()
    with pytest.raises(asmv.AsmvError):
        asmv.Context(0)


def test_strided_regions_cover_each_element_once():
    """The regions of a strided view cover exactly its elements' bytes."""
    import numpy as np
    base = 1 << 30
    a = np.zeros((6, 10, 12), np.float16)
    for view in (a, a[:, 2:9, :], a[::2, :, 3:7], a.transpose(1, 0, 2)[:, :, ::3], a[:, :, 5]):
        strides = [s // a.itemsize for s in view.strides]
        off0 = (view.__array_interface__["data"][0] - a.__array_interface__["data"][0]) // 2
        regs = asmv.strided_regions(base + 2 * off0, view.shape, strides, "f16")
        covered = []
        for r in regs:
            start = (r.alloc - base) // 2
            covered.extend(range(start, start + r.n_elems))
        idx = np.arange(a.size).reshape(a.shape)
        # element offsets of the view, in row-major order of the view
        view_idx = np.lib.stride_tricks.as_strided(idx.ravel()[off0:], view.shape,
                                                   [s // 2 * 8 for s in view.strides])
        assert covered == view_idx.ravel().tolist()
        assert len(regs) <= view.size


def test_candidate_tables_must_match_the_reference_length():
    """Every wrapper refuses a candidate table of another length before it
    reaches the C call, which would read n candidate regions."""
    ref = [asmv.make_region(0x10000, 8, "f32"), asmv.make_region(0x20000, 8, "f32")]
    short = ref[:1]
    with pytest.raises(ValueError):
        asmv.compare_noalloc(ref, short, {"f32": (0.0, 0.0)})
    ctx = asmv.Context.__new__(asmv.Context)          # no device needed: the check comes first
    with pytest.raises(ValueError):
        ctx.compare(ref, short, {"f32": (0.0, 0.0)})
    with pytest.raises(ValueError):
        ctx.compare_batched(ref, [ref, short], {"f32": (0.0, 0.0)})
    with pytest.raises(ValueError):
        ctx.compare_eq(ref, [short], {"f32": (0.0, 0.0)})
    with pytest.raises(ValueError):
        ctx.compare_eq_digits(ref, [ref + ref], {"f32": (0.0, 0.0)})


def test_debug_bounds_build_exports_the_same_calls():
    """libasmv_debug.so (the same sources with device bounds checks) exports
    every declared call and says which build it is; the widening hook exists
    only there."""
    from paper_2608_20711_gb300 import build
    path = build.build(debug_bounds=True)
    D = ctypes.CDLL(path)
    for name in _declared_functions():
        assert hasattr(D, name), name
    L = _lib()
    assert D.asmv_debug_bounds() == 1
    assert L.asmv_debug_bounds() == 0
    D.asmv_ctx_debug_widen.argtypes = [ctypes.c_void_p, ctypes.c_uint64]
    assert D.asmv_ctx_debug_widen(None, 0) == asmv.EINVAL
    assert L.asmv_ctx_debug_widen(None, 0) == asmv.EINVAL
    D.asmv_strerror.restype = ctypes.c_char_p
    assert b"allocation" in D.asmv_strerror(asmv.EBOUNDS)


def test_gpu_test_helpers_compile(tmp_path):
    """The CUDA helper that the GPU tests build against the fill's headers
    still compiles for sm_103a (compile only: no GPU here)."""
    import shutil
    import subprocess
    if shutil.which("nvcc") is None:
        pytest.skip("nvcc not on PATH")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    subprocess.check_call(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-c",
                           "-I", os.path.join(root, "paper_2608_20711_gb300", "csrc"),
                           "-o", str(tmp_path / "radius_sqrt_check.o"),
                           os.path.join(root, "tests", "helpers", "radius_sqrt_check.cu")])
