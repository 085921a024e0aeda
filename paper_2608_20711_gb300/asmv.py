"""ctypes binding of the C ABI in include/asmv.h (argument marshalling only).

Every step of the fill, guard check and comparison runs in the CUDA
kernels of libasmv.so; this module converts Python region descriptions to
the C structs, passes raw device addresses and a CUDA stream handle, and
turns status codes into exceptions.  There is no fallback: if the library
is missing or the GPU is absent, calls fail loudly.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Iterable, List, Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
# ASMV_DEBUG_BOUNDS=1 in the environment loads the debug-bounds build
# (libasmv_debug.so: every device access checked against its allocation).
DEBUG_BOUNDS = os.environ.get("ASMV_DEBUG_BOUNDS", "0") not in ("", "0")
LIB_PATH = os.path.join(HERE, "libasmv_debug.so" if DEBUG_BOUNDS else "libasmv.so")

# asmv_dtype / asmv_dist codes
F32, BF16, F16, F8E4M3, I32, I8, U8_OPAQUE = range(7)
F8E5M2, F8E4M3FNUZ, F8E5M2FNUZ, F64, I16, I64 = range(7, 13)
NDTYPES = 13
DIST_RAW, DIST_UNIFORM, DIST_NORMAL, DIST_INT_RANGE, DIST_NONE = range(5)
DTYPE_CODE = {"f32": F32, "bf16": BF16, "f16": F16, "f8e4m3": F8E4M3, "i32": I32,
              "i8": I8, "u8": U8_OPAQUE, "f8e5m2": F8E5M2, "f8e4m3fnuz": F8E4M3FNUZ,
              "f8e5m2fnuz": F8E5M2FNUZ, "f64": F64, "i16": I16, "i64": I64}
DIST_CODE = {"raw": DIST_RAW, "uniform": DIST_UNIFORM, "normal": DIST_NORMAL,
             "int_range": DIST_INT_RANGE, "none": DIST_NONE}
OK, EINVAL, ECUDA, ETIMEOUT, ENOMEM, EBOUNDS = 0, -1, -2, -3, -4, -5


def dtype_code(dtype) -> int:
    """The ABI code of a dtype name (or a code, returned as is)."""
    return DTYPE_CODE[dtype] if isinstance(dtype, str) else int(dtype)


U64_NONE = (1 << 64) - 1


class Region(ctypes.Structure):
    """asmv_region (56 bytes)."""
    _fields_ = [("alloc", ctypes.c_uint64), ("n_elems", ctypes.c_uint64),
                ("dtype", ctypes.c_uint32), ("dist", ctypes.c_uint32),
                ("guard_lo", ctypes.c_uint32), ("guard_hi", ctypes.c_uint32),
                ("region_id", ctypes.c_uint32), ("canary", ctypes.c_uint8),
                ("pad_", ctypes.c_uint8 * 3), ("p0", ctypes.c_double), ("p1", ctypes.c_double)]


class Tol(ctypes.Structure):
    _fields_ = [("atol", ctypes.c_double), ("rtol", ctypes.c_double)]


class Stats(ctypes.Structure):
    """asmv_stats (64 bytes)."""
    _fields_ = [("mismatches", ctypes.c_uint64), ("first_mismatch", ctypes.c_uint64),
                ("max_abs_err", ctypes.c_double), ("max_rel_err", ctypes.c_double),
                ("nonfinite_mismatches", ctypes.c_uint64), ("guard_bad_bytes", ctypes.c_uint64),
                ("first_guard_bad", ctypes.c_uint64), ("ref_guard_bad_bytes", ctypes.c_uint64)]


class EqResult(ctypes.Structure):
    """asmv_eq (40 bytes): the Eq. 1 terms of one region."""
    _fields_ = [("sum_rc", ctypes.c_double), ("sum_rr", ctypes.c_double),
                ("sum_cc", ctypes.c_double), ("cos", ctypes.c_double),
                ("flags", ctypes.c_uint32), ("eq", ctypes.c_uint32)]


class Timing(ctypes.Structure):
    """asmv_timing (32 bytes)."""
    _fields_ = [("median_ms", ctypes.c_double), ("mean_ms", ctypes.c_double),
                ("cv", ctypes.c_double), ("r", ctypes.c_uint64)]


class GateParams(ctypes.Structure):
    _fields_ = [("eps", ctypes.c_double), ("k", ctypes.c_double), ("s_floor", ctypes.c_double)]


GATE_EPS, GATE_K, GATE_S_FLOOR = 0.002, 0.85, 1.0     # Eq. 2 constants used in the paper (Sec. 5)
LAUNCH_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p)

STATS_FIELDS = [f for f, _ in Stats._fields_]
EQ_FIELDS = [f for f, _ in EqResult._fields_]
EQ_COS, EQ_LINF, EQ_INT, EQ_GUARD = 1, 2, 4, 8
THETA, TAU = 0.9999, 1e-3          # Eq. 1 thresholds used in the paper (Sec. 5)
assert ctypes.sizeof(Region) == 56 and ctypes.sizeof(Stats) == 64
assert ctypes.sizeof(EqResult) == 40

ABI_FUNCTIONS = ("asmv_ctx_create", "asmv_ctx_destroy", "asmv_fill", "asmv_guard_check",
                 "asmv_compare", "asmv_compare_batched", "asmv_check_regions",
                 "asmv_ctx_set_timing", "asmv_ctx_kernel_ms", "asmv_ctx_cuda_error",
                 "asmv_ctx_launches", "asmv_strerror", "asmv_abi_version",
                 "asmv_compare_noalloc", "asmv_compare_eq", "asmv_exact_to_double",
                 "asmv_timing_summary", "asmv_commit_gate", "asmv_time_launches",
                 "asmv_restore", "asmv_capture", "asmv_va_granularity", "asmv_va_map",
                 "asmv_va_address", "asmv_va_size", "asmv_va_unmap", "asmv_ctx_set_wait_rounds",
                 "asmv_compare_eq_digits", "asmv_eq_from_digits", "asmv_eq_digit_base",
                 "asmv_debug_bounds", "asmv_ctx_debug_widen", "asmv_ctx_set_sm_limit",
                 "asmv_fill_order")
EQ_DIGITS = 20                           # signed 64-bit digits per exact Eq. 1 sum
EQ64_DIGITS = 136                        # ... when the region table holds a binary64 region
NOALLOC_SCRATCH_BYTES = 1 << 20
WAIT_ROUNDS = 20000                      # default bound of the compare's device waits


class AsmvError(RuntimeError):
    def __init__(self, status: int, message: str, cuda_error: int = 0):
        super().__init__("asmv status %d (%s)%s" % (
            status, message, ", cudaError %d" % cuda_error if cuda_error else ""))
        self.status = status
        self.cuda_error = cuda_error


_lib = None


def lib():
    """Load libasmv.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("%s is not built: run paper_2608_20711_gb300.build.build(%s)"
                               % (os.path.basename(LIB_PATH), "debug_bounds=True" if DEBUG_BOUNDS else ""))
        L = ctypes.CDLL(LIB_PATH)
        vp, sz = ctypes.c_void_p, ctypes.c_size_t
        RP, SP, TP = ctypes.POINTER(Region), ctypes.POINTER(Stats), ctypes.POINTER(Tol)
        L.asmv_ctx_create.argtypes = [ctypes.POINTER(vp), ctypes.c_int]
        L.asmv_ctx_destroy.argtypes = [vp]
        L.asmv_ctx_destroy.restype = None
        L.asmv_fill.argtypes = [vp, RP, sz, ctypes.c_uint64, vp]
        L.asmv_guard_check.argtypes = [vp, RP, sz, SP, vp]
        L.asmv_compare.argtypes = [vp, RP, RP, sz, TP, SP, vp]
        L.asmv_compare_batched.argtypes = [vp, RP, ctypes.POINTER(RP), sz, sz, TP, SP, vp]
        L.asmv_check_regions.argtypes = [RP, sz, ctypes.c_int]
        L.asmv_fill_order.argtypes = [RP, sz, ctypes.POINTER(ctypes.c_uint32)]
        L.asmv_ctx_set_timing.argtypes = [vp, ctypes.c_int]
        L.asmv_ctx_kernel_ms.argtypes = [vp, ctypes.POINTER(ctypes.c_float)]
        L.asmv_ctx_cuda_error.argtypes = [vp]
        L.asmv_ctx_launches.argtypes = [vp]
        L.asmv_ctx_launches.restype = ctypes.c_uint64
        L.asmv_ctx_set_wait_rounds.argtypes = [vp, ctypes.c_uint32]
        L.asmv_debug_bounds.argtypes = []
        L.asmv_ctx_set_sm_limit.argtypes = [vp, ctypes.c_int]
        L.asmv_ctx_debug_widen.argtypes = [vp, ctypes.c_uint64]
        L.asmv_strerror.argtypes = [ctypes.c_int]
        L.asmv_strerror.restype = ctypes.c_char_p
        L.asmv_abi_version.argtypes = []
        L.asmv_compare_noalloc.argtypes = [RP, RP, sz, TP, SP, vp]
        L.asmv_compare_eq.argtypes = [vp, RP, ctypes.POINTER(RP), sz, sz, TP, ctypes.c_double,
                                      ctypes.c_double, SP, ctypes.POINTER(EqResult), vp]
        i64p = ctypes.POINTER(ctypes.c_int64)
        L.asmv_compare_eq_digits.argtypes = [vp, RP, ctypes.POINTER(RP), sz, sz, TP, SP, i64p, vp]
        L.asmv_eq_from_digits.argtypes = [ctypes.POINTER(ctypes.c_uint32), sz, sz, SP, i64p,
                                          ctypes.c_double, ctypes.c_double, ctypes.POINTER(EqResult)]
        L.asmv_eq_digit_base.argtypes = [ctypes.c_uint32, ctypes.POINTER(ctypes.c_int)]
        L.asmv_exact_to_double.argtypes = [ctypes.POINTER(ctypes.c_int64), ctypes.c_int,
                                           ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
        dp = ctypes.POINTER(ctypes.c_double)
        L.asmv_timing_summary.argtypes = [dp, sz, ctypes.POINTER(Timing)]
        L.asmv_commit_gate.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_double,
                                       ctypes.c_double, ctypes.POINTER(GateParams), dp,
                                       ctypes.POINTER(ctypes.c_int)]
        L.asmv_time_launches.argtypes = [LAUNCH_FN, vp, ctypes.c_int, sz, dp, vp,
                                         ctypes.POINTER(ctypes.c_int)]
        u64p = ctypes.POINTER(ctypes.c_uint64)
        L.asmv_restore.argtypes = [vp, RP, u64p, sz, vp]
        L.asmv_capture.argtypes = [vp, RP, u64p, sz, vp]
        L.asmv_va_granularity.argtypes = [ctypes.c_int, ctypes.POINTER(sz)]
        L.asmv_va_map.argtypes = [ctypes.c_int, ctypes.c_uint64, sz, ctypes.POINTER(vp)]
        L.asmv_va_address.argtypes = [vp]
        L.asmv_va_address.restype = ctypes.c_uint64
        L.asmv_va_size.argtypes = [vp]
        L.asmv_va_size.restype = sz
        L.asmv_va_unmap.argtypes = [vp]
        _lib = L
    return _lib


def strerror(status: int) -> str:
    return lib().asmv_strerror(status).decode()


def region_array(regions: Sequence) -> ctypes.Array:
    """ctypes array of Region from Region instances or dicts."""
    arr = (Region * max(1, len(regions)))()
    for i, r in enumerate(regions):
        if isinstance(r, Region):
            arr[i] = r
        else:
            arr[i] = make_region(**r)
    return arr


def make_region(alloc: int, n_elems: int, dtype, dist="raw", guard_lo=0, guard_hi=0,
                region_id=0, canary=0xA5, p0=0.0, p1=0.0) -> Region:
    r = Region()
    r.alloc = int(alloc)
    r.n_elems = int(n_elems)
    r.dtype = DTYPE_CODE[dtype] if isinstance(dtype, str) else int(dtype)
    r.dist = DIST_CODE[dist] if isinstance(dist, str) else int(dist)
    r.guard_lo = int(guard_lo)
    r.guard_hi = int(guard_hi)
    r.region_id = int(region_id)
    r.canary = int(canary)
    r.p0 = float(p0)
    r.p1 = float(p1)
    return r


def regions_in_arena(specs: Iterable, base: int) -> List[Region]:
    """Regions of workload specs (objects with dtype, n_elems, dist, p0, p1,
    guard_lo, guard_hi, canary, region_id, offset) placed at `base`."""
    return [make_region(base + s.offset, s.n_elems, s.dtype, s.dist, s.guard_lo, s.guard_hi,
                        s.region_id, s.canary, s.p0, s.p1) for s in specs]


def strided_regions(base: int, shape: Sequence[int], strides: Sequence[int], dtype,
                    region_id0: int = 0, canary: int = 0xA5) -> List[Region]:
    """A non-contiguous tensor (element strides, row-major shape) as one
    region per contiguous run of its innermost dimension(s): runs are merged
    while the strides are those of a contiguous block.  Region ids count up
    from region_id0 in row-major order; no guard bands (the gaps between runs
    belong to other data)."""
    shape, strides = list(shape), list(strides)
    if len(shape) != len(strides) or any(n < 0 for n in shape):
        raise ValueError("shape and strides must have the same length")
    code = DTYPE_CODE[dtype] if isinstance(dtype, str) else int(dtype)
    size = [4, 2, 2, 1, 4, 1, 1, 1, 1, 1, 8, 2, 8][code]
    if 0 in shape:
        return []
    # innermost dimensions that form one contiguous run
    run, k = 1, len(shape)
    while k > 0 and strides[k - 1] == run:
        run *= shape[k - 1]
        k -= 1
    if k == len(shape):               # innermost stride not 1: runs of one element
        run = 1
    outer = shape[:k]
    out = []
    idx = [0] * len(outer)
    while True:
        off = sum(i * st for i, st in zip(idx, strides[:k]))
        out.append(make_region(base + off * size, run, code, "raw", 0, 0,
                               region_id0 + len(out), canary))
        d = len(outer) - 1
        while d >= 0:
            idx[d] += 1
            if idx[d] < outer[d]:
                break
            idx[d] = 0
            d -= 1
        if d < 0:
            return out


def tol_array(tol: Optional[Dict] = None) -> ctypes.Array:
    """Per-dtype tolerances: dict of dtype name/code -> (atol, rtol) or an
    object with .atol/.rtol; unspecified float dtypes get (0, 0)."""
    arr = (Tol * NDTYPES)()
    for k, v in (tol or {}).items():
        code = DTYPE_CODE[k] if isinstance(k, str) else int(k)
        if hasattr(v, "atol"):
            arr[code] = Tol(float(v.atol), float(v.rtol))
        else:
            arr[code] = Tol(float(v[0]), float(v[1]))
    return arr


def stats_dicts(arr, count: int) -> List[dict]:
    return [{f: getattr(arr[i], f) for f in STATS_FIELDS} for i in range(count)]


def check_regions(regions: Sequence, for_fill: bool = False) -> int:
    """Host-only table validation (no GPU needed); returns the status."""
    arr = region_array(regions)
    return lib().asmv_check_regions(arr, len(regions), 1 if for_fill else 0)


def fill_order(regions: Sequence) -> List[int]:
    """The order asmv_fill lays out the regions' tiles in (host only);
    raises AsmvError for a table the fill would reject."""
    arr = region_array(regions)
    out = (ctypes.c_uint32 * max(1, len(regions)))()
    rc = lib().asmv_fill_order(arr, len(regions), out)
    if rc != OK:
        raise AsmvError(rc, lib().asmv_strerror(rc).decode())
    return [int(out[k]) for k in range(len(regions))]


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        try:
            import torch
            return torch.cuda.current_stream().cuda_stream
        except Exception:
            return None
    if hasattr(stream, "cuda_stream"):
        return stream.cuda_stream
    return int(stream)


def _same_lengths(ref: Sequence, cands: Sequence[Sequence]):
    """The C calls read as many candidate regions as there are reference
    regions: a shorter candidate table would be read past its end."""
    for j, c in enumerate(cands):
        if len(c) != len(ref):
            raise ValueError("candidate %d has %d regions, the reference %d" % (j, len(c), len(ref)))


class Context:
    """One asmv context on one CUDA device (not thread-safe)."""

    def __init__(self, device: int = 0):
        self._lib = lib()
        h = ctypes.c_void_p()
        rc = self._lib.asmv_ctx_create(ctypes.byref(h), int(device))
        if rc != OK:
            raise AsmvError(rc, strerror(rc))
        self._h = h
        self.device = device

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            self._lib.asmv_ctx_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def _check(self, rc):
        if rc != OK:
            raise AsmvError(rc, strerror(rc), self._lib.asmv_ctx_cuda_error(self._h))

    @property
    def launches(self) -> int:
        return int(self._lib.asmv_ctx_launches(self._h))

    def set_sm_limit(self, sms: int = 0):
        """asmv_ctx_set_sm_limit: later launches of this context size their
        grids for at most `sms` SMs (0: all), leaving the rest to other work."""
        self._check(self._lib.asmv_ctx_set_sm_limit(self._h, int(sms)))

    def debug_widen(self, nbytes: int):
        """Test hook of the debug-bounds build (asmv_ctx_debug_widen): later
        fills run each payload loop nbytes past its end, and the device
        checks refuse those stores (the call returns EBOUNDS)."""
        self._check(self._lib.asmv_ctx_debug_widen(self._h, int(nbytes)))

    def set_wait_rounds(self, rounds: int = None):
        """Bound of the compare pipeline's device waits (tries of up to
        100 us); None restores the default.  0 makes every compare with a
        non-empty payload return ETIMEOUT (a test of that path)."""
        r = WAIT_ROUNDS if rounds is None else int(rounds)
        self._check(self._lib.asmv_ctx_set_wait_rounds(self._h, r))

    def set_timing(self, enable: bool = True):
        self._check(self._lib.asmv_ctx_set_timing(self._h, 1 if enable else 0))

    def kernel_ms(self) -> float:
        ms = ctypes.c_float()
        self._check(self._lib.asmv_ctx_kernel_ms(self._h, ctypes.byref(ms)))
        return float(ms.value)

    def fill(self, regions: Sequence, seed: int, stream=None):
        arr = region_array(regions)
        self._check(self._lib.asmv_fill(self._h, arr, len(regions), int(seed),
                                        _stream_handle(stream)))

    def guard_check(self, regions: Sequence, stream=None) -> List[dict]:
        arr = region_array(regions)
        out = (Stats * max(1, len(regions)))()
        self._check(self._lib.asmv_guard_check(self._h, arr, len(regions), out,
                                               _stream_handle(stream)))
        return stats_dicts(out, len(regions))

    def compare(self, ref: Sequence, cand: Sequence, tol, stream=None) -> List[dict]:
        _same_lengths(ref, [cand])
        ra, ca = region_array(ref), region_array(cand)
        out = (Stats * max(1, len(ref)))()
        self._check(self._lib.asmv_compare(self._h, ra, ca, len(ref), tol_array(tol)
                                           if not isinstance(tol, ctypes.Array) else tol,
                                           out, _stream_handle(stream)))
        return stats_dicts(out, len(ref))

    def compare_batched(self, ref: Sequence, cands: Sequence[Sequence], tol,
                        stream=None) -> List[List[dict]]:
        _same_lengths(ref, cands)
        n, k = len(ref), len(cands)
        ra = region_array(ref)
        cas = [region_array(c) for c in cands]
        ptrs = (ctypes.POINTER(Region) * max(1, k))(*[ctypes.cast(c, ctypes.POINTER(Region))
                                                      for c in cas])
        out = (Stats * max(1, k * n))()
        self._check(self._lib.asmv_compare_batched(
            self._h, ra, ptrs, k, n,
            tol_array(tol) if not isinstance(tol, ctypes.Array) else tol, out,
            _stream_handle(stream)))
        flat = stats_dicts(out, k * n)
        return [flat[j * n:(j + 1) * n] for j in range(k)]

    def restore(self, regions: Sequence, src: Sequence[int], stream=None):
        """asmv_restore (Tier 2): payload i <- device buffer src[i]; guard
        bands <- canary.  Asynchronous on the stream."""
        arr = region_array(regions)
        a = (ctypes.c_uint64 * max(1, len(regions)))(*[int(x) for x in src])
        self._check(self._lib.asmv_restore(self._h, arr, a, len(regions), _stream_handle(stream)))

    def capture(self, regions: Sequence, dst: Sequence[int], stream=None):
        """asmv_capture: device buffer dst[i] <- payload i.  Asynchronous."""
        arr = region_array(regions)
        a = (ctypes.c_uint64 * max(1, len(regions)))(*[int(x) for x in dst])
        self._check(self._lib.asmv_capture(self._h, arr, a, len(regions), _stream_handle(stream)))

    def compare_eq(self, ref: Sequence, cands: Sequence[Sequence], tol, theta: float = THETA,
                   tau: float = TAU, stream=None):
        """asmv_compare_eq: (stats, eq) with stats[j][i] as compare_batched
        and eq[j][i] the Eq. 1 terms of candidate j on region i."""
        _same_lengths(ref, cands)
        n, k = len(ref), len(cands)
        ra = region_array(ref)
        cas = [region_array(c) for c in cands]
        ptrs = (ctypes.POINTER(Region) * max(1, k))(*[ctypes.cast(c, ctypes.POINTER(Region))
                                                      for c in cas])
        st = (Stats * max(1, k * n))()
        eq = (EqResult * max(1, k * n))()
        self._check(self._lib.asmv_compare_eq(
            self._h, ra, ptrs, k, n,
            tol_array(tol) if not isinstance(tol, ctypes.Array) else tol,
            float(theta), float(tau), st, eq, _stream_handle(stream)))
        flat = stats_dicts(st, k * n)
        eqs = [{f: getattr(eq[x], f) for f in EQ_FIELDS} for x in range(k * n)]
        return ([flat[j * n:(j + 1) * n] for j in range(k)],
                [eqs[j * n:(j + 1) * n] for j in range(k)])

    def compare_eq_digits(self, ref: Sequence, cands: Sequence[Sequence], tol, stream=None):
        """asmv_compare_eq_digits: (stats, digits) with stats[j][i] as
        compare_batched and digits[i, slot, d] the unrounded Eq. 1 sums
        (int64, shape (n, 1 + 2k, D), D = EQ_DIGITS, or EQ64_DIGITS when a
        region is binary64): the per-shard result of a check split across
        processes (see eq_from_digits)."""
        _same_lengths(ref, cands)
        n, k = len(ref), len(cands)
        ra = region_array(ref)
        nd = digits_per_slot([ra[i].dtype for i in range(n)])
        cas = [region_array(c) for c in cands]
        ptrs = (ctypes.POINTER(Region) * max(1, k))(*[ctypes.cast(c, ctypes.POINTER(Region))
                                                      for c in cas])
        st = (Stats * max(1, k * n))()
        dig = np.zeros(max(1, n * (1 + 2 * k) * nd), np.int64)
        self._check(self._lib.asmv_compare_eq_digits(
            self._h, ra, ptrs, k, n,
            tol_array(tol) if not isinstance(tol, ctypes.Array) else tol,
            st, dig.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), _stream_handle(stream)))
        flat = stats_dicts(st, k * n)
        return ([flat[j * n:(j + 1) * n] for j in range(k)],
                dig[:n * (1 + 2 * k) * nd].reshape(n, 1 + 2 * k, nd))


def stats_array(stats: Sequence[dict]) -> ctypes.Array:
    """asmv_stats entries from statistics dicts (as stats_dicts returns them)."""
    arr = (Stats * max(1, len(stats)))()
    for i, d in enumerate(stats):
        for f in STATS_FIELDS:
            setattr(arr[i], f, d[f])
    return arr


def eq_from_digits(dtypes: Sequence, stats: Sequence[Sequence[dict]], digits: np.ndarray,
                   theta: float = None, tau: float = None) -> List[List[dict]]:
    """asmv_eq_from_digits: eq[j][i] of candidate j on region i from
    statistics stats[j][i] and the digit vectors digits[i, slot, d] (as
    Context.compare_eq_digits returns them, possibly summed over shards).
    Host only."""
    theta = THETA if theta is None else theta
    tau = TAU if tau is None else tau
    n, k = len(dtypes), len(stats)
    codes = (ctypes.c_uint32 * max(1, n))(*[dtype_code(d) for d in dtypes])
    st = stats_array([s for row in stats for s in row])
    dig = np.ascontiguousarray(np.asarray(digits, dtype=np.int64).reshape(-1))
    nd = digits_per_slot(dtypes)
    if dig.size != n * (1 + 2 * k) * nd:
        raise ValueError("digits must have shape (n, 1 + 2k, %d)" % nd)
    out = (EqResult * max(1, k * n))()
    rc = lib().asmv_eq_from_digits(codes, k, n, st, dig.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                                   float(theta), float(tau), out)
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    eqs = [{f: getattr(out[x], f) for f in EQ_FIELDS} for x in range(k * n)]
    return [eqs[j * n:(j + 1) * n] for j in range(k)]


def digits_per_slot(dtypes: Sequence) -> int:
    """Digits per exact sum in the digit-vector calls for a table of these
    dtypes: EQ64_DIGITS if any region is binary64, else EQ_DIGITS."""
    return EQ64_DIGITS if any(dtype_code(d) == F64 for d in dtypes) else EQ_DIGITS


def eq_digit_base(dtype) -> int:
    """asmv_eq_digit_base: the binary weight of digit 0 of a float dtype's sums."""
    out = ctypes.c_int()
    rc = lib().asmv_eq_digit_base(dtype_code(dtype), ctypes.byref(out))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return out.value


def exact_to_double(digits: Sequence[int], base_exp: int) -> float:
    """asmv_exact_to_double: sum_k digits[k] 2^(32k + base_exp), rounded to
    the nearest double (host only)."""
    arr = (ctypes.c_int64 * max(1, len(digits)))(*[int(d) for d in digits])
    out = ctypes.c_double()
    rc = lib().asmv_exact_to_double(arr, len(digits), int(base_exp), ctypes.byref(out))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return out.value


def timing_summary(samples_ms: Sequence[float]) -> dict:
    """asmv_timing_summary: median, mean and cv of timing samples."""
    arr = (ctypes.c_double * max(1, len(samples_ms)))(*[float(x) for x in samples_ms])
    out = Timing()
    rc = lib().asmv_timing_summary(arr, len(samples_ms), ctypes.byref(out))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return {"median_ms": out.median_ms, "mean_ms": out.mean_ms, "cv": out.cv, "r": int(out.r)}


def commit_gate(all_eq: bool, s_cand: float, s_best: float, cv: float, eps: float = GATE_EPS,
                k: float = GATE_K, s_floor: float = GATE_S_FLOOR):
    """asmv_commit_gate (Eq. 2): returns (m_star, commit)."""
    m = ctypes.c_double()
    c = ctypes.c_int()
    rc = lib().asmv_commit_gate(1 if all_eq else 0, float(s_cand), float(s_best), float(cv),
                                ctypes.byref(GateParams(eps, k, s_floor)), ctypes.byref(m),
                                ctypes.byref(c))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return m.value, bool(c.value)


def time_launches(fn, r: int, warmup: int = 3, stream=None) -> List[float]:
    """asmv_time_launches: fn(stream_handle) enqueues the work to time; returns
    the device time of each of r calls (ms), after `warmup` untimed calls."""
    handle = _stream_handle(stream)
    err: List[BaseException] = []

    def cb(_user, st):
        if err:
            return
        try:
            fn(st or 0)                  # a null stream handle arrives as None
        except BaseException as e:       # re-raised below, after the C call returns
            err.append(e)
    cfn = LAUNCH_FN(cb)
    out = (ctypes.c_double * max(1, r))()
    cuda_err = ctypes.c_int()
    rc = lib().asmv_time_launches(cfn, None, int(warmup), int(r), out, handle,
                                  ctypes.byref(cuda_err))
    if err:
        raise err[0]
    if rc != OK:
        raise AsmvError(rc, strerror(rc), cuda_err.value)
    return [out[i] for i in range(r)]


def va_granularity(device: int = 0) -> int:
    g = ctypes.c_size_t()
    rc = lib().asmv_va_granularity(int(device), ctypes.byref(g))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return int(g.value)


class VaMapping:
    """asmv_va_map: device memory at a chosen virtual address (0: any)."""

    def __init__(self, nbytes: int, addr: int = 0, device: int = 0):
        self._lib = lib()
        h = ctypes.c_void_p()
        rc = self._lib.asmv_va_map(int(device), int(addr), int(nbytes), ctypes.byref(h))
        if rc != OK:
            raise AsmvError(rc, strerror(rc))
        self._h = h
        self.address = int(self._lib.asmv_va_address(h))
        self.size = int(self._lib.asmv_va_size(h))

    def unmap(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            rc = self._lib.asmv_va_unmap(self._h)
            if rc != OK:
                raise AsmvError(rc, strerror(rc))
            self._h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.unmap()


def compare_noalloc(ref: Sequence, cand: Sequence, tol, stream=None) -> List[dict]:
    """asmv_compare_noalloc: the check of one candidate on the current CUDA
    device, for callers that must not allocate device memory (no context;
    the plan and statistics live in the library's fixed device scratch).
    Raises AsmvError on a non-OK status, ValueError when the candidate's
    table is not as long as the reference's."""
    _same_lengths(ref, [cand])
    L = lib()
    ra, ca = region_array(ref), region_array(cand)
    out = (Stats * max(1, len(ref)))()
    rc = L.asmv_compare_noalloc(ra, ca, len(ref),
                                tol_array(tol) if not isinstance(tol, ctypes.Array) else tol,
                                out, _stream_handle(stream))
    if rc != OK:
        raise AsmvError(rc, strerror(rc))
    return stats_dicts(out, len(ref))
