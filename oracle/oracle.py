"""ctypes view of the CPU oracle (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline and
reference legs import this module.  It loads oracle/liboracle.so, which
shares no code with the CUDA library: it is the plain, slow definition of
the guarded fill and of the per-element equivalence check (AsmEvo, Sec. 3.2
Eq. 1; Sec. 3.4 Tier 1 and Tier 2), in fp64 where the check is floating
point.

Arrays are numpy; every call passes raw pointers of C-contiguous arrays.
"""
import ctypes
import os
import threading

import numpy as np

from . import build as _build

F32, BF16, F16, F8E4M3, I32, I8, U8 = range(7)
F8E5M2, F8E4M3FNUZ, F8E5M2FNUZ, F64, I16, I64 = range(7, 13)
NDTYPES = 13
RAW, UNIFORM, NORMAL, INT_RANGE, NONE = range(5)
DTYPE_SIZE = {F32: 4, BF16: 2, F16: 2, F8E4M3: 1, I32: 4, I8: 1, U8: 1, F8E5M2: 1,
              F8E4M3FNUZ: 1, F8E5M2FNUZ: 1, F64: 8, I16: 2, I64: 8}
FLOAT_DTYPES = (F32, BF16, F16, F8E4M3, F8E5M2, F8E4M3FNUZ, F8E5M2FNUZ, F64)
U64_NONE = (1 << 64) - 1
# codes by the names the workload descriptions use
CODE_OF_DTYPE = {"f32": F32, "bf16": BF16, "f16": F16, "f8e4m3": F8E4M3, "i32": I32,
                 "i8": I8, "u8": U8, "f8e5m2": F8E5M2, "f8e4m3fnuz": F8E4M3FNUZ,
                 "f8e5m2fnuz": F8E5M2FNUZ, "f64": F64, "i16": I16, "i64": I64}
CODE_OF_DIST = {"raw": RAW, "uniform": UNIFORM, "normal": NORMAL, "int_range": INT_RANGE,
                "none": NONE}

_i64p = ctypes.POINTER(ctypes.c_int64)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_u32p = ctypes.POINTER(ctypes.c_uint32)
_f32p = ctypes.POINTER(ctypes.c_float)
_f64p = ctypes.POINTER(ctypes.c_double)
_u64p = ctypes.POINTER(ctypes.c_uint64)


class _Stats(ctypes.Structure):
    _fields_ = [("mismatches", ctypes.c_uint64),
                ("first_mismatch", ctypes.c_uint64),
                ("max_abs_err", ctypes.c_double),
                ("max_rel_err", ctypes.c_double),
                ("nonfinite_mismatches", ctypes.c_uint64)]


class _RegionStats(ctypes.Structure):
    _fields_ = _Stats._fields_ + [("guard_bad_bytes", ctypes.c_uint64),
                                  ("first_guard_bad", ctypes.c_uint64),
                                  ("ref_guard_bad_bytes", ctypes.c_uint64)]


STATS_FIELDS = [f for f, _ in _RegionStats._fields_]

_lib = None
_lock = threading.Lock()


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _load(_build.build())
    return _lib


class use_library:
    """Context manager: route this module's calls to another build of the
    oracle (the tests use it to run the pins against planted mistakes)."""

    def __init__(self, path):
        self.path = path

    def __enter__(self):
        global _lib
        with _lock:
            self.saved = _lib
            _lib = _load(self.path)
        return self

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self.saved


def _load(path):
    L = ctypes.CDLL(path)
    c = ctypes
    L.oracle_philox4x32_10.argtypes = [_u32p, _u32p, _u32p]
    L.oracle_philox_many.argtypes = [_u32p, _u32p, c.c_uint64, _u32p]
    L.oracle_ln_u24_many.argtypes = [_u32p, c.c_uint64, _f32p]
    L.oracle_sincos_2pi_u24_many.argtypes = [_u32p, c.c_uint64, _f32p, _f32p]
    L.oracle_boxmuller_many.argtypes = [_u32p, _u32p, c.c_uint64, _f32p, _f32p]
    L.oracle_boxmuller_consts.argtypes = [_f32p]
    L.oracle_ln_table.argtypes = [_f32p]
    L.oracle_narrow_tables.argtypes = [_f32p]
    L.oracle_radius16_many.argtypes = [_u32p, c.c_uint64, _f32p]
    L.oracle_angle16_many.argtypes = [_u32p, c.c_uint64, _f32p, _f32p]
    L.oracle_normal16_many.argtypes = [_u32p, c.c_uint64, c.c_float, c.c_float, _f32p, _f32p]
    L.oracle_normal8_many.argtypes = [_u32p, c.c_uint64, c.c_float, c.c_float, _f32p, _f32p]
    L.oracle_encode_many.argtypes = [_f32p, c.c_uint64, c.c_int, _u8p]
    L.oracle_decode_many.argtypes = [_u8p, c.c_uint64, c.c_int, _f64p]
    L.oracle_fill_payload.argtypes = [_u8p, c.c_int, c.c_int, c.c_uint64,
                                      c.c_uint64, c.c_uint32, c.c_double,
                                      c.c_double, c.c_uint64]
    L.oracle_fill_payload.restype = c.c_int
    L.oracle_fill_guards.argtypes = [_u8p, c.c_uint64, c.c_uint32,
                                     c.c_uint32, c.c_uint8]
    L.oracle_guard_check.argtypes = [_u8p, c.c_uint64, c.c_uint32, c.c_uint32,
                                     c.c_uint8, _u64p, _u64p]
    L.oracle_compare_range.argtypes = [_u8p, _u8p, c.c_int, c.c_uint64,
                                       c.c_uint64, c.c_double, c.c_double,
                                       c.POINTER(_Stats)]
    L.oracle_compare_region.argtypes = [
        _u8p, c.c_uint32, c.c_uint32, c.c_uint8,
        _u8p, c.c_uint32, c.c_uint32, c.c_uint8,
        c.c_uint64, c.c_int, c.c_double, c.c_double,
        c.POINTER(_RegionStats)]
    L.oracle_eq_sums_range.argtypes = [_u8p, _u8p, c.c_int, c.c_uint64,
                                       c.c_uint64, _i64p]
    L.oracle_eq64_sums_range.argtypes = [_u8p, _u8p, c.c_uint64, c.c_uint64, _i64p]
    L.oracle_restore_region.argtypes = [_u8p, c.c_uint64, c.c_uint32, c.c_uint32,
                                        c.c_uint8, _u8p]
    return L


def _ptr(a, t):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(t)


def _bytes_view(a):
    a = np.ascontiguousarray(a)
    return a.view(np.uint8).reshape(-1)


# ---------------------------------------------------------------- primitives
def philox(ctr, key):
    """Philox4x32-10 blocks: ctr (n,4) uint32, key (n,2) uint32 -> (n,4)."""
    ctr = np.ascontiguousarray(ctr, dtype=np.uint32).reshape(-1, 4)
    key = np.ascontiguousarray(key, dtype=np.uint32).reshape(-1, 2)
    assert ctr.shape[0] == key.shape[0]
    out = np.empty_like(ctr)
    lib().oracle_philox_many(_ptr(ctr, _u32p), _ptr(key, _u32p), ctr.shape[0],
                             _ptr(out, _u32p))
    return out


def ln_u24(k):
    k = np.ascontiguousarray(k, dtype=np.uint32)
    out = np.empty(k.shape, np.float32)
    lib().oracle_ln_u24_many(_ptr(k, _u32p), k.size, _ptr(out, _f32p))
    return out


def sincos_2pi_u24(k):
    k = np.ascontiguousarray(k, dtype=np.uint32)
    sn = np.empty(k.shape, np.float32)
    cs = np.empty(k.shape, np.float32)
    lib().oracle_sincos_2pi_u24_many(_ptr(k, _u32p), k.size, _ptr(sn, _f32p),
                                     _ptr(cs, _f32p))
    return sn, cs


def boxmuller(w0, w1):
    w0 = np.ascontiguousarray(w0, dtype=np.uint32)
    w1 = np.ascontiguousarray(w1, dtype=np.uint32)
    z0 = np.empty(w0.shape, np.float32)
    z1 = np.empty(w0.shape, np.float32)
    lib().oracle_boxmuller_many(_ptr(w0, _u32p), _ptr(w1, _u32p), w0.size,
                                _ptr(z0, _f32p), _ptr(z1, _f32p))
    return z0, z1


def boxmuller_consts():
    """[ln2 head, ln2 tail, 1/3, sin coefficients r^1..r^9, cos r^0..r^10]."""
    out = np.empty(14, np.float32)
    lib().oracle_boxmuller_consts(_ptr(out, _f32p))
    return out


def ln_table():
    """(129, 3) array: inv_j, head_j, tail_j of the ln reduction."""
    out = np.empty(129 * 3, np.float32)
    lib().oracle_ln_table(_ptr(out, _f32p))
    return out.reshape(129, 3)


def narrow_tables():
    """The tables of the 16-bit and 8-bit NORMAL fill: A (512), B (512) of
    the radius chords, sin and cos (256 each) of the angles 2 pi (j + 1/2)
    / 256, the 8-bit radii (256) and the angle step RN32(2 pi / 65536)."""
    out = np.empty(1793, np.float32)
    lib().oracle_narrow_tables(_ptr(out, _f32p))
    return {"A": out[:512].copy(), "B": out[512:1024].copy(), "sin": out[1024:1280].copy(),
            "cos": out[1280:1536].copy(), "r8": out[1536:1792].copy(), "c16": out[1792]}


def radius16(k):
    k = np.ascontiguousarray(k, dtype=np.uint32)
    out = np.empty(k.shape, np.float32)
    lib().oracle_radius16_many(_ptr(k, _u32p), k.size, _ptr(out, _f32p))
    return out


def angle16(a):
    """(sin, cos) of the angle 2 pi (a + 1/2) / 65536 as the 16-bit fill
    forms it."""
    a = np.ascontiguousarray(a, dtype=np.uint32)
    sn = np.empty(a.shape, np.float32)
    cs = np.empty(a.shape, np.float32)
    lib().oracle_angle16_many(_ptr(a, _u32p), a.size, _ptr(sn, _f32p), _ptr(cs, _f32p))
    return sn, cs


def normal16(w, mean=0.0, sd=1.0):
    """The pair (v0, v1) the 16-bit NORMAL fill draws from 32-bit words w."""
    w = np.ascontiguousarray(w, dtype=np.uint32)
    v0 = np.empty(w.shape, np.float32)
    v1 = np.empty(w.shape, np.float32)
    lib().oracle_normal16_many(_ptr(w, _u32p), w.size, float(mean), float(sd),
                               _ptr(v0, _f32p), _ptr(v1, _f32p))
    return v0, v1


def normal8(h, mean=0.0, sd=1.0):
    """The pair (v0, v1) the 8-bit NORMAL fill draws from 16-bit halves h."""
    h = np.ascontiguousarray(h, dtype=np.uint32)
    v0 = np.empty(h.shape, np.float32)
    v1 = np.empty(h.shape, np.float32)
    lib().oracle_normal8_many(_ptr(h, _u32p), h.size, float(mean), float(sd),
                              _ptr(v0, _f32p), _ptr(v1, _f32p))
    return v0, v1


def encode(x, dtype):
    """fp32 array -> raw bytes of the float dtype (RNE)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.size * DTYPE_SIZE[dtype], np.uint8)
    lib().oracle_encode_many(_ptr(x, _f32p), x.size, dtype, _ptr(out, _u8p))
    return out


def decode(raw, dtype):
    """raw bytes -> float64 values of the dtype (exact)."""
    raw = _bytes_view(raw)
    n = raw.size // DTYPE_SIZE[dtype]
    out = np.empty(n, np.float64)
    lib().oracle_decode_many(_ptr(raw, _u8p), n, dtype, _ptr(out, _f64p))
    return out


# ---------------------------------------------------------------- fill
def fill_payload(payload, dtype, dist, i0, i1, region_id, p0, p1, seed):
    """Write elements [i0, i1) of `payload` (uint8 view of element 0 on)."""
    assert payload.dtype == np.uint8 and payload.flags["C_CONTIGUOUS"]
    assert i1 * DTYPE_SIZE[dtype] <= payload.size
    rc = lib().oracle_fill_payload(_ptr(payload, _u8p), dtype, dist, i0, i1,
                                   region_id, float(p0), float(p1), seed)
    if rc != 0:
        raise ValueError("distribution %d does not apply to dtype %d" % (dist, dtype))


def _split(n, parts):
    parts = max(1, min(parts, n)) if n else 1
    edges = [n * k // parts for k in range(parts + 1)]
    return list(zip(edges[:-1], edges[1:]))


def _run_threads(fns):
    if len(fns) == 1:
        fns[0]()
        return
    ts = [threading.Thread(target=f) for f in fns]
    for t in ts:
        t.start()
    for t in ts:
        t.join()


def fill_region(alloc, n_elems, dtype, dist, guard_lo, guard_hi, region_id,
                canary, p0, p1, seed, threads=1):
    """Guarded fill of one allocation (uint8 array covering the whole
    allocation: low guard, payload, high guard)."""
    nbytes = n_elems * DTYPE_SIZE[dtype]
    assert alloc.size >= guard_lo + nbytes + guard_hi
    payload = alloc[guard_lo:guard_lo + nbytes]
    lib().oracle_fill_guards(_ptr(alloc, _u8p), nbytes, guard_lo, guard_hi, canary)
    fns = [lambda a=a, b=b: fill_payload(payload, dtype, dist, a, b, region_id, p0, p1, seed)
           for a, b in _split(n_elems, threads)]
    _run_threads(fns)


def guard_check(alloc, payload_bytes, guard_lo, guard_hi, canary):
    bad = ctypes.c_uint64()
    first = ctypes.c_uint64()
    lib().oracle_guard_check(_ptr(alloc, _u8p), payload_bytes, guard_lo, guard_hi,
                             canary, ctypes.byref(bad), ctypes.byref(first))
    return int(bad.value), int(first.value)


# ---------------------------------------------------------------- compare
def compare_range(ref_payload, cand_payload, dtype, i0, i1, atol, rtol):
    st = _Stats()
    lib().oracle_compare_range(_ptr(ref_payload, _u8p), _ptr(cand_payload, _u8p),
                               dtype, i0, i1, float(atol), float(rtol), ctypes.byref(st))
    return {f: getattr(st, f) for f, _ in _Stats._fields_}


def merge_partials(parts):
    """Combine range results: sums, min of first index, max of the maxima."""
    out = {"mismatches": 0, "first_mismatch": U64_NONE, "max_abs_err": 0.0,
           "max_rel_err": 0.0, "nonfinite_mismatches": 0}
    for p in parts:
        out["mismatches"] += p["mismatches"]
        out["first_mismatch"] = min(out["first_mismatch"], p["first_mismatch"])
        out["max_abs_err"] = max(out["max_abs_err"], p["max_abs_err"])
        out["max_rel_err"] = max(out["max_rel_err"], p["max_rel_err"])
        out["nonfinite_mismatches"] += p["nonfinite_mismatches"]
    return out


def compare_payload(ref_payload, cand_payload, dtype, n_elems, atol, rtol, threads=1):
    parts = [None] * len(_split(n_elems, threads))

    def job(k, a, b):
        parts[k] = compare_range(ref_payload, cand_payload, dtype, a, b, atol, rtol)
    _run_threads([lambda k=k, a=a, b=b: job(k, a, b)
                  for k, (a, b) in enumerate(_split(n_elems, threads))])
    return merge_partials(parts)


def compare_region(ref_alloc, ref_glo, ref_ghi, ref_canary, cand_alloc, cand_glo,
                   cand_ghi, cand_canary, n_elems, dtype, atol, rtol, threads=1):
    """Full per-region statistics (8 fields), guards included."""
    if threads <= 1:
        st = _RegionStats()
        lib().oracle_compare_region(_ptr(ref_alloc, _u8p), ref_glo, ref_ghi, ref_canary,
                                    _ptr(cand_alloc, _u8p), cand_glo, cand_ghi, cand_canary,
                                    n_elems, dtype, float(atol), float(rtol), ctypes.byref(st))
        return {f: getattr(st, f) for f in STATS_FIELDS}
    nbytes = n_elems * DTYPE_SIZE[dtype]
    out = compare_payload(ref_alloc[ref_glo:ref_glo + nbytes],
                          cand_alloc[cand_glo:cand_glo + nbytes], dtype, n_elems,
                          atol, rtol, threads)
    out["guard_bad_bytes"], out["first_guard_bad"] = guard_check(
        cand_alloc, nbytes, cand_glo, cand_ghi, cand_canary)
    out["ref_guard_bad_bytes"] = guard_check(ref_alloc, nbytes, ref_glo, ref_ghi,
                                             ref_canary)[0]
    return out


def host_threads():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ------------------------------------------- Eq. 1 aggregate (cosine) terms
EQ_DIGITS, EQ_BASE = 20, -320
EQ_COS, EQ_LINF, EQ_INT, EQ_GUARD = 1, 2, 4, 8
THETA, TAU = 0.9999, 1e-3          # the paper's thresholds for Eq. 1 (Sec. 5)


def eq_sums_range(ref_payload, cand_payload, dtype, i0, i1):
    """Exact S_rc, S_rr, S_cc over elements [i0, i1), as Python integers
    scaled by 2^-EQ_BASE (value = integer * 2^EQ_BASE)."""
    out = np.zeros(3 * EQ_DIGITS, np.int64)
    lib().oracle_eq_sums_range(_ptr(ref_payload, _u8p), _ptr(cand_payload, _u8p),
                               dtype, i0, i1, _ptr(out, _i64p))
    vals = []
    for s in range(3):
        d = out[s * EQ_DIGITS:(s + 1) * EQ_DIGITS]
        vals.append(sum(int(d[k]) << (32 * k) for k in range(EQ_DIGITS)))
    return tuple(vals)


def exact_to_double(v):
    """The integer v * 2^EQ_BASE rounded to the nearest fp64, ties to even
    (Python's int / int true division rounds correctly)."""
    return v / (1 << -EQ_BASE)


# Binary64 regions (reading R11 of the C oracle): products up to 106 bits,
# sums kept exactly at the binary point 2^EQ64_BASE.
EQ64_DIGITS, EQ64_BASE = 136, -2148


def eq64_sums_range(ref_payload, cand_payload, i0, i1):
    """Exact S_rc, S_rr, S_cc of two binary64 payloads over elements
    [i0, i1), as Python integers scaled by 2^-EQ64_BASE."""
    out = np.zeros(3 * EQ64_DIGITS, np.int64)
    lib().oracle_eq64_sums_range(_ptr(ref_payload, _u8p), _ptr(cand_payload, _u8p), i0, i1,
                                 _ptr(out, _i64p))
    vals = []
    for s in range(3):
        d = out[s * EQ64_DIGITS:(s + 1) * EQ64_DIGITS]
        vals.append(sum(int(d[k]) << (32 * k) for k in range(EQ64_DIGITS)))
    return tuple(vals)


def round_scaled(v, e):
    """The integer v times 2^e rounded to the nearest fp64, ties to even,
    with gradual underflow and overflow to an infinity of v's sign (Python's
    int-to-float conversion and int / int division both round correctly and
    raise OverflowError exactly when the rounded value overflows)."""
    if v == 0:
        return 0.0
    try:
        return float(v << e) if e >= 0 else v / (1 << -e)
    except OverflowError:
        return float("inf") if v > 0 else float("-inf")


def eq_cos_exact(v_rc, v_rr, v_cc, base):
    """c_x of Eq. 1 from exact sums S = v * 2^base, without overflow or
    underflow of the intermediate sums: with 2p and 2q the even exponents
    that bring S_rr and S_cc into [1, 4), the cosine is formed in fp64 from
    RN(S_rc 2^-(p+q)), RN(S_rr 2^-2p) and RN(S_cc 2^-2q) -- the same number
    as the plain formula, whose sums of binary64 values can leave the double
    range.  1 when both sums of squares are 0, 0 when exactly one is."""
    import math
    if v_rr == 0 and v_cc == 0:
        return 1.0
    if v_rr == 0 or v_cc == 0:
        return 0.0
    p = (v_rr.bit_length() - 1 + base) // 2          # floor, also below zero
    q = (v_cc.bit_length() - 1 + base) // 2
    x = round_scaled(v_rc, base - p - q)
    y = round_scaled(v_rr, base - 2 * p)
    z = round_scaled(v_cc, base - 2 * q)
    return x / (math.sqrt(y) * math.sqrt(z))


def eq_cos(s_rc, s_rr, s_cc):
    """c_x of Eq. 1 from the rounded sums, in fp64: S_rc / (sqrt(S_rr) *
    sqrt(S_cc)); 1 when both vectors are zero, 0 when exactly one is."""
    import math
    if s_rr == 0.0 and s_cc == 0.0:
        return 1.0
    if s_rr == 0.0 or s_cc == 0.0:
        return 0.0
    return s_rc / (math.sqrt(s_rr) * math.sqrt(s_cc))


def eq_sums(ref_payload, cand_payload, dtype, n_elems, threads=1):
    """The three sums of one float region, each exact then rounded to fp64,
    and the cosine c_x.  Binary64 sums round with gradual underflow and
    overflow to infinity, and their cosine comes from the scaled exact sums
    (eq_cos_exact); for the other formats the sums stay well inside the
    normal double range and c_x is eq_cos of the rounded sums."""
    spans = _split(n_elems, threads)
    parts = [None] * len(spans)

    def job(k, a, b):
        if dtype == F64:
            parts[k] = eq64_sums_range(ref_payload, cand_payload, a, b)
        else:
            parts[k] = eq_sums_range(ref_payload, cand_payload, dtype, a, b)
    _run_threads([lambda k=k, a=a, b=b: job(k, a, b) for k, (a, b) in enumerate(spans)])
    tot = [sum(p[j] for p in parts) for j in range(3)]
    if dtype == F64:
        out = {"sum_rc": round_scaled(tot[0], EQ64_BASE), "sum_rr": round_scaled(tot[1], EQ64_BASE),
               "sum_cc": round_scaled(tot[2], EQ64_BASE)}
        out["cos"] = eq_cos_exact(tot[0], tot[1], tot[2], EQ64_BASE)
        return out
    out = {"sum_rc": exact_to_double(tot[0]), "sum_rr": exact_to_double(tot[1]),
           "sum_cc": exact_to_double(tot[2])}
    out["cos"] = eq_cos(out["sum_rc"], out["sum_rr"], out["sum_cc"])
    return out


def eq_verdict(stats, sums, dtype, theta=THETA, tau=TAU):
    """Eq. 1 for one region: c_x >= theta, ||Delta||_inf <= tau, and iota
    (bit-exact integer and opaque buffers, intact candidate guard bands).
    Float regions: the L-infinity term is the exact max |c - r| over finite
    pairs and fails on any NaN/Inf-position mismatch.  S_rc sums over pairs
    with both values finite, S_rr over finite r, S_cc over finite c.  Integer and opaque
    regions have no cosine (NaN) and pass the two float terms."""
    flt = dtype in FLOAT_DTYPES
    out = dict(sums) if flt else {"sum_rc": 0.0, "sum_rr": 0.0, "sum_cc": 0.0}
    if not flt:
        out["cos"] = float("nan")
    elif "cos" not in out:
        out["cos"] = eq_cos(out["sum_rc"], out["sum_rr"], out["sum_cc"])
    flags = 0
    if not flt or out["cos"] >= theta:
        flags |= EQ_COS
    if not flt or (stats["max_abs_err"] <= tau and stats["nonfinite_mismatches"] == 0):
        flags |= EQ_LINF
    if flt or stats["mismatches"] == 0:
        flags |= EQ_INT
    if stats["guard_bad_bytes"] == 0:
        flags |= EQ_GUARD
    out["flags"] = flags
    out["eq"] = int(flags == EQ_COS | EQ_LINF | EQ_INT | EQ_GUARD)
    return out


# ------------------------------------------------------- Tier 2 restore
def restore_region(alloc, payload_bytes, guard_lo, guard_hi, canary, captured):
    """Write the canary over both guard bands of `alloc` (a uint8 array of
    guard_lo + payload_bytes + guard_hi bytes) and the captured bytes over
    its payload."""
    assert alloc.size >= guard_lo + payload_bytes + guard_hi and captured.size >= payload_bytes
    lib().oracle_restore_region(_ptr(alloc, _u8p), payload_bytes, guard_lo, guard_hi, canary,
                                _ptr(np.ascontiguousarray(captured), _u8p))
