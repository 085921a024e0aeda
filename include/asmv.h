/*
 * asmv.h -- C ABI of the GB300 differential-oracle hot path.
 *
 * The library implements the data-parallel core of the differential oracle
 * that gates every candidate kernel in AsmEvo (arXiv 2608.20711):
 *
 *   - Tier 1 guarded input synthesis (Sec. 3.4, "Tier 1: synthetic
 *     inference"): every allocation a kernel references is filled with
 *     deterministic seeded values, and guard bands on both sides of the
 *     payload are set to a canary byte so that out-of-bounds writes become
 *     visible.
 *   - The equivalence check eq(K', x) of Eq. 1 (Sec. 3.2, R2) applied to the
 *     captured output regions (Sec. 3.4, "Tier 2: real-dispatch capture"):
 *     floating-point outputs are checked against a tolerance, integer
 *     buffers, opaque state and guard bytes must match byte-exactly (the
 *     iota term of Eq. 1).  The tolerance is applied per element with a
 *     per-dtype (atol, rtol): element r (reference) and c (candidate) match
 *     iff |c - r| <= atol + rtol*|r|, evaluated in fp64 on the exactly
 *     decoded values.  Per region the library reports the mismatch count,
 *     the first mismatching element, the exact fp64 maximum absolute and
 *     relative error over finite pairs (the ||Delta||_inf of Eq. 1 is
 *     max_abs_err when nonfinite_mismatches == 0), NaN/Inf-position
 *     mismatches and guard-band damage.
 *
 * All device work runs in CUDA kernels on the caller's stream.  There is no
 * CPU fallback: a call whose tables point at host memory fails with
 * ASMV_EINVAL.
 *
 * Threading: a context is not thread-safe.  Use one context per host
 * thread; calls on one context are ordered on the device even when they
 * name different streams (each call waits for the previous call's use of
 * the context's workspace).
 */
#ifndef ASMV_H_
#define ASMV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ASMV_ABI_VERSION 3

/* A CUDA stream (the same type as cudaStream_t); NULL is the legacy
 * default stream. */
typedef struct CUstream_st *asmv_stream_t;

/* Element types of a region.  Float types are compared with the tolerance
 * test; integer and opaque types bit-exactly (Sec. 3.4, Tier 2). */
typedef enum {
  ASMV_F32 = 0,        /* IEEE binary32 */
  ASMV_BF16 = 1,       /* bfloat16 */
  ASMV_F16 = 2,        /* IEEE binary16 */
  ASMV_F8E4M3 = 3,     /* OCP FP8 E4M3 (no Inf; S.1111.111 is NaN; max 448) */
  ASMV_I32 = 4,        /* two's complement int32 */
  ASMV_I8 = 5,         /* two's complement int8 */
  ASMV_U8_OPAQUE = 6,  /* opaque bytes (compared as unsigned 8-bit values) */
  ASMV_F8E5M2 = 7,     /* OCP FP8 E5M2 (bias 15; Inf and NaN at exponent 31; max 57344) */
  ASMV_F8E4M3FNUZ = 8, /* FP8 E4M3 "fnuz": bias 8, finite, no -0, 0x80 is NaN; max 240 */
  ASMV_F8E5M2FNUZ = 9, /* FP8 E5M2 "fnuz": bias 16, finite, no -0, 0x80 is NaN; max 57344 */
  ASMV_F64 = 10,       /* IEEE binary64 */
  ASMV_I16 = 11,       /* two's complement int16 */
  ASMV_I64 = 12,       /* two's complement int64 */
  ASMV_NDTYPES = 13
} asmv_dtype;

/* Payload distributions of asmv_fill (Sec. 3.4, Tier 1: deterministic
 * inputs from random seeds).  Element i draws from Philox4x32-10 with
 * key = (seed lo, seed hi) and counter = (block lo, block hi, region_id, 0):
 *   RAW       payload byte j is byte (j mod 16) of block (j div 16); the
 *             block's four 32-bit words in order, each little-endian.
 *             Any dtype.
 *   UNIFORM   float dtypes: a fraction f, v = p0 + f*(p1 - p0) in fp32
 *             (p0, p1 and p1 - p0 rounded to fp32 first; multiply then add),
 *             then round-to-nearest-even to the dtype (every fp8 format
 *             saturates at its largest finite value; fnuz formats give +0 for
 *             a zero result; binary64 is the exact widening of the fp32
 *             value).  fp32 and binary64: w = word (i mod 4) of block
 *             (i div 4), f = (w >> 8) * 2^-24.  16-bit formats: h = half
 *             (i mod 2) (low half first) of word (i mod 8) div 2 of block
 *             (i div 8), f = h * 2^-16.  8-bit formats: b = byte (i mod 4) of
 *             word (i mod 16) div 4 of block (i div 16), f = b * 2^-8.
 *   NORMAL    fp32 and binary64: Box-Muller on words (0,1) and (2,3) of
 *             block (i div 4): u1 = ((w0 >> 8) + 1) 2^-24, u2 = (w1 >> 8)
 *             2^-24, z0 = sqrt(-2 ln u1) cos(2 pi u2), z1 = ... sin(2 pi u2);
 *             element 4b+2p+t is z_t of pair p; v = p0 + p1*z in fp32, then
 *             RNE to the dtype.  ln and sincos are fixed fp32 series
 *             evaluations, so results are bit-reproducible.
 *             16-bit formats: element i is v_(i mod 2) of the pair drawn from
 *             word (i mod 8) div 2 of block (i div 8): radius from the low
 *             half k, u = (k + 1/2) 2^-16, rho = sqrt(-2 ln u) as a chord over
 *             one of 512 cells (within 2^-13); angle from the high half a,
 *             theta = 2 pi (a + 1/2) / 65536, as a table angle
 *             2 pi (j + 1/2) / 256 (j = a div 256) turned to first order;
 *             v0 = p1 rho cos theta + p0, v1 = p1 rho sin theta + p0 (one fma
 *             each after rs = rho p1).  8-bit formats: element i is
 *             v_(i mod 2) of the pair drawn from half (i mod 4) div 2 of word
 *             (i mod 16) div 4 of block (i div 16): radius index = its low
 *             byte k, rho = sqrt(-2 ln((k + 1/2) / 256)); angle index = its
 *             high byte j, theta = 2 pi (j + 1/2) / 256.  Every constant is
 *             the correctly rounded fp32 value of its closed form and every
 *             step one IEEE fp32 operation in a fixed order, so the bytes are
 *             reproducible on any IEEE machine.
 *   INT_RANGE integer dtypes: w = word (i mod 4) of block (i div 4),
 *             v = lo + ((w*(hi-lo)) >> 32)
 *             with lo = p0, hi = p1 (integers; 1 <= hi - lo <= 2^32 and
 *             [lo, hi) inside the dtype's range; for int64 |p0|, |p1| <= 2^53).
 *   NONE      the payload is left untouched; only guard bands are written. */
typedef enum {
  ASMV_DIST_RAW = 0,
  ASMV_DIST_UNIFORM = 1,
  ASMV_DIST_NORMAL = 2,
  ASMV_DIST_INT_RANGE = 3,
  ASMV_DIST_NONE = 4
} asmv_dist;

/* One guarded allocation (Sec. 3.4: a referenced device-memory region with
 * guard regions initialised with canaries).  Layout in device memory:
 *   [alloc, alloc+guard_lo)                   low guard band
 *   [alloc+guard_lo, +n_elems*size(dtype))    payload
 *   [payload end, +guard_hi)                  high guard band
 * All three lie in one device allocation owned by the caller.  56 bytes. */
typedef struct {
  uint64_t alloc;      /* device address of the allocation start */
  uint64_t n_elems;    /* payload elements (may be 0) */
  uint32_t dtype;      /* asmv_dtype */
  uint32_t dist;       /* asmv_dist; read by asmv_fill only */
  uint32_t guard_lo;   /* guard bytes below the payload (may be 0) */
  uint32_t guard_hi;   /* guard bytes above the payload (may be 0) */
  uint32_t region_id;  /* Philox counter word 2 for this region's payload */
  uint8_t canary;      /* guard byte value */
  uint8_t pad_[3];
  double p0, p1;       /* distribution parameters (see asmv_dist) */
} asmv_region;

/* Per-dtype tolerance, indexed by asmv_dtype; entries of integer and opaque
 * dtypes are ignored.  Both must be >= 0 and not NaN for float dtypes. */
typedef struct {
  double atol;
  double rtol;
} asmv_tol;

/* Per-region result (64 bytes). */
typedef struct {
  uint64_t mismatches;           /* elements failing the check (incl. non-finite) */
  uint64_t first_mismatch;       /* lowest failing element index; UINT64_MAX if none */
  double max_abs_err;            /* max over finite pairs of |c - r| (exact fp64; binary64
                                    pairs: the rounded difference; int64: the exact
                                    difference rounded once); 0 if none */
  double max_rel_err;            /* max over finite pairs of |c - r| / |r|; r == 0 gives
                                    0 when c == r, else +Inf */
  uint64_t nonfinite_mismatches; /* failing pairs with a NaN or Inf on either side */
  uint64_t guard_bad_bytes;      /* guard bytes != canary (candidate side, or the region
                                    itself for asmv_guard_check) */
  uint64_t first_guard_bad;      /* lowest such byte offset from alloc; UINT64_MAX if none */
  uint64_t ref_guard_bad_bytes;  /* asmv_compare*: damaged reference guard bytes */
} asmv_stats;

/* Status codes.  A failed call leaves out_host untouched. */
#define ASMV_OK 0
#define ASMV_EINVAL (-1)    /* bad argument or table (see each call) */
#define ASMV_ECUDA (-2)     /* a CUDA runtime call failed; see asmv_ctx_cuda_error */
#define ASMV_ETIMEOUT (-3)  /* a bounded device wait expired */
#define ASMV_ENOMEM (-4)    /* workspace or staging allocation failed */
#define ASMV_EBOUNDS (-5)   /* debug-bounds build only: a device access fell outside its allocation */

typedef struct asmv_ctx asmv_ctx;

/* Create a context on CUDA device `device`.  The context owns a device
 * workspace (region tables, statistics) and pinned host staging, both grown
 * on demand.  Returns ASMV_OK and *out, or EINVAL (null out, bad device),
 * ECUDA, ENOMEM. */
int asmv_ctx_create(asmv_ctx **out, int device);

/* Release the context (synchronises its outstanding work).  NULL is a no-op. */
void asmv_ctx_destroy(asmv_ctx *ctx);

/* Tier 1 guarded fill (Sec. 3.4, Tier 1).  Writes every region's payload
 * from its distribution and both guard bands with its canary.  The table is
 * copied before return; the fill itself is asynchronous on `stream`.
 * EINVAL: null ctx/table with n > 0, unknown dtype or dist, a distribution
 * that does not apply to the dtype or parameters out of range, size
 * overflow, a zero alloc address with a non-empty allocation, overlapping
 * allocations, or memory that is not device memory of ctx's device (or
 * that ends past its allocation). */
int asmv_fill(asmv_ctx *ctx, const asmv_region *regions, size_t n, uint64_t seed,
              asmv_stream_t stream);

/* Guard-band integrity (the "intact out-of-bounds guards" of the iota term
 * of Eq. 1, Sec. 3.2).  For each region, counts guard bytes that differ
 * from its canary and the first such offset from alloc (low band first).
 * out_host[i] receives guard_bad_bytes and first_guard_bad; the other
 * fields are their empty values (0, UINT64_MAX).  Synchronous: returns
 * after the results are in out_host.  Errors as asmv_fill (overlap is
 * allowed), plus EINVAL for null out_host. */
int asmv_guard_check(asmv_ctx *ctx, const asmv_region *regions, size_t n,
                     asmv_stats *out_host, asmv_stream_t stream);

/* The equivalence check (Eq. 1 per element, Sec. 3.2; Tier 2 rule, Sec.
 * 3.4) of n (reference, candidate) region pairs: ref[i] against cand[i].
 * Pairs must agree in dtype and n_elems.  Candidate guards feed
 * guard_bad_bytes / first_guard_bad, reference guards ref_guard_bad_bytes.
 * tol has ASMV_NDTYPES entries.  Synchronous.  EINVAL as asmv_guard_check,
 * plus dtype/count disagreement and invalid tolerances. */
int asmv_compare(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *cand,
                 size_t n, const asmv_tol *tol, asmv_stats *out_host,
                 asmv_stream_t stream);

/* The check over many candidates at once (the eq loop of Algorithm 1 run
 * for k candidates against one oracle output): cands[j] is an array of n
 * regions matching ref; out_host has k*n entries, out_host[j*n + i] being
 * compare(ref[i], cands[j][i]).  Each reference tile is read from device
 * memory once per group of up to 8 candidates.  Synchronous.  Errors as
 * asmv_compare, plus EINVAL for k == 0 or a null cands entry. */
int asmv_compare_batched(asmv_ctx *ctx, const asmv_region *ref,
                         const asmv_region *const *cands, size_t k, size_t n,
                         const asmv_tol *tol, asmv_stats *out_host,
                         asmv_stream_t stream);

/* ---------------------------------------------------------------------
 * Eq. 1 as a whole (Sec. 3.2): eq(K', x) = c_x >= theta AND
 * ||K'(x) - O(x)||_inf <= tau AND iota(K', x), with c_x the cosine of the
 * candidate and reference outputs and iota requiring bit-exact integer and
 * opaque buffers and intact guard bands.  The paper uses theta = 0.9999 and
 * tau = 1e-3 (Sec. 5).  Per region:
 *   - float regions: sum_rc = sum of r*c over pairs with both values finite,
 *     sum_rr = sum of r*r over finite r, sum_cc = sum of c*c over finite c;
 *     each is the exact sum rounded once to the nearest double (ties to
 *     even), so it does not depend on the grid or the order of elements.
 *     cos = sum_rc / (sqrt(sum_rr) * sqrt(sum_cc)) in double, 1 when both
 *     sums of squares are 0, 0 when exactly one is.  The L-infinity term is
 *     max_abs_err of asmv_stats (exact, finite pairs) <= tau together with
 *     no NaN/Inf-position mismatch.
 *   - integer and opaque regions: sums 0, cos NaN; the cosine and
 *     L-infinity terms hold, the integer term needs mismatches == 0.
 *   - every region: the guard term needs guard_bad_bytes == 0 (the
 *     candidate's bands; the reference's are reported, not judged).
 * ------------------------------------------------------------------- */
#define ASMV_EQ_COS   1u   /* c_x >= theta */
#define ASMV_EQ_LINF  2u   /* ||Delta||_inf <= tau and no NaN/Inf-position mismatch */
#define ASMV_EQ_INT   4u   /* integer / opaque payload bit-exact */
#define ASMV_EQ_GUARD 8u   /* candidate guard bands intact */

typedef struct {
  double sum_rc, sum_rr, sum_cc;
  double cos;
  uint32_t flags;       /* the ASMV_EQ_* terms that hold */
  uint32_t eq;          /* 1 iff all four hold */
} asmv_eq;              /* 40 bytes */

/* asmv_compare_batched plus the Eq. 1 terms: stats_host[j*n + i] as there,
 * eq_host[j*n + i] the Eq. 1 result of candidate j on region i (k*n entries
 * each, caller-owned).  theta is any finite double; tau a finite double
 * >= 0.  Float regions of more than 2^31 elements are rejected (the exact
 * sums keep per-digit counts below 2^31).  Binary64 regions: the exact sums
 * (products of 106 bits, 2^-2148 .. 2^2048) are rounded with gradual
 * underflow and overflow to +-Inf, so sum_* may be Inf, subnormal or 0 for
 * outputs near the ends of the double range; cos is formed from the exact
 * sums scaled by powers of two (sum_rr by 2^-2p and sum_cc by 2^-2q into
 * [1, 4), sum_rc by 2^-(p+q)), which is the same cosine and stays finite.
 * Synchronous.  Errors as asmv_compare_batched, plus EINVAL for a null
 * eq_host, a non-finite theta or tau, a negative tau, or such a region. */
int asmv_compare_eq(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                    size_t k, size_t n, const asmv_tol *tol, double theta, double tau,
                    asmv_stats *stats_host, asmv_eq *eq_host, asmv_stream_t stream);

/* Eq. 1 over a check split across processes (each takes an element range
 * of every region): each process returns its exact sums unrounded, the
 * digit vectors are added element-wise over the processes and the
 * statistics merged, and asmv_eq_from_digits gives the verdict of the
 * whole -- the same result as one asmv_compare_eq over the whole regions.
 *
 * asmv_compare_eq_digits: the statistics of asmv_compare_batched in
 * stats_host[j*n + i], and the exact sums of region i in
 *   digits_host[(i*(1 + 2k) + slot) * D + d]     (k*n and n*(1+2k)*D entries)
 * as signed 64-bit digits, digit d weighing 2^(32 d + base) with base =
 * asmv_eq_digit_base(dtype of region i).  D = ASMV_EQ_DIGITS (20) unless
 * the table holds a binary64 region, whose sums need ASMV_EQ64_DIGITS
 * (136): then D = 136 for every region, and the digits of the other
 * regions beyond their first 20 are zero.  Slot 0 holds sum r*r; slots
 * 1 + 2j and 2 + 2j hold candidate j's two further sums (for fp16 and the
 * fp8 formats other than E4M3 these are sum r*d and sum d*d with d = c - r,
 * otherwise sum r*c and sum c*c); every slot is a sum over elements, so
 * shards add.  Digits of integer and opaque regions are zero.  Errors as
 * asmv_compare_eq (theta and tau are not taken), with digits_host in place
 * of eq_host.  Synchronous. */
#define ASMV_EQ_DIGITS 20
#define ASMV_EQ64_DIGITS 136
int asmv_compare_eq_digits(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                           size_t k, size_t n, const asmv_tol *tol, asmv_stats *stats_host,
                           int64_t *digits_host, asmv_stream_t stream);

/* Host only: the Eq. 1 results eq_out[j*n + i] (as asmv_compare_eq) from
 * statistics and digit vectors laid out as asmv_compare_eq_digits returns
 * them (possibly the sums over shards; any signed digit values are
 * accepted), for regions of dtypes[i] (D follows from them as above).
 * Makes no CUDA call.  EINVAL for a null pointer with k*n > 0, k == 0, an
 * unknown dtype, theta or tau as asmv_compare_eq, digits of a format other
 * than binary64 whose sum is outside the normal double range (or, with
 * D = 136, does not fit its first 20 digits), or a negative sum of squares
 * of a binary64 region. */
int asmv_eq_from_digits(const uint32_t *dtypes, size_t k, size_t n, const asmv_stats *stats,
                        const int64_t *digits, double theta, double tau, asmv_eq *eq_out);

/* The binary weight of digit 0 of the exact sums of a float dtype, in
 * *base (-2148 for binary64).  EINVAL for other dtypes or a null base. */
int asmv_eq_digit_base(uint32_t dtype, int *base);

/* The integer sum_k digits[k] * 2^(32 k + base_exp) (k < ndigits, each
 * digit a signed 64-bit value) rounded to the nearest double, ties to even;
 * the conversion asmv_compare_eq applies to its exact sums.  Host only,
 * makes no CUDA call.  EINVAL for a null pointer, ndigits outside
 * [1, 64], or a result outside the normal double range (which the sums of
 * the formats other than binary64 never reach; asmv_compare_eq rounds the
 * 136-digit binary64 sums itself, with gradual underflow and overflow to
 * +-Inf). */
int asmv_exact_to_double(const int64_t *digits, int ndigits, int base_exp, double *out);

/* ---------------------------------------------------------------------
 * GatedEval timing and the commit gate (Sec. 3.4, Algorithm 1; Eq. 2).
 * Correctness first (asmv_compare_eq over every evaluated input), then
 * timing: warm-up launches, then R launches each timed with its own pair of
 * CUDA events; the latency is their median.  The speedup of a candidate c
 * is s(c) = T(K0) / T(c).  Eq. 2 commits c only if it is equivalent on
 * every input and
 *   s(c) >= max(m*, s_floor),   m* = (1 + max(eps, k * cv)) * s(K*),
 * with K* the current verified best (s(K0) = 1) and cv the coefficient of
 * variation of the timings.  The paper uses eps = 0.002, k = 0.85,
 * s_floor = 1.0 (Sec. 5).
 * ------------------------------------------------------------------- */
#define ASMV_GATE_EPS     0.002
#define ASMV_GATE_K       0.85
#define ASMV_GATE_S_FLOOR 1.0

typedef struct {
  double median_ms;   /* median (mean of the two middle samples when R is even) */
  double mean_ms;     /* sum in sample order, divided by R */
  double cv;          /* sqrt(sum (x - mean)^2 / (R - 1)) / mean; 0 when R == 1 */
  uint64_t r;         /* number of samples */
} asmv_timing;        /* 32 bytes */

typedef struct { double eps, k, s_floor; } asmv_gate_params;

/* Median, mean and coefficient of variation of r timing samples, each
 * operation in double in the order stated above.  EINVAL for a null
 * pointer, r == 0, or a sample that is not finite and positive. */
int asmv_timing_summary(const double *samples_ms, size_t r, asmv_timing *out);

/* Eq. 2: *m_star = (1 + max(eps, k * cv)) * s_best (multiply k*cv, take the
 * max, add 1, multiply by s_best), *commit = all_eq && s_cand >=
 * max(*m_star, s_floor).  EINVAL for null pointers, non-finite or negative
 * arguments, or s_best == 0. */
int asmv_commit_gate(int all_eq, double s_cand, double s_best, double cv,
                     const asmv_gate_params *params, double *m_star, int *commit);

/* Launch callback: enqueue the kernel(s) to time on `stream`. */
typedef void (*asmv_launch_fn)(void *user, asmv_stream_t stream);

/* Event-timed launches: `warmup` untimed calls of fn, then r calls, each
 * bracketed by its own pair of CUDA events recorded on `stream`;
 * samples_ms[i] is the device time of call i.  Synchronises the stream
 * once at the end.  Runs on the current CUDA device; the events are
 * created and destroyed inside the call.  EINVAL for a null fn or
 * samples_ms or r == 0; ECUDA if event creation, recording or timing
 * fails (the CUDA error is returned through *cuda_error when it is not
 * null). */
int asmv_time_launches(asmv_launch_fn fn, void *user, int warmup, size_t r,
                       double *samples_ms, asmv_stream_t stream, int *cuda_error);

/* ---------------------------------------------------------------------
 * Tier 2 replay (Sec. 3.4): a captured dispatch is replayed against memory
 * restored to its captured pre-dispatch state, at the original virtual
 * addresses when the kernel arguments hold absolute pointers.
 * ------------------------------------------------------------------- */

/* Restore: for each region i, copy payload_bytes(i) bytes from the device
 * address src[i] (the captured pre-dispatch payload, any alignment) into
 * the region's payload, and write the region's canary over both guard
 * bands.  One kernel for the whole table; asynchronous on `stream`.
 * EINVAL: as asmv_fill's table rules without the distribution rules
 * (allocations must not overlap), a null src with n > 0, a null src[i]
 * for a non-empty payload, a source that is not device memory of ctx's
 * device or that overlaps a region's allocation. */
int asmv_restore(asmv_ctx *ctx, const asmv_region *regions, const uint64_t *src, size_t n,
                 asmv_stream_t stream);

/* Capture: for each region i, copy its payload into the device address
 * dst[i] (payload_bytes(i) bytes, any alignment); guard bands are neither
 * read nor written.  Asynchronous on `stream`.  EINVAL as asmv_restore,
 * with destinations that must not overlap one another or any region. */
int asmv_capture(asmv_ctx *ctx, const asmv_region *regions, const uint64_t *dst, size_t n,
                 asmv_stream_t stream);

/* Device memory at a chosen virtual address.  asmv_va_map reserves `bytes`
 * (rounded up to the allocation granularity) of virtual address space at
 * `addr` (0: the driver chooses), backs it with physical memory of
 * `device`, maps it and grants the device read/write access.  addr must be
 * a multiple of asmv_va_granularity(device).  EINVAL for a null out, zero
 * bytes, a misaligned addr, or an addr whose range the driver cannot give
 * (in use); ENOMEM when memory is short; ECUDA otherwise.  Memory from
 * asmv_va_map is valid in every call above.  asmv_va_unmap waits for the
 * device to go idle, then unmaps and frees. */
typedef struct asmv_va asmv_va;
int asmv_va_granularity(int device, size_t *out);
int asmv_va_map(int device, uint64_t addr, size_t bytes, asmv_va **out);
uint64_t asmv_va_address(const asmv_va *va);
size_t asmv_va_size(const asmv_va *va);
int asmv_va_unmap(asmv_va *va);

/* Host-only validation of a region table, the checks every call above
 * makes before touching the device, except the device-memory checks.
 * for_fill != 0 adds the distribution and overlap rules of asmv_fill.
 * Makes no CUDA call.  Returns ASMV_OK or ASMV_EINVAL. */
int asmv_check_regions(const asmv_region *regions, size_t n, int for_fill);

/* The order in which asmv_fill lays out the table's tiles (Sec. 3.4, Tier 1:
 * the fill itself does not depend on it): order[k] is the table index of the
 * k-th region, the regions grouped by the code that fills them
 * (distribution, then dtype; RAW of any dtype is one kind) and in table
 * order within a kind.  order holds n entries, owned by the caller.  Host
 * only, no CUDA call; returns ASMV_EINVAL for a table asmv_fill would reject
 * (order untouched) or a null order with n > 0. */
int asmv_fill_order(const asmv_region *regions, size_t n, uint32_t *order);

/* Kernel timing: when enabled, each call records CUDA events around its
 * kernel launch on the call's stream; asmv_ctx_kernel_ms then returns the
 * device time of the last call's kernel (waiting for it to finish).
 * EINVAL for a null ctx or ms, or when timing is off / nothing ran. */
int asmv_ctx_set_timing(asmv_ctx *ctx, int enable);
int asmv_ctx_kernel_ms(asmv_ctx *ctx, float *ms);

/* The CUDA error code behind the last ASMV_ECUDA on this context (0 if none). */
int asmv_ctx_cuda_error(const asmv_ctx *ctx);

/* Number of kernels this context has launched since creation. */
uint64_t asmv_ctx_launches(const asmv_ctx *ctx);

/* Every device wait of the compare pipeline is bounded: ASMV_WAIT_ROUNDS
 * tries of up to 100 us.  A wait that runs out sets the launch's error word,
 * the kernel lets the copies it issued land and returns, and the call
 * returns ASMV_ETIMEOUT with out_host untouched and the context usable.
 * This sets, per context, the bound of one of those waits: the copy
 * producer's wait for a stage the checking warps have released.  Meant for
 * tests of the timeout path: with 0 the producer gives up as soon as it
 * needs a stage back (in any CTA with more than four tiles), its checking
 * warps then wait in vain for the next tile until their own default bound
 * runs out (about 2 s), and the call returns ASMV_ETIMEOUT.  EINVAL for a
 * null ctx. */
#define ASMV_WAIT_ROUNDS 20000u
int asmv_ctx_set_wait_rounds(asmv_ctx *ctx, uint32_t rounds);

/* Bound the SMs that the launches of ctx may occupy: every later call sizes
 * its persistent grid as if the device had `sms` SMs (0, or a value at or
 * above the device's count, restores all of them), which leaves the other
 * SMs to work on other streams.  Results do not depend on the bound.
 * ASMV_EINVAL for a null ctx or a negative count. */
int asmv_ctx_set_sm_limit(asmv_ctx *ctx, int sms);

/* The debug-bounds build.  libasmv_debug.so is this library compiled with
 * device bounds checks (ASMV_DEBUG_BOUNDS=1): every region descriptor and
 * guard segment carries the allocation it lies in, and every global load
 * and store of the fill, the compare (bulk copies into shared memory, the
 * byte-granular reads of ragged chunks, the guard reads) and the restore /
 * capture is checked against it.  An access outside is skipped, never
 * made: the kernel sets a bit in the launch's error word and goes on, and
 * the call returns ASMV_EBOUNDS (the fill and the restore then read the
 * word back and synchronise their stream).  Results are otherwise those of
 * the normal build, bit for bit.  The Eq. 1 sums kernels are not checked.
 * asmv_debug_bounds() returns 1 in that build and 0 in the normal one. */
int asmv_debug_bounds(void);

/* Test hook of the debug-bounds build: every later asmv_fill on ctx runs its
 * payload loop `bytes` past the end of each non-empty payload, while the
 * allocations it checks against stay those of the table, so the checks
 * refuse the extra stores.  A test gives the region an allocation larger
 * than the table says, so that even an unchecked store would stay inside
 * real memory.  0 turns it off.  ASMV_EINVAL for a null ctx, and in the
 * normal build, where the hook does not exist. */
int asmv_ctx_debug_widen(asmv_ctx *ctx, uint64_t bytes);

/* Static description of a status code. */
const char *asmv_strerror(int status);

/* ASMV_ABI_VERSION of the loaded library. */
int asmv_abi_version(void);

/* Size of the fixed device scratch behind asmv_compare_noalloc. */
#define ASMV_NOALLOC_SCRATCH_BYTES (1u << 20)

/* asmv_compare for callers that must not allocate memory (the paper has no
 * counterpart; this is a convenience of this library).  A harness that
 * replays captured dispatches at their original virtual addresses needs
 * its reserved address space left untouched, and one that times candidate
 * kernels cannot take the device-wide synchronisation an allocation may
 * bring; neither can create a context, whose workspace and staging are
 * allocated.  This call needs no context, and once the library's device
 * code is loaded on a device it allocates nothing: the launch plan and the
 * statistics live in a file-scope device array of
 * ASMV_NOALLOC_SCRATCH_BYTES, staged through a static host buffer.
 *   - Loading.  With lazy module loading (the CUDA default) the library's
 *     device code, and this array with it, is placed in device memory the
 *     first time the context uses it, so the first call on a device (or any
 *     earlier call of this library on it) does allocate.  A caller that
 *     reserves or replays fixed addresses must make one call of its own
 *     (an empty table, n = 0 with valid tolerances, does not load; use a
 *     one-region table) before it reserves them.  The array then stays in
 *     the context until the context is destroyed.
 *   - Runs on the calling thread's current CUDA device.  Every call looks
 *     up the array's address in the current context (this allocates
 *     nothing), so a context that was reset and created again is handled.
 *   - Stream capture: the call copies its plan from pageable host memory
 *     and synchronises its stream, both of which are illegal while a stream
 *     is being captured.  It must not be called while its stream, or any
 *     other stream, is being captured.
 *   - ref/cand/n/tol/out_host/stream as asmv_compare (one candidate).
 *   - The plan must fit the scratch: regions (32 B each, plus one), one
 *     candidate address (8 B) and one statistics entry (64 B) per region,
 *     32 B per 4 KiB of guard band on either side, each part rounded to
 *     256 B, plus one 64-byte error entry.  Larger tables, and every table
 *     asmv_compare would reject, return ASMV_EINVAL.
 *   - Every call reuses the same scratch and overwrites the previous
 *     call's contents (the statistics are reset by each call).  Calls that
 *     overlap on the GPU, on any streams or host threads, race; host
 *     threads are serialised by a lock, but the caller must order the GPU
 *     work of successive calls (the call synchronises its own stream).
 * Returns ASMV_OK, ASMV_EINVAL, ASMV_ECUDA or ASMV_ETIMEOUT. */
int asmv_compare_noalloc(const asmv_region *ref, const asmv_region *cand, size_t n,
                         const asmv_tol *tol, asmv_stats *out_host, asmv_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* ASMV_H_ */
