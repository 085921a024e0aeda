// compare.cu -- the equivalence check of AsmEvo Eq. 1 applied per element
// to captured output regions (Sec. 3.2 R2; Sec. 3.4 Tier 2: floats within
// tolerance, integers / opaque bytes / guard bands byte-exact), for one
// reference against K <= 8 candidates in one pass.
//
// Statistics are defined in fp64 on exactly decoded values:
//   d = RN64(|c - r|), bound = RN64(atol + RN64(rtol*|r|)), mismatch iff
//   d > bound; max_abs = max d, max_rel = max RN64(d/|r|) over finite pairs.
// GB300's fp64 rate is far below what a per-element fp64 evaluation at HBM
// speed would need, so every element first goes through an fp32 screen
// that decides the common cases exactly and sends the rest to the fp64
// path.  Let D = |c - r| (exact real), s32 = RN32(c - r), as = |s32|,
// b = atol + rtol*|r| (exact real), B the fp64 bound above.
//
//  (1) Definite match: as < lo, lo = RN32(rlo*|r| + alo) with
//      rlo <= rtol(1-2^-21), alo <= atol(1-2^-21) (alo = -2^-100 when
//      atol < 2^-100).  lo > 0 forces b > 2^-100; then
//      D <= as(1+2^-24) < lo(1+2^-24) <= b(1-2^-22) < B, so d <= B.
//      (Differences below 2^-125 are exact in fp32, so no subnormal slack
//      is needed on as.)
//  (2) Definite mismatch: hi < as <= FLT_MAX, hi = RN32(rhi*|r| + ahi) with
//      rhi >= rtol(1+2^-21), ahi >= atol(1+2^-21) + 2^-100; then
//      D >= as(1-2^-24) > b(1+2^-22) + 2^-101 > B, so d > B.
//  Anything else (ambiguous band, NaN/Inf on either side, fp32 overflow of
//  c - r) is evaluated exactly in fp64.
//  (3) max_abs: when as < |r|/2 the pair is within a factor of two, so
//      c - r is exact in fp32 (Sterbenz) and as equals D; such "plain"
//      elements update an fp32 running maximum m32 with fmaxf, exactly.
//      Every other element goes to the exact path, which keeps the fp64
//      maximum of RN64(D).  max_abs = max(m32, that maximum).
//  (4) max_rel: a thread keeps its exact maximum Rmax and T = RD32(Rmax).
//      An element with as < |r|/2 is plain (as = D = d, see (3)), and it
//      can raise the maximum only if RN64(D/|r|) > Rmax, hence only if
//      D/|r| > Rmax >= T, i.e. as > T*|r| (RN64 is monotone and Rmax is a
//      double).  The screen flags as > y, y = RD32(Tp*|r|) (one fma rounded
//      down), Tp = min(T, 1/2 -): as > Tp*|r| >= y.  An element whose
//      relative error equals Rmax (as = T*|r| exactly) is not flagged and
//      cannot change the maximum; as = 0 is never flagged.  Flagged
//      elements get the exact RN64(d/|r|).  Since y <= Tp*|r| < |r|/2,
//      every element with as >= |r|/2 -- every element whose c - r may be
//      inexact -- is flagged as well, and r = 0 makes y = 0, so every
//      nonzero difference from a zero reference is flagged.
//  The 16-bit and 8-bit formats are screened in their own format instead
//  (fp16, each fp8 format through its exact fp16 value, bf16), two
//  elements per packed instruction.  With s = RN(c - r) in the format,
//  a = |s|, and per reference element (formed once for all candidates)
//  lo = max(RZ(lo32), 0), hi = RZ(hi32), where lo32 and hi32 are the fp32
//  bounds of (1) and (2) and RZ rounds them to the format toward zero,
//  and y = max(RN(T'*|r| - tiny), 0), tiny the format's least subnormal:
//  (5) The bracket: where c - r is exact (see (6)), a = D is a value of the
//      format.  a <= lo gives D <= lo32 < B (proof (1); lo = 0 gives D = 0),
//      a match.  a > hi gives a > hi32, since a and hi are values of the
//      format and RZ rounds the non-negative hi32 down, hence D > B (proof
//      (2)), a mismatch.  So the band left to the exact path, lo < a <= hi,
//      holds a value of the format only where one lies within the 2^-21
//      margins of the fp32 bounds.
//  (6) y <= T|r| and y < |r|/2: T' = RD(Tp (1 - m)) with Tp = min(T, 1/2-),
//      m = 2^-9 (fp16) or 2^-7 (bf16), which covers the rounding of the
//      multiply-add (2^-11, resp. 2^-9, relatively; tiny/2 absolutely);
//      so y <= T'|r| (1 + 2^-11) < Tp|r| or, subnormal, y <= T'|r| - tiny/2;
//      the max with 0 keeps y >= 0.  An element with a <= y is therefore
//      exact (if c - r were inexact, |c - r| >= |r| / 2 by Sterbenz's lemma
//      and exact subnormal arithmetic, so a >= RN(|r|/2) > y) and cannot
//      raise max_rel (a/|r| <= T <= Rmax, and RN64 is monotone).
//  (7) Elements with a > y (compared unordered, so a NaN difference counts)
//      and ambiguous elements (lo < a <= hi) send the chunk to the exact
//      path.  |r| is replaced by NaN where r is not finite (|r|*0 + |r|),
//      which makes y = 0 there (and hi infinite or NaN, never exceeded), so
//      every non-finite value on either side is flagged: y is finite
//      wherever r is, and an infinite or NaN difference is not below it.  Otherwise d = a, a match iff
//      a <= lo, a mismatch iff a > hi, and max_abs takes the running
//      maximum of a in the format (exact).  The fp32 screen takes the same
//      NaN |r|, with which neither (1) nor (2) can hold.
// The maxima are order-independent (max of exact values), counts are sums
// and first_mismatch a minimum, so any grid gives bit-identical results.
//
// Work split: one CTA of 16 warps per SM.  The last warp streams each tile
// of the reference and of the K <= 8 candidates into shared memory with
// bulk copies (two to four stages, as fit, mbarrier-completed).  Each of the
// 15 checking warps takes whole rows of 32 chunks of the tile and checks
// every candidate against them: a lane reads its reference chunk once,
// forms its per-element bounds once, and screens the K candidate chunks at
// the same position, so neither device memory nor the screen's reference
// work is paid per candidate.  Chunks the screen cannot settle are queued
// per warp with their candidate and drained lane-parallel; their statistics
// go to the warp's per-candidate entries in shared memory.  A lane keeps
// the screen's counts and maxima per candidate in registers, and the warp
// merges them into the global entries when its CTA moves to the next
// region.  Sixteen warps in all, four per SM sub-partition, leave each
// thread 128 registers (a seventeenth would put five warps on one
// sub-partition and cap every thread at 96, which spilled in the candidate
// loop): 5088 GB/s against 4864 with 16 checking warps, and 2788 with 8
// (fp16 [32768,32768] x 8 candidates).
//
// Roofline: HBM reads of reference + candidate payloads (reference once per
// launch of up to 8 candidates).  The packed screen is about 12 instructions
// per pair of candidate elements plus 3 per reference pair shared by the
// candidates.
#include <float.h>
#include <math_constants.h>
#include <atomic>
#include <mutex>
#include "device.cuh"

namespace asmv {
namespace {

struct Hot {
  uint32_t cnt;          // mismatches in the current region (per thread; < 2^32 for any HBM size)
  uint32_t nonfin;       // NaN/Inf-position mismatches
  unsigned long long first;   // lowest mismatching element index seen (~0 if none)
  float m32;             // exact max |c - r| over plain elements (see (3))
  float T;               // relative-error screen threshold
  // exact maxima as bit patterns of non-negative doubles (integer order =
  // numeric order), so that comparing them stays off the fp64 pipe
  unsigned long long dabs;   // max |c - r| over exact-path elements
  unsigned long long drel;   // max relative error
};

__device__ __forceinline__ unsigned long long dbits(double x) {
  return (unsigned long long)__double_as_longlong(x);
}

__device__ __forceinline__ float tfloor(double d) {
  return __double2float_rd(d);                               // <= d
}

__device__ __forceinline__ void rel_update(Hot &h, double d, double r64) {
  const double ar = fabs(r64);
  const double rel = (ar != 0.0) ? __ddiv_rn(d, ar) : (d == 0.0 ? 0.0 : CUDART_INF);
  const unsigned long long b = dbits(rel);
  if (b > h.drel) { h.drel = b; h.T = tfloor(rel); }
}

// rel_update for the binary64 and integer paths, where every differing
// element comes here: the exact RN64(d/|r|) enters the maximum only if it
// can exceed it, and a negative RN64(d - T|r|) (one fma; negative only when
// the exact value is) proves d/|r| < T <= Rmax, so the division is skipped.
__device__ __forceinline__ void rel_update_guarded(Hot &h, double d, double r64) {
  if (__fma_rn(-(double)h.T, fabs(r64), d) < 0.0) return;
  rel_update(h, d, r64);
}

// Exact fp64 evaluation of one float pair; returns the mismatch bit.
__device__ __forceinline__ uint32_t exact_float(float r, float c, Hot &h, const TolF &t) {
  const bool rn = isnan(r), cn = isnan(c), ri = isinf(r), ci = isinf(c);
  if (rn | cn | ri | ci) {
    const bool match = (rn && cn) || (ri && ci && (signbit(r) == signbit(c)));
    if (!match) h.nonfin++;
    return match ? 0u : 1u;
  }
  const double r64 = (double)r, c64 = (double)c;
  const double d = fabs(__dsub_rn(c64, r64));
  const double bound = __dadd_rn(t.atol, __dmul_rn(t.rtol, fabs(r64)));
  h.dabs = umax64(h.dabs, dbits(d));
  rel_update(h, d, r64);
  return d > bound ? 1u : 0u;
}

// Exact fp64 evaluation of one binary64 pair; returns the mismatch bit.
__device__ __forceinline__ uint32_t exact_double(double r64, double c64, Hot &h, const TolF &t) {
  const bool rn = isnan(r64), cn = isnan(c64), ri = isinf(r64), ci = isinf(c64);
  if (rn | cn | ri | ci) {
    const bool match = (rn && cn) || (ri && ci && (signbit(r64) == signbit(c64)));
    if (!match) h.nonfin++;
    return match ? 0u : 1u;
  }
  const double d = fabs(__dsub_rn(c64, r64));
  const double bound = __dadd_rn(t.atol, __dmul_rn(t.rtol, fabs(r64)));
  h.dabs = umax64(h.dabs, dbits(d));
  rel_update_guarded(h, d, r64);
  return d > bound ? 1u : 0u;
}

// Exact evaluation of one differing int64 pair: |c - r| formed in 128 bits
// (it can reach 2^64 - 1) and rounded once; |r| rounded once.
__device__ __forceinline__ void exact_int64(long long r, long long c, Hot &h) {
  const unsigned long long dlo = (c >= r) ? (unsigned long long)c - (unsigned long long)r
                                          : (unsigned long long)r - (unsigned long long)c;
  const double d = __ull2double_rn(dlo);               // |c - r| < 2^64 fits the unsigned difference
  h.dabs = umax64(h.dabs, dbits(d));
  rel_update_guarded(h, d, __ll2double_rn(r));
}

// Exact evaluation of one differing integer pair (always a mismatch).
__device__ __forceinline__ void exact_int(int64_t r, int64_t c, Hot &h) {
  const int64_t dd = c - r;
  const double d = (double)(dd < 0 ? -dd : dd);     // exact: |d| < 2^33
  h.dabs = umax64(h.dabs, dbits(d));
  rel_update_guarded(h, d, (double)r);
}

__device__ __forceinline__ uint32_t word_of(const uint4 &v, int w) {
  return w == 0 ? v.x : (w == 1 ? v.y : (w == 2 ? v.z : v.w));
}

template <uint32_t DT> struct Fmt;
template <> struct Fmt<kF32> { static constexpr int E = 4; };
template <> struct Fmt<kBF16> { static constexpr int E = 8; };
template <> struct Fmt<kF16> { static constexpr int E = 8; };
template <> struct Fmt<kF8> { static constexpr int E = 16; };
template <> struct Fmt<kI32> { static constexpr int E = 4; };
template <> struct Fmt<kI8> { static constexpr int E = 16; };
template <> struct Fmt<kU8> { static constexpr int E = 16; };
template <> struct Fmt<kF8E5M2> { static constexpr int E = 16; };
template <> struct Fmt<kF8E4FNUZ> { static constexpr int E = 16; };
template <> struct Fmt<kF8E5FNUZ> { static constexpr int E = 16; };
template <> struct Fmt<kF64> { static constexpr int E = 2; };
template <> struct Fmt<kI16> { static constexpr int E = 8; };
template <> struct Fmt<kI64> { static constexpr int E = 2; };


// Element j of a chunk decoded to fp32 (float dtypes; runtime j).
template <uint32_t DT>
__device__ __forceinline__ float elem_f32(const uint4 &v, int j) {
  if (DT == kF32) return __uint_as_float(word_of(v, j));
  if (DT == kBF16) return __uint_as_float(((word_of(v, j >> 1) >> (16 * (j & 1))) & 0xFFFFu) << 16);
  if (DT == kF16) return __half2float(__ushort_as_half((unsigned short)(word_of(v, j >> 1) >> (16 * (j & 1)))));
  const uint32_t b = (word_of(v, j >> 2) >> (8 * (j & 3))) & 0xFFu;
  return f16x2_to_f32(fp8x2_to_half2_bits<DT>(b)).x;
}

template <uint32_t DT>
__device__ __forceinline__ int64_t elem_int(const uint4 &v, int j) {
  if (DT == kI64) return (int64_t)(((unsigned long long)word_of(v, 2 * j + 1) << 32) | word_of(v, 2 * j));
  if (DT == kI16) return (int64_t)(int16_t)(word_of(v, j >> 1) >> (16 * (j & 1)));
  if (DT == kI32) return (int64_t)(int32_t)word_of(v, j);
  const uint32_t b = (word_of(v, j >> 2) >> (8 * (j & 3))) & 0xFFu;
  if (DT == kI8) return (int64_t)(int8_t)b;
  return (int64_t)b;
}

template <uint32_t DT>
__device__ __forceinline__ uint32_t elem_bits(const uint4 &v, int j) {
  return __float_as_uint(elem_f32<DT>(v, j));
}

template <uint32_t DT> __device__ __forceinline__ constexpr bool is_int_dt() {
  return DT == kI32 || DT == kI8 || DT == kU8 || DT == kI16 || DT == kI64;
}

// ---------------------------------------------------------------- queue
// Chunks the screen cannot settle are queued per warp in shared memory with
// their candidate, as copies, and re-examined element by element,
// lane-parallel, once the queue is half full after a row and when the
// warp's run over a region ends, instead of diverging inside the screen.
// 24 entries per warp leave room for three stages of the 8-candidate launch
// in the 227 KiB a CTA may take (with 32 it gets two: 5262 against 5772 GB/s).
constexpr uint32_t kQueue = 24;           // chunk entries per warp

struct QEntry {
  uint4 R, C;                             // the raw 16-byte chunks
  unsigned long long e0;                  // element index of the chunk's first element
  uint32_t k, pad_;                       // the candidate
};

struct Queue {
  QEntry e[kQueue];
  uint32_t count;
};

// A warp's statistics of one candidate that do not live in its lanes'
// registers: everything the exact path finds, and the first mismatch the
// screen finds.  In shared memory, merged with shared-memory atomics.
struct ExactStats {
  unsigned long long first, dabs, drel;
  uint32_t cnt, nonfin, m32;              // m32: bits of a non-negative float
  uint32_t th;                            // the screen's relative-error threshold (rel_threshold of drel)
};

// Shared memory of a compare CTA: [barriers][queues][exact statistics]
// [stages].  Declared once here so that every function that takes a part
// of it addresses it as shared memory.
extern __shared__ __align__(128) unsigned char cmp_smem[];
constexpr uint32_t kQueueOff = 128;
constexpr uint32_t kExactOff = kQueueOff + kConsumerWarps * sizeof(Queue);
constexpr uint32_t kStageOff = (kExactOff + kConsumerWarps * kMaxCands * sizeof(ExactStats) + 127) / 128 * 128;
static_assert(kStages * 2 * sizeof(uint64_t) <= kQueueOff, "barriers overlap the queues");

__device__ __forceinline__ Queue *queue_of(uint32_t warp) {
  return reinterpret_cast<Queue *>(cmp_smem + kQueueOff) + warp;
}
__device__ __forceinline__ ExactStats *exact_of(uint32_t warp) {
  return reinterpret_cast<ExactStats *>(cmp_smem + kExactOff) + warp * kMaxCands;
}

// 0.5 (1 - 2^-20): below this fraction of |r|, c - r is exact in fp32.
#define ASMV_HALF_LESS 0x1.fffff8p-2f

// Exact bookkeeping of one differing float element of a queued chunk: the
// fp32 screen again, with fp64 only for what it cannot settle (ambiguous
// band, non-finite values, |c-r| >= |r|/2, or a possible new max_rel).
__device__ __forceinline__ uint32_t settle_float(float r, float c, Hot &h, const TolF &t) {
  const float s = __fsub_rn(c, r);
  const float as = fabsf(s), ar = fabsf(r);
  const bool ok = as < __fmaf_rn(t.rlo, ar, t.alo);
  const bool bad = (as > __fmaf_rn(t.rhi, ar, t.ahi)) & (as <= FLT_MAX);
  const bool plain = as < __fmul_rn(0.5f, ar);          // c - r exact (Sterbenz)
  if ((ok | bad) && plain) {
    h.m32 = fmaxf(h.m32, as);
    if (!(__fmaf_rn(-h.T, ar, as) < 0.0f)) rel_update(h, (double)as, (double)r);
    return bad ? 1u : 0u;
  }
  return exact_float(r, c, h, t);
}

template <uint32_t DT>
__device__ __forceinline__ void settle_chunk(const QEntry &e, Hot &h, const TolF &t) {
  constexpr int E = Fmt<DT>::E;
  uint32_t bad = 0;
#pragma unroll 1
  for (int j = 0; j < E; ++j) {
    if (DT == kI64) {
      const int64_t r = elem_int<DT>(e.R, j), c = elem_int<DT>(e.C, j);
      if (r != c) { exact_int64(r, c, h); bad |= 1u << j; }
    } else if (is_int_dt<DT>()) {
      const int64_t r = elem_int<DT>(e.R, j), c = elem_int<DT>(e.C, j);
      if (r != c) { exact_int(r, c, h); bad |= 1u << j; }
    } else if (DT == kF64) {
      const unsigned long long rb = ((unsigned long long)word_of(e.R, 2 * j + 1) << 32) | word_of(e.R, 2 * j);
      const unsigned long long cb = ((unsigned long long)word_of(e.C, 2 * j + 1) << 32) | word_of(e.C, 2 * j);
      if (rb != cb)
        bad |= exact_double(__longlong_as_double((long long)rb), __longlong_as_double((long long)cb), h,
                            t) << j;
    } else {
      const uint32_t rb = elem_bits<DT>(e.R, j), cb = elem_bits<DT>(e.C, j);
      if (rb != cb) bad |= settle_float(__uint_as_float(rb), __uint_as_float(cb), h, t) << j;
    }
  }
  if (bad) {
    h.cnt += __popc(bad);
    h.first = umin64(h.first, e.e0 + (unsigned long long)(__ffs(bad) - 1));
  }
}

__device__ __forceinline__ void reset_hot(Hot &h) {
  h.cnt = 0; h.nonfin = 0; h.first = ~0ull;
  h.m32 = 0.0f; h.T = 0.0f; h.dabs = 0; h.drel = 0;
}


// Settle one queued chunk exactly and merge its statistics into the warp's
// entry of its candidate.  The exact path's relative-error threshold is the
// entry's current maximum (any value not above the maximum is valid).
template <uint32_t DT>
__device__ __forceinline__ void settle_into(const QEntry &e, ExactStats *ex, const TolF &t) {
  ExactStats &x = ex[e.k];
  Hot h;
  reset_hot(h);
  h.T = tfloor(__longlong_as_double((long long)x.drel));
  settle_chunk<DT>(e, h, t);
  if (h.cnt) atomicAdd(&x.cnt, h.cnt);
  if (h.nonfin) atomicAdd(&x.nonfin, h.nonfin);
  if (h.first != ~0ull) atomicMin(&x.first, h.first);
  if (h.m32 > 0.0f) atomicMax(&x.m32, __float_as_uint(h.m32));
  if (h.dabs) atomicMax(&x.dabs, h.dabs);
  if (h.drel) atomicMax(&x.drel, h.drel);
}

template <uint32_t DT> __device__ __forceinline__ uint32_t rel_threshold(unsigned long long drel);

// Drain the warp's queue: lanes take chunks in turn; then the screen's
// thresholds of the K candidates follow their new maxima.
template <uint32_t DT>
__device__ __forceinline__ void drain(uint32_t warp, uint32_t K, const TolF *tp) {
  Queue *q = queue_of(warp);
  ExactStats *ex = exact_of(warp);
  const TolF t = *tp;
  __syncwarp();
  const uint32_t n = min(q->count, kQueue), lane = threadIdx.x & 31;
  for (uint32_t j = lane; j < n; j += 32) settle_into<DT>(q->e[j], ex, t);
  __syncwarp();
  if (lane == 0) q->count = 0;
  if (lane < K) ex[lane].th = rel_threshold<DT>(ex[lane].drel);
  __syncwarp();
}

// Queue a chunk of candidate k; false if the queue is full (the caller
// drains it and tries again).
__device__ __forceinline__ bool try_push(const uint4 &R, const uint4 &C, unsigned long long e0, uint32_t k,
                                         Queue *q) {
  const uint32_t slot = atomicAdd(&q->count, 1u);
  if (slot >= kQueue) return false;
  QEntry e;
  e.R = R; e.C = C; e.e0 = e0; e.k = k; e.pad_ = 0u;
  q->e[slot] = e;
  return true;
}

// ---------------------------------------------------------------- screens
// Which screen a dtype takes: packed in the stored format (fp16, the fp8
// formats through fp16, bf16), scalar fp32, or none (integers, opaque
// bytes and binary64 chunks that differ always take the exact path).
template <uint32_t DT> __device__ __forceinline__ constexpr bool packed_dt() {
  return DT == kF16 || DT == kBF16 || is_fp8(DT);
}
template <uint32_t DT> __device__ __forceinline__ constexpr int pairs_of() {
  return is_fp8(DT) ? 8 : 4;               // packed words per chunk
}

// One packed word in the screen's format (fp16 for fp16 and fp8, bf16).
template <uint32_t DT> struct P2 { using T = __half2; };
template <> struct P2<kBF16> { using T = __nv_bfloat162; };

template <class T> __device__ __forceinline__ T as2(uint32_t w) { return *reinterpret_cast<const T *>(&w); }
template <class T> __device__ __forceinline__ uint32_t bits2(T v) { return *reinterpret_cast<const uint32_t *>(&v); }

// Packed word p of a chunk in the screen's format: fp16 and bf16 words as
// stored, fp8 bytes 2p, 2p+1 widened to their exact fp16 values.
template <uint32_t DT>
__device__ __forceinline__ uint32_t word2(const uint4 &v, int p) {
  if (is_fp8(DT)) return fp8x2_to_half2_bits<DT>(word_of(v, p >> 1) >> (16 * (p & 1)));
  return word_of(v, p);
}

// The screen's per-candidate threshold from the warp's exact maximum of the
// relative error: Tp = min(RD32(max), 1/2-) as a float (fp32 screen), or
// T' = RD(Tp (1 - m)) in the packed format, in both halves (see (6)).
template <uint32_t DT>
__device__ __forceinline__ uint32_t rel_threshold(unsigned long long drel) {
  const float Tp = fminf(tfloor(__longlong_as_double((long long)drel)), ASMV_HALF_LESS);
  if (DT == kBF16) {
    const uint32_t h = __bfloat16_as_ushort(__float2bfloat16_rd(__fmul_rd(Tp, 1.0f - 0x1p-7f)));
    return h | (h << 16);
  }
  if (packed_dt<DT>()) {
    const uint32_t h = __half_as_ushort(__float2half_rd(__fmul_rd(Tp, 1.0f - 0x1p-9f)));
    return h | (h << 16);
  }
  return __float_as_uint(Tp);
}

// A lane's screen statistics of one candidate (its threshold is warp-wide,
// in ExactStats::th).
struct Cand {
  uint32_t cnt;        // mismatches the screen settled
  uint32_t cm;         // running maximum of |c - r| over settled elements: packed bits, or float bits
};

// Two non-negative floats rounded toward zero (= down) to the screen's
// format; x in the low half.
template <uint32_t DT>
__device__ __forceinline__ uint32_t rz_pack(float2 v) {
  uint32_t d;
  if (DT == kBF16) asm("cvt.rz.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(v.y), "f"(v.x));
  else asm("cvt.rz.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(v.y), "f"(v.x));
  return d;
}

// A packed word of the screen's format as two exact floats.
template <uint32_t DT>
__device__ __forceinline__ float2 widen2(uint32_t w) {
  if (DT == kBF16) return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
  return f16x2_to_f32(w);
}

// The reference side of a chunk, formed once for all candidates.
template <uint32_t DT> struct RefPrep {
  static constexpr int NP = pairs_of<DT>();
  uint32_t r[NP], ar[NP], lo[NP], hi[NP];  // packed: r, |r|, lo, hi; fp32: floats (NP = 4)
};

// The fp32 bounds' constants, held in registers by the checking loop.
struct Bounds {
  float rlo, alo, rhi, ahi;
};

template <uint32_t DT>
__device__ __forceinline__ void prepare(const uint4 &R, const Bounds &b, RefPrep<DT> &P) {
  if (packed_dt<DT>()) {
    using T2 = typename P2<DT>::T;
    const T2 zero = as2<T2>(0u);
#pragma unroll
    for (int p = 0; p < RefPrep<DT>::NP; ++p) {
      P.r[p] = word2<DT>(R, p);
      // |r|, or NaN where r is not finite (|r| * 0 + |r|), so that y = 0 there
      const T2 ar0 = __habs2(as2<T2>(P.r[p]));
      P.ar[p] = bits2(__hfma2(ar0, zero, ar0));
      const float2 f = widen2<DT>(bits2(ar0));
      const float2 lo = make_float2(__fmaf_rn(b.rlo, f.x, b.alo), __fmaf_rn(b.rlo, f.y, b.alo));
      const float2 hi = make_float2(__fmaf_rn(b.rhi, f.x, b.ahi), __fmaf_rn(b.rhi, f.y, b.ahi));
      P.lo[p] = bits2(__hmax2(as2<T2>(rz_pack<DT>(lo)), zero));
      P.hi[p] = rz_pack<DT>(hi);
    }
  } else {
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float r = __uint_as_float(word_of(R, w)), ar = __fmaf_rn(fabsf(r), 0.0f, fabsf(r));
      P.r[w] = __float_as_uint(r);
      P.ar[w] = __float_as_uint(ar);
      P.lo[w] = __float_as_uint(__fmaf_rn(b.rlo, ar, b.alo));
      P.hi[w] = __float_as_uint(__fmaf_rn(b.rhi, ar, b.ahi));
    }
  }
}

// Screen one candidate chunk C against the prepared reference chunk.
// Returns true when the chunk needs the exact path; otherwise `bad` holds
// its definite mismatches (packed screens: bit p for element 2p, bit 16 + p
// for element 2p + 1; fp32: bit w for element w) and the lane's running
// maximum of |c - r| takes the chunk's.
template <uint32_t DT>
__device__ __forceinline__ bool screen_chunk(const RefPrep<DT> &P, const uint4 &C, uint32_t thr, Cand &cd,
                                             uint32_t &bad) {
  uint32_t rare = 0, b = 0;
  if (packed_dt<DT>()) {
    using T2 = typename P2<DT>::T;
    const T2 zero = as2<T2>(0u);
    const T2 negtiny = as2<T2>(0x80018001u);               // -(least subnormal), both halves
    const T2 th = as2<T2>(thr);
    T2 cmc = zero;
#pragma unroll
    for (int p = 0; p < RefPrep<DT>::NP; ++p) {
      const T2 s = __hsub2(as2<T2>(word2<DT>(C, p)), as2<T2>(P.r[p]));
      const T2 a = __habs2(s);
      const T2 y = __hmax2(__hfma2(th, as2<T2>(P.ar[p]), negtiny), zero);
      const uint32_t mlo = __hgt2_mask(a, as2<T2>(P.lo[p]));
      const uint32_t mhi = __hgt2_mask(a, as2<T2>(P.hi[p]));
      const uint32_t my = __hgtu2_mask(a, y);              // unordered: NaN is flagged
      rare |= my | (mlo & ~mhi);
      b |= mhi & (0x00010001u << p);
      cmc = __hmax2(cmc, a);
    }
    if (rare) return true;
    cd.cm = bits2(__hmax2(as2<T2>(cd.cm), cmc));
  } else {
    const float Tp = __uint_as_float(thr);
    float cmc = 0.0f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float s = __fsub_rn(__uint_as_float(word_of(C, w)), __uint_as_float(P.r[w]));
      const float as = fabsf(s), ar = __uint_as_float(P.ar[w]);
      const bool ok = as < __uint_as_float(P.lo[w]);
      const bool bd = as > __uint_as_float(P.hi[w]);
      rare |= (uint32_t)((!(ok | bd)) | (as > __fmul_rd(Tp, ar)));
      b |= (bd ? 1u : 0u) << w;
      cmc = fmaxf(cmc, as);
    }
    if (rare) return true;
    cd.cm = __float_as_uint(fmaxf(__uint_as_float(cd.cm), cmc));
  }
  bad = b;
  return false;
}

// The lowest element of a chunk's mismatch bits (see screen_chunk).
template <uint32_t DT>
__device__ __forceinline__ uint32_t first_of(uint32_t bad) {
  if (packed_dt<DT>()) {
    const uint32_t ev = __ffs(bad & 0xFFFFu), od = __ffs(bad >> 16);      // 1-based, 0 if none
    const uint32_t e = ev ? 2u * (ev - 1u) : 64u, o = od ? 2u * (od - 1u) + 1u : 64u;
    return min(e, o);
  }
  return __ffs(bad) - 1u;
}

// The value of a lane's running maximum (packed: the larger half).
template <uint32_t DT>
__device__ __forceinline__ float cm_value(uint32_t cm) {
  if (DT == kBF16) {
    const float2 f = __bfloat1622float2(as2<__nv_bfloat162>(cm));
    return fmaxf(f.x, f.y);
  }
  if (packed_dt<DT>()) {
    const float2 f = __half22float2(as2<__half2>(cm));
    return fmaxf(f.x, f.y);
  }
  return __uint_as_float(cm);
}

__device__ __forceinline__ uint4 load_chunk(uint64_t base, uint64_t c, uint64_t full, uint64_t bytes,
                                            bool vec) {
  if (vec && c < full) return ldg16(base + 16 * c);
  return load_bytes(base + 16 * c, (uint32_t)umin64(16, bytes - 16 * c));
}

// Chunk c of region ri read from device memory: the reference (k < 0) or
// candidate k.  In the debug-bounds build a read outside the allocation is
// skipped (zeros) and reported.
__device__ __forceinline__ uint4 load_region_chunk(const CmpParams &p, uint32_t ri, const CmpRegion &r, int k,
                                                   uint64_t c) {
  const uint64_t base = k < 0 ? r.ref : p.cands[(size_t)k * p.nregions + ri];
#if ASMV_DEBUG_BOUNDS
  const Span sp = k < 0 ? r.alloc : p.cand_allocs[(size_t)k * p.nregions + ri];
  if (!in_alloc(sp, base + 16 * c, umin64(16, r.bytes - 16 * c), p.err)) return make_uint4(0u, 0u, 0u, 0u);
#endif
  return load_chunk(base, c, r.bytes >> 4, r.bytes, false);
}

// ---------------------------------------------------------------- pipeline
// mbarrier helpers (shared::cta addresses).  Waits are bounded: after
// `rounds` tries of up to kWaitHintNs each, the wait reports failure.  The
// producer's wait for a free stage takes the launch's bound
// (CmpParams::wait_rounds; 0 gives up without trying, which makes its
// consumers' waits run out: the test of this path); every other wait takes
// kWaitRounds.
constexpr uint32_t kWaitHintNs = 100000;

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{ .reg .b64 st; mbarrier.arrive.shared::cta.b64 st, [%0]; }" :: "r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t tx) {
  asm volatile("{ .reg .b64 st; mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1; }"
               :: "r"(bar), "r"(tx) : "memory");
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t rounds) {
  for (uint32_t i = 0; i < rounds; ++i) {
    uint32_t done;
    asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;"
                 " selp.u32 %0, 1, 0, p; }"
                 : "=r"(done) : "r"(bar), "r"(parity), "r"(kWaitHintNs) : "memory");
    if (done) return true;
  }
  return false;
}
// 1-D bulk copy global -> shared, completing `bytes` on the mbarrier.
__device__ __forceinline__ void bulk_load(uint32_t dst, uint64_t src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}

// Tile geometry of tile t of region r (tile_bytes per tile).
struct TileInfo {
  uint64_t off;        // byte offset of the tile in the payload
  uint32_t nloc;       // 16-byte chunks in the tile (last may be short)
  uint32_t nsm;        // chunks staged in shared memory (whole 16-byte chunks of vec regions)
};
__device__ __forceinline__ TileInfo tile_info(const CmpRegion &r, uint64_t t, uint32_t tile_bytes) {
  TileInfo ti;
  ti.off = (t - r.tile0) * (uint64_t)tile_bytes;
  const uint64_t nb = umin64(tile_bytes, r.bytes - ti.off);
  ti.nloc = (uint32_t)((nb + 15) >> 4);
  ti.nsm = r.vec ? (uint32_t)(nb >> 4) : 0u;
  return ti;
}

// Pipeline position shared by a consumer warp's calls: the next stage and
// the phase its full barrier completes next (the stage index wraps at the
// launch's depth, and the phase flips with each wrap).
struct Cursor {
  uint32_t s;          // stage of the next tile
  uint32_t ph;         // parity of its full barrier's next phase
  uint32_t ok;         // every wait succeeded
};

// One lane's chunk i of a tile against every candidate.  STAGED: the
// reference and every candidate chunk are in the stage (the common case);
// otherwise (the short last chunk of a region, or a region not 16-byte
// aligned) they are read from device memory.  Chunks the screen cannot
// settle are queued; bit k of `retry` is set where the queue was full.
template <uint32_t DT, int KMAX, bool STAGED>
__device__ __forceinline__ void check_chunk(const CmpParams &p, uint32_t ri, const CmpRegion &r,
                                            const uint4 *stage, uint32_t tbc, uint64_t c, uint32_t K,
                                            const Bounds &bnd, Queue *q, ExactStats *ex,
                                            Cand (&cs)[KMAX], uint32_t &found, uint32_t &retry) {
  constexpr int E = Fmt<DT>::E;
  // With one candidate the reference side is prepared only for a chunk that
  // differs (most chunks of a nearly equal candidate do not); with several,
  // once before the candidates.
  constexpr bool kScreened = !is_int_dt<DT>() && DT != kF64;
  const uint4 R = STAGED ? stage[0] : load_region_chunk(p, ri, r, -1, c);
  RefPrep<DT> P;
  if (kScreened && KMAX > 1) prepare<DT>(R, bnd, P);
#pragma unroll
  for (int k = 0; k < KMAX; ++k) {
    if (k >= (int)K) break;
    const uint4 C = STAGED ? stage[(1 + k) * tbc] : load_region_chunk(p, ri, r, k, c);
    if (((R.x ^ C.x) | (R.y ^ C.y) | (R.z ^ C.z) | (R.w ^ C.w)) == 0u) continue;
    if (kScreened && KMAX == 1) prepare<DT>(R, bnd, P);
    uint32_t bad = 0;
    if (is_int_dt<DT>() || DT == kF64 || screen_chunk<DT>(P, C, ex[k].th, cs[k], bad)) {
      if (!try_push(R, C, c * E, (uint32_t)k, q)) retry |= 1u << k;
    } else if (bad) {
      cs[k].cnt += __popc(bad);
      if (!((found >> k) & 1u)) {
        found |= 1u << k;
        atomicMin(&ex[k].first, c * E + first_of<DT>(bad));
      }
    }
  }
}

// Chunks that found the queue full (bit k of `retry`: candidate k): drain
// the queue and queue them again, re-read from the stage (`staged`) or from
// device memory; every round queues at least min(32, what is left).
// Warp-wide.
template <uint32_t DT>
__device__ __forceinline__ void requeue(const CmpParams &p, uint32_t ri, const uint4 *stage, uint32_t tbc,
                                     uint64_t c, bool staged, uint32_t retry, uint32_t warp, uint32_t K,
                                     const TolF *tol) {
  constexpr int E = Fmt<DT>::E;
  Queue *q = queue_of(warp);
  const CmpRegion r = p.regions[ri];
  while (__any_sync(0xFFFFFFFFu, retry)) {
    drain<DT>(warp, K, tol);
    while (retry) {
      const uint32_t k = __ffs(retry) - 1;
      const uint4 R = staged ? stage[0] : load_region_chunk(p, ri, r, -1, c);
      const uint4 C = staged ? stage[(size_t)(1 + k) * tbc] : load_region_chunk(p, ri, r, (int)k, c);
      if (!try_push(R, C, c * E, k, q)) break;
      retry &= retry - 1;
    }
    __syncwarp();
  }
}

// A warp's share of the tiles [t, t_end) of region ri, every candidate:
// for every tile, wait for its stage, check rows warp, warp + 15, ... of 32
// chunks, release the stage; then merge the region's statistics.  KMAX is
// the most candidates the instance checks.
template <uint32_t DT, int KMAX>
__device__ __noinline__ void run(const CmpParams &p, uint32_t ri, uint64_t t, uint64_t t_end,
                                 uint32_t warp, Cursor *cur) {
  const CmpRegion r = p.regions[ri];
  const uint32_t K = p.K, TB = p.tile_bytes, lane = threadIdx.x & 31;
  const uint32_t stage_bytes = (1 + K) * TB, tbc = TB >> 4;
  uint64_t *full = reinterpret_cast<uint64_t *>(cmp_smem);
  uint64_t *empty = full + kStages;
  Queue *q = queue_of(warp);
  ExactStats *ex = exact_of(warp);
  const TolF *tol = &p.tol[is_int_dt<DT>() ? 0 : DT];
  Bounds bnd;
  bnd.rlo = tol->rlo; bnd.alo = tol->alo; bnd.rhi = tol->rhi; bnd.ahi = tol->ahi;
  if (lane < K) {
    ExactStats &x = ex[lane];
    x.first = ~0ull; x.dabs = 0; x.drel = 0; x.cnt = 0; x.nonfin = 0; x.m32 = 0;
    x.th = rel_threshold<DT>(0ull);
  }
  __syncwarp();
  Cand cs[KMAX];
#pragma unroll
  for (int k = 0; k < KMAX; ++k) {
    cs[k].cnt = 0u; cs[k].cm = 0u;
  }
  uint32_t found = 0;                      // bit k: this lane's first mismatch for k is recorded
  const uint32_t nst = p.nstages;
  uint32_t s = cur->s, ph = cur->ph;
  for (; t < t_end; ++t) {
    if (!mbar_wait(smem_addr(&full[s]), ph, kWaitRounds)) { cur->ok = 0; break; }
    const TileInfo ti = tile_info(r, t, TB);
    const uint4 *stage = reinterpret_cast<const uint4 *>(cmp_smem + kStageOff + (size_t)s * stage_bytes);
    const uint64_t c0 = ti.off >> 4;
    const bool all_staged = ti.nsm == ti.nloc;
    // every bound below is the same for all lanes of the warp, so the
    // warp-wide __syncwarp and drain are reached by every lane
    for (uint32_t row = warp * 32; row < ti.nloc; row += 32 * kConsumerWarps) {
      const uint32_t i = row + lane;
      uint32_t retry = 0;                  // bit k: candidate k's chunk found the queue full
      if (i < ti.nloc) {
        if (all_staged)
          check_chunk<DT, KMAX, true>(p, ri, r, stage + i, tbc, c0 + i, K, bnd, q, ex, cs, found, retry);
        else
          check_chunk<DT, KMAX, false>(p, ri, r, stage + i, tbc, c0 + i, K, bnd, q, ex, cs, found, retry);
      }
      __syncwarp();
      if (__any_sync(0xFFFFFFFFu, retry))
        requeue<DT>(p, ri, stage + i, tbc, c0 + i, i < ti.nsm, retry, warp, K, tol);
      if (q->count >= kQueue / 2) drain<DT>(warp, K, tol);
    }
    // queued entries are copies, so the stage is released at once
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&empty[s]));
    if (++s == nst) { s = 0; ph ^= 1u; }
  }
  cur->s = s;
  cur->ph = ph;
  if (!cur->ok) return;
  __syncwarp();
  if (q->count) drain<DT>(warp, K, tol);
  // merge the region's statistics of every candidate into its global entry
#pragma unroll
  for (int k = 0; k < KMAX; ++k) {
    if (k >= (int)K) break;
    unsigned long long cnt = cs[k].cnt;
    float m = cm_value<DT>(cs[k].cm);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
      m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    }
    if (lane == 0) {
      const ExactStats &x = ex[k];
      StatsDev *st = p.stats + (size_t)k * p.nregions + ri;
      cnt += x.cnt;
      const unsigned long long ab =
          umax64(x.dabs, umax64(dbits((double)m), dbits((double)__uint_as_float(x.m32))));
      if (cnt) atomicAdd(&st->mismatches, cnt);
      if (x.nonfin) atomicAdd(&st->nonfinite, (unsigned long long)x.nonfin);
      if (x.first != ~0ull) atomicMin(&st->first, x.first);
      if (ab) atomicMax(&st->abs_bits, ab);
      if (x.drel) atomicMax(&st->rel_bits, x.drel);
    }
  }
  __syncwarp();
}

template <int KMAX>
__device__ __forceinline__ void run_dispatch(const CmpParams &p, uint32_t ri, uint64_t t, uint64_t t_end,
                                             uint32_t warp, Cursor *cur) {
#define ASMV_RUN(DT) run<DT, KMAX>(p, ri, t, t_end, warp, cur)
  switch (p.regions[ri].dtype) {
    case kF32: ASMV_RUN(kF32); break;
    case kBF16: ASMV_RUN(kBF16); break;
    case kF16: ASMV_RUN(kF16); break;
    case kF8: ASMV_RUN(kF8); break;
    case kI32: ASMV_RUN(kI32); break;
    case kI8: ASMV_RUN(kI8); break;
    case kF8E5M2: ASMV_RUN(kF8E5M2); break;
    case kF8E4FNUZ: ASMV_RUN(kF8E4FNUZ); break;
    case kF8E5FNUZ: ASMV_RUN(kF8E5FNUZ); break;
    case kF64: ASMV_RUN(kF64); break;
    case kI16: ASMV_RUN(kI16); break;
    case kI64: ASMV_RUN(kI64); break;
    default: ASMV_RUN(kU8); break;
  }
#undef ASMV_RUN
}

// Guard segments: one warp per segment; bad bytes and the first bad offset.
__device__ void guard_phase(const CmpParams &p, uint32_t warp, uint32_t nwarps) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t gw = (uint64_t)blockIdx.x * nwarps + warp;
  const uint64_t nw = (uint64_t)gridDim.x * nwarps;
  for (uint64_t s = gw; s < p.nsegs; s += nw) {
    const GuardSeg g = p.segs[s];
#if ASMV_DEBUG_BOUNDS
    if (!in_alloc(g.alloc, g.ptr, g.len, p.err)) continue;
#endif
    const uint8_t *src = reinterpret_cast<const uint8_t *>(g.ptr);
    unsigned long long bad = 0, first = ~0ull;
    for (uint32_t j = lane; j < g.len; j += 32) {
      if (__ldg(src + j) != g.canary) { ++bad; first = umin64(first, g.offset + j); }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      bad += __shfl_xor_sync(0xFFFFFFFFu, bad, o);
      first = umin64(first, __shfl_xor_sync(0xFFFFFFFFu, first, o));
    }
    if (lane == 0 && bad) {
      StatsDev *st = p.seg_stats + g.stats;
      if (g.kind == kSegRef) {
        atomicAdd(&st->ref_guard_bad, bad);
      } else {
        atomicAdd(&st->guard_bad, bad);
        atomicMin(&st->guard_first, first);
      }
    }
  }
}

// Warps 0..kConsumerWarps-1 check; the last warp feeds the stages.  Stage s
// holds the reference tile and the K candidate tiles (tile_bytes each);
// full[s] completes when its bulk copies land, empty[s] when every
// consumer warp has finished with it.
template <int KMAX>
__global__ void __launch_bounds__(kCmpThreads, 1) compare_kernel(const __grid_constant__ CmpParams p) {
  uint64_t *full = reinterpret_cast<uint64_t *>(cmp_smem);
  uint64_t *empty = full + kStages;
  const uint32_t nst = p.nstages;                            // pipeline depth, 2 to 4
  unsigned char *bufs = cmp_smem + kStageOff;
  const uint32_t K = p.K, TB = p.tile_bytes;
  const uint32_t stage_bytes = (1 + K) * TB;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x < kConsumerWarps) queue_of(threadIdx.x)->count = 0;
  if (threadIdx.x == 0) {
    for (uint32_t s = 0; s < nst; ++s) {
      mbar_init(smem_addr(&full[s]), 1);
      mbar_init(smem_addr(&empty[s]), kConsumerWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const uint64_t G = gridDim.x, b = blockIdx.x;
  const uint64_t t0 = p.ntiles * b / G, t1 = p.ntiles * (b + 1) / G;
  bool ok = true;
  if (warp == kConsumerWarps) {
    // producer
    if (lane == 0 && t0 < t1) {
      uint32_t ri = find_region(p.regions, p.nregions, t0);
      uint32_t u = 0, s = 0, ph = 0;       // tiles issued; stage and phase of the next
      for (uint64_t t = t0; t < t1 && ok; ++t, ++u) {
        while (p.regions[ri + 1].tile0 <= t) ++ri;
        if (u >= nst && !mbar_wait(smem_addr(&empty[s]), ph ^ 1u, p.wait_rounds)) {
          ok = false;
          break;
        }
        const CmpRegion r = p.regions[ri];
        const TileInfo ti = tile_info(r, t, TB);
        uint32_t nb = ti.nsm * 16u;
        const uint32_t fb = smem_addr(&full[s]);
#if ASMV_DEBUG_BOUNDS
        // a tile with any copy outside its allocation is not copied (its
        // stage is left as it was; the launch reports the error)
        bool inside = in_alloc(r.alloc, r.ref + ti.off, nb, p.err);
        for (uint32_t k = 0; k < K; ++k)
          inside = inside && in_alloc(p.cand_allocs[(size_t)k * p.nregions + ri],
                                      p.cands[(size_t)k * p.nregions + ri] + ti.off, nb, p.err);
        if (!inside) nb = 0;
#endif
        mbar_arrive_tx(fb, nb * (1 + K));
        if (nb) {
          const uint32_t dst = smem_addr(bufs + (size_t)s * stage_bytes);
          bulk_load(dst, r.ref + ti.off, nb, fb);
          for (uint32_t k = 0; k < K; ++k)
            bulk_load(dst + (1 + k) * TB, p.cands[(size_t)k * p.nregions + ri] + ti.off, nb, fb);
        }
        if (++s == nst) { s = 0; ph ^= 1u; }
      }
      if (!ok) atomicOr(p.err, 1u);
      // Let every copy issued land before the CTA can exit: consumers that
      // gave up on a wait leave their stages unread.  Each stage's latest
      // phase is the one awaited; in a run without errors these have
      // completed already.
      for (uint32_t v = (u >= nst ? u - nst : 0); v < u; ++v)
        mbar_wait(smem_addr(&full[v % nst]), (v / nst) & 1u, kWaitRounds);
    }
  } else if (t0 < t1) {
    // consumers: one call per run of tiles of the same region
    Cursor cur;
    cur.s = 0;
    cur.ph = 0;
    cur.ok = 1;
    uint32_t ri = find_region(p.regions, p.nregions, t0);
    uint64_t t = t0;
    while (t < t1 && cur.ok) {
      while (p.regions[ri + 1].tile0 <= t) ++ri;
      const uint64_t t_end = umin64(t1, p.regions[ri + 1].tile0);
      run_dispatch<KMAX>(p, ri, t, t_end, warp, &cur);
      t = t_end;
    }
    if (!cur.ok && lane == 0) atomicOr(p.err, 1u);
  }
  guard_phase(p, warp, kConsumerWarps + 1);
}

}  // namespace

size_t compare_smem_bytes(uint32_t K, uint32_t tile_bytes, uint32_t nstages) {
  return kStageOff + (size_t)nstages * (1 + K) * tile_bytes;
}

// Tiles of a launch group of up to K candidates: two rows of 32 chunks per
// checking warp for one candidate (15 KiB), one row otherwise (7.5 KiB),
// over as many stages as fit (compare_stages).  Whole rows per warp keep
// the warps of a stage equally loaded.
static_assert(kConsumerWarps == 15, "tile sizes are whole rows of the checking warps");
uint32_t compare_tile_bytes(uint32_t K) {
  return K <= 1 ? 15360u : 7680u;
}

// The deepest pipeline (4, 3, else 2 stages) within the 227 KiB of shared
// memory a CTA may take (the checking loop spills nothing, so L1 needs
// little of the SM's 256 KiB).
constexpr size_t kCmpSmemBudget = kMaxSmemPerCta;
uint32_t compare_stages(uint32_t K, uint32_t tile_bytes) {
  for (uint32_t n = 4; n > 2; --n)
    if (compare_smem_bytes(K, tile_bytes, n) <= kCmpSmemBudget) return n;
  return 2u;
}

namespace {
// The kernel instance of a launch: whether a warp checks one candidate or
// up to kMaxCands (the pipeline depth is a launch parameter).
using CmpKernel = void (*)(const CmpParams);
CmpKernel compare_instance(uint32_t K) {
  return K <= 1 ? compare_kernel<1> : compare_kernel<kMaxCands>;
}

// The dynamic shared memory limit of every instance, raised once per device
// to the most any launch uses (a per-launch call would add its host latency
// to every compare).  0: not yet, 1: done; a failure is returned every time.
constexpr int kMaxDevices = 64;
std::atomic<int> g_smem_set[kMaxDevices];
std::mutex g_smem_mutex;

int prepare_compare(size_t smem) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return (int)e;
  if (dev < 0 || dev >= kMaxDevices || smem > kMaxSmemPerCta) return (int)cudaErrorInvalidValue;
  if (g_smem_set[dev].load(std::memory_order_acquire)) return (int)cudaSuccess;
  std::lock_guard<std::mutex> lock(g_smem_mutex);
  if (g_smem_set[dev].load(std::memory_order_relaxed)) return (int)cudaSuccess;
  for (uint32_t k : {1u, 2u})
    if ((e = cudaFuncSetAttribute(compare_instance(k), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kMaxSmemPerCta)) != cudaSuccess)
      return (int)e;
  g_smem_set[dev].store(1, std::memory_order_release);
  return (int)cudaSuccess;
}
}  // namespace

int launch_compare(const CmpParams &p, int grid, void *stream) {
  if (p.nstages < 2 || p.nstages > (uint32_t)kStages) return (int)cudaErrorInvalidValue;
  const size_t smem = compare_smem_bytes(p.K, p.tile_bytes, p.nstages);
  const int rc = prepare_compare(smem);
  if (rc != (int)cudaSuccess) return rc;
  compare_instance(p.K)<<<grid, kCmpThreads, smem, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
