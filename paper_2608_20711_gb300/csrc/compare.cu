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
// The maxima are order-independent (max of exact values), counts are sums
// and first_mismatch a minimum, so any grid gives bit-identical results.
//
// Work split: one CTA of 17 warps per SM.  The last warp streams each tile
// of the reference and of the K <= 8 candidates into shared memory with
// bulk copies (two or four stages, as fit, mbarrier-completed; the kernel
// is instantiated per depth); the 16 checking warps are
// divided among the candidates, so device memory sees the reference once
// per tile.  Chunks the screen cannot settle are queued per warp and
// drained lane-parallel.  Each lane keeps its statistics in registers and
// a warp merges them into the global entries with atomics when its CTA
// moves to the next region.
//
// Roofline: HBM reads of reference + candidate payloads (reference once per
// launch of up to 8 candidates); the screen costs about 10 fp32 operations
// per differing element (its three thresholds on packed f32x2 for the 16-
// and 8-bit formats), so dense small differences are also ALU-heavy.
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

// Chunks the screen cannot settle are queued per warp in shared memory and
// re-examined element by element once per tile, lane-parallel, instead of
// diverging inside the screen.
// 32 entries per warp: with 64 the 4096-region snapshot ran 4 % slower
// (the queues' shared memory comes out of L1), with 16 no faster.
constexpr uint32_t kQueue = 32;           // chunk entries per warp

struct QEntry {
  uint4 R, C;                             // the raw 16-byte chunks
  unsigned long long e0;                  // element index of the chunk's first element
};

struct Queue {
  QEntry e[kQueue];
  uint32_t count;
};

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

// Drain the warp's queue: lanes take chunks in turn; then every lane
// adopts the warp's largest exact relative error (only the overall maximum
// matters, so a shared threshold is as valid as a per-lane one).
template <uint32_t DT>
__device__ __noinline__ Hot drain(Queue *q, Hot h, const TolF t) {
  __syncwarp();
  const uint32_t n = min(q->count, kQueue);
  for (uint32_t j = threadIdx.x & 31; j < n; j += 32) settle_chunk<DT>(q->e[j], h, t);
  __syncwarp();
  if ((threadIdx.x & 31) == 0) q->count = 0;
  unsigned long long rb = h.drel;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rb = umax64(rb, __shfl_xor_sync(0xFFFFFFFFu, rb, o));
  if (rb > h.drel) { h.drel = rb; h.T = tfloor(__longlong_as_double((long long)rb)); }
  __syncwarp();
  return h;
}

// A chunk that found the queue full is settled in its own lane.
template <uint32_t DT>
__device__ __noinline__ Hot settle_overflow(const QEntry e, Hot h, const TolF t) {
  settle_chunk<DT>(e, h, t);
  return h;
}

// Queue one chunk.
template <uint32_t DT>
__device__ __forceinline__ void push_chunk(const uint4 &R, const uint4 &C, unsigned long long e0,
                                           Queue *q, Hot &h, const TolF &t) {
  const uint32_t slot = atomicAdd(&q->count, 1u);
  QEntry e;
  e.R = R; e.C = C; e.e0 = e0;
  if (slot < kQueue) q->e[slot] = e;
  else h = settle_overflow<DT>(e, h, t);
}

// Screen of one element whose difference s is exact when it matters.
// Returns the definite-mismatch bit; sets `rare` when the element needs the
// exact path; accumulates the chunk's largest |s|.
__device__ __forceinline__ uint32_t screen(float r, float s, float Tp, const TolF &t, bool &rare,
                                          float &cm) {
  const float as = fabsf(s), ar = fabsf(r);
  const float lo = __fmaf_rn(t.rlo, ar, t.alo);
  const float hi = __fmaf_rn(t.rhi, ar, t.ahi);
  const float y = __fmul_rd(Tp, ar);
  const bool ok = as < lo;
  const bool bad = as > hi;
  rare |= (!(ok | bad)) | (as > y);
  cm = fmaxf(cm, as);
  return bad ? 1u : 0u;
}

__device__ __forceinline__ float2 ffma2_rd(float2 a, float2 b, float2 c) {
  unsigned long long d;
  asm("fma.rm.f32x2 %0, %1, %2, %3;"
      : "=l"(d)
      : "l"(*reinterpret_cast<unsigned long long *>(&a)), "l"(*reinterpret_cast<unsigned long long *>(&b)),
        "l"(*reinterpret_cast<unsigned long long *>(&c)));
  return *reinterpret_cast<float2 *>(&d);
}

// screen() of the two elements of a pair, their three bounds formed by
// packed fp32 multiply-adds (each lane rounded exactly as the scalar one).
// Returns the definite-mismatch bits (element 0 in bit 0).
__device__ __forceinline__ uint32_t screen2(float2 r, float2 s, float Tp, const TolF &t, bool &rare,
                                           float &cm) {
  const float2 ar = make_float2(fabsf(r.x), fabsf(r.y));
  const float2 lo = __ffma2_rn(make_float2(t.rlo, t.rlo), ar, make_float2(t.alo, t.alo));
  const float2 hi = __ffma2_rn(make_float2(t.rhi, t.rhi), ar, make_float2(t.ahi, t.ahi));
  const float2 y = ffma2_rd(make_float2(Tp, Tp), ar, make_float2(0.0f, 0.0f));   // RD32(Tp*|r|)
  const float a0 = fabsf(s.x), a1 = fabsf(s.y);
  const bool ok0 = a0 < lo.x, bad0 = a0 > hi.x, ok1 = a1 < lo.y, bad1 = a1 > hi.y;
  rare |= (!(ok0 | bad0)) | (a0 > y.x) | (!(ok1 | bad1)) | (a1 > y.y);
  cm = fmaxf(cm, fmaxf(a0, a1));
  return (bad0 ? 1u : 0u) | (bad1 ? 2u : 0u);
}

// One 16-byte chunk whose first element has index e0.
//  - Equal chunks cost one comparison.
//  - 16- and 8-bit floats subtract in their own format (one packed
//    instruction per pair): the result is exact whenever |c-r| < |r|/2
//    (Sterbenz), and every other element fails |s| < Tp*|r| <= |r|/2.
//  - A packed s*0 accumulation turns any NaN or Inf into a NaN sentinel.
//  - A chunk with any element the screen cannot settle is queued whole.
template <uint32_t DT>
__device__ __forceinline__ void chunk(const uint4 &R, const uint4 &C, uint64_t e0, Hot &h,
                                      const TolF &t, Queue *q) {
  if (R.x == C.x && R.y == C.y && R.z == C.z && R.w == C.w) return;
  if (is_int_dt<DT>() || DT == kF64) {
    push_chunk<DT>(R, C, e0, q, h, t);          // integer and binary64 differences are evaluated exactly
    return;
  }
  const float Tp = fminf(h.T, ASMV_HALF_LESS);
  bool rare = false;
  float cm = 0.0f;
  uint32_t bad = 0;
  if (DT == kF32) {
    float acc = 0.0f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float r = __uint_as_float(word_of(R, w)), c = __uint_as_float(word_of(C, w));
      const float s = __fsub_rn(c, r);
      acc = __fmaf_rn(s, 0.0f, acc);
      bad |= screen(r, s, Tp, t, rare, cm) << w;
    }
    rare |= !(acc == 0.0f);
  } else if (DT == kBF16) {
    __nv_bfloat162 acc = __float2bfloat162_rn(0.0f);
    const __nv_bfloat162 zero = acc;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t rw = word_of(R, w), cw = word_of(C, w);
      const __nv_bfloat162 s2 = __hsub2(*reinterpret_cast<const __nv_bfloat162 *>(&cw),
                                        *reinterpret_cast<const __nv_bfloat162 *>(&rw));
      acc = __hfma2(s2, zero, acc);
      const uint32_t sw = *reinterpret_cast<const uint32_t *>(&s2);
      bad |= screen2(make_float2(__uint_as_float(rw << 16), __uint_as_float(rw & 0xFFFF0000u)),
                     make_float2(__uint_as_float(sw << 16), __uint_as_float(sw & 0xFFFF0000u)), Tp, t,
                     rare, cm) << (2 * w);
    }
    const uint32_t aw = *reinterpret_cast<const uint32_t *>(&acc);
    rare |= (aw & 0x7FFF7FFFu) != 0u;
  } else {
    // fp16, and fp8 widened to fp16 (exact)
    __half2 acc = __float2half2_rn(0.0f);
    const __half2 zero = acc;
    constexpr int WORDS = (DT == kF16) ? 4 : 8;        // half2 pairs per chunk
#pragma unroll
    for (int w = 0; w < WORDS; ++w) {
      uint32_t rw, cw;
      if (DT == kF16) { rw = word_of(R, w); cw = word_of(C, w); }
      else {
        rw = fp8x2_to_half2_bits<DT>(word_of(R, w >> 1) >> (16 * (w & 1)));
        cw = fp8x2_to_half2_bits<DT>(word_of(C, w >> 1) >> (16 * (w & 1)));
      }
      const __half2 s2 = __hsub2(*reinterpret_cast<const __half2 *>(&cw),
                                 *reinterpret_cast<const __half2 *>(&rw));
      acc = __hfma2(s2, zero, acc);
      bad |= screen2(f16x2_to_f32(rw), __half22float2(s2), Tp, t, rare, cm) << (2 * w);
    }
    const uint32_t aw = *reinterpret_cast<const uint32_t *>(&acc);
    rare |= (aw & 0x7FFF7FFFu) != 0u;
  }
  if (rare) {
    push_chunk<DT>(R, C, e0, q, h, t);
    return;
  }
  h.m32 = fmaxf(h.m32, cm);
  if (bad) {
    h.cnt += __popc(bad);
    h.first = umin64(h.first, e0 + (uint64_t)(__ffs(bad) - 1));
  }
}

__device__ __forceinline__ void reset_hot(Hot &h) {
  h.cnt = 0; h.nonfin = 0; h.first = ~0ull;
  h.m32 = 0.0f; h.T = 0.0f; h.dabs = 0; h.drel = 0;
}

// Merge a warp's statistics for region `ri`, candidate k into the global
// entry with order-independent atomics; then reset.
__device__ __forceinline__ void flush(Hot &h, const CmpParams &p, uint32_t k, uint32_t ri) {
  unsigned long long cnt = h.cnt, nonfin = h.nonfin;
  unsigned long long first = h.first;
  unsigned long long ab = umax64(h.dabs, dbits((double)h.m32));
  unsigned long long rb = h.drel;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
    nonfin += __shfl_xor_sync(0xFFFFFFFFu, nonfin, o);
    first = umin64(first, __shfl_xor_sync(0xFFFFFFFFu, first, o));
    ab = umax64(ab, __shfl_xor_sync(0xFFFFFFFFu, ab, o));
    rb = umax64(rb, __shfl_xor_sync(0xFFFFFFFFu, rb, o));
  }
  if ((threadIdx.x & 31) == 0) {
    StatsDev *st = p.stats + (size_t)k * p.nregions + ri;
    if (cnt) atomicAdd(&st->mismatches, cnt);
    if (nonfin) atomicAdd(&st->nonfinite, nonfin);
    if (first != ~0ull) atomicMin(&st->first, first);
    if (ab) atomicMax(&st->abs_bits, ab);
    if (rb) atomicMax(&st->rel_bits, rb);
  }
  reset_hot(h);
}

__device__ __forceinline__ uint4 load_chunk(uint64_t base, uint64_t c, uint64_t full, uint64_t bytes,
                                            bool vec) {
  if (vec && c < full) return ldg16(base + 16 * c);
  return load_bytes(base + 16 * c, (uint32_t)umin64(16, bytes - 16 * c));
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

// Pipeline position shared by a consumer warp's calls.
struct Cursor {
  uint32_t u;          // stage uses consumed so far
  uint32_t ok;         // every wait succeeded
};

// The last rows of a short tile: lanes past its end are predicated off and
// chunks beyond the staged part come from global memory.
template <uint32_t DT>
__device__ __noinline__ Hot tail_rows(const CmpRegion r, uint64_t cbase, const TileInfo ti,
                                      const uint4 *sref, const uint4 *scand, uint32_t row,
                                      uint32_t stride, Hot h, const TolF tol, Queue *q) {
  constexpr int E = Fmt<DT>::E;
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t c0 = ti.off >> 4, full_chunks = r.bytes >> 4;
  for (; row < ti.nloc; row += stride) {
    const uint32_t i = row + lane;
    if (i < ti.nloc) {
      uint4 R, C;
      if (i < ti.nsm) { R = sref[i]; C = scand[i]; }
      else {
        R = load_chunk(r.ref, c0 + i, full_chunks, r.bytes, false);
        C = load_chunk(cbase, c0 + i, full_chunks, r.bytes, false);
      }
      chunk<DT>(R, C, (c0 + i) * E, h, tol, q);
    }
    __syncwarp();
    if (q->count >= kQueue / 2) h = drain<DT>(q, h, tol);
  }
  return h;
}

// A warp's share of the tiles [t, t_end) of one region for its candidate:
// for every tile, wait for its stage, check chunks part*32 + lane + j*32*W
// (staged chunks from shared memory, the rest from global), release the
// stage.  One call per run of tiles keeps the per-tile cost to the waits.
// NST is the launch's pipeline depth (stage u % NST, phase (u / NST) & 1).
template <uint32_t DT, uint32_t NST>
__device__ __noinline__ Hot run(const CmpRegion r, uint64_t cbase, uint64_t t, uint64_t t_end,
                                const unsigned char *bufs, uint32_t stage_bytes, uint32_t cand_off,
                                uint64_t *full, uint64_t *empty, uint32_t tile_bytes, uint32_t part,
                                uint32_t W, bool active, Hot h, const TolF tol, Queue *q,
                                Cursor *cur) {
  constexpr int E = Fmt<DT>::E;
  constexpr int U = 2;
  const uint32_t stride = 32 * W;
  const uint32_t lane = threadIdx.x & 31;
  uint32_t u = cur->u;
  for (; t < t_end; ++t, ++u) {
    const uint32_t s = u % NST;
    if (!mbar_wait(smem_addr(&full[s]), (u / NST) & 1u, kWaitRounds)) { cur->ok = 0; break; }
    if (active) {
      const TileInfo ti = tile_info(r, t, tile_bytes);
      const uint4 *sref = reinterpret_cast<const uint4 *>(bufs + (size_t)s * stage_bytes);
      const uint4 *scand = reinterpret_cast<const uint4 *>(bufs + (size_t)s * stage_bytes + cand_off);
      const uint64_t c0 = ti.off >> 4;
      // Rows of U*32*W chunks; every loop bound below is the same for all
      // lanes of the warp, so the warp-wide __syncwarp and drain are reached
      // by every lane.  Whole rows come from shared memory; the last rows of
      // a short tile go through the predicated tail.
      uint32_t row = part * 32;
      for (; row + (U - 1) * stride + 31 < ti.nsm; row += U * stride) {
        uint4 R[U], C[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          R[k] = sref[row + lane + k * stride];
          C[k] = scand[row + lane + k * stride];
        }
#pragma unroll
        for (int k = 0; k < U; ++k) chunk<DT>(R[k], C[k], (c0 + row + lane + k * stride) * E, h, tol, q);
        __syncwarp();
        if (q->count >= kQueue / 2) h = drain<DT>(q, h, tol);
      }
      if (row < ti.nloc) h = tail_rows<DT>(r, cbase, ti, sref, scand, row, stride, h, tol, q);
      __syncwarp();
      if (q->count) h = drain<DT>(q, h, tol);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&empty[s]));
  }
  cur->u = u;
  return h;
}

template <uint32_t NST>
__device__ __forceinline__ Hot run_dispatch(const CmpParams &p, const CmpRegion &r, uint64_t cbase,
                                            uint64_t t, uint64_t t_end, const unsigned char *bufs,
                                            uint32_t stage_bytes, uint32_t cand_off, uint64_t *full,
                                            uint64_t *empty, uint32_t part, uint32_t W, bool active,
                                            Hot h, Queue *q, Cursor *cur) {
  const uint32_t TB = p.tile_bytes;
#define ASMV_RUN(DT, TOL) run<DT, NST>(r, cbase, t, t_end, bufs, stage_bytes, cand_off, full, empty, TB, \
                                  part, W, active, h, TOL, q, cur)
  switch (r.dtype) {
    case kF32: return ASMV_RUN(kF32, p.tol[kF32]);
    case kBF16: return ASMV_RUN(kBF16, p.tol[kBF16]);
    case kF16: return ASMV_RUN(kF16, p.tol[kF16]);
    case kF8: return ASMV_RUN(kF8, p.tol[kF8]);
    case kI32: return ASMV_RUN(kI32, p.tol[0]);
    case kI8: return ASMV_RUN(kI8, p.tol[0]);
    case kF8E5M2: return ASMV_RUN(kF8E5M2, p.tol[kF8E5M2]);
    case kF8E4FNUZ: return ASMV_RUN(kF8E4FNUZ, p.tol[kF8E4FNUZ]);
    case kF8E5FNUZ: return ASMV_RUN(kF8E5FNUZ, p.tol[kF8E5FNUZ]);
    case kF64: return ASMV_RUN(kF64, p.tol[kF64]);
    case kI16: return ASMV_RUN(kI16, p.tol[0]);
    case kI64: return ASMV_RUN(kI64, p.tol[0]);
    default: return ASMV_RUN(kU8, p.tol[0]);
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
template <uint32_t NST>
__global__ void __launch_bounds__(kCmpThreads, 1) compare_kernel(const CmpParams p) {
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem);
  uint64_t *empty = full + kStages;
  constexpr uint32_t nst = NST;                              // pipeline depth, 2 or 4
  Queue *queues = reinterpret_cast<Queue *>(smem + 128);
  unsigned char *bufs = smem + 128 + kConsumerWarps * sizeof(Queue);
  const uint32_t K = p.K, TB = p.tile_bytes;
  const uint32_t stage_bytes = (1 + K) * TB;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x < kConsumerWarps) queues[threadIdx.x].count = 0;
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
      uint32_t u = 0;
      for (uint64_t t = t0; t < t1 && ok; ++t, ++u) {
        while (p.regions[ri + 1].tile0 <= t) ++ri;
        const uint32_t s = u % nst;
        if (u >= nst && !mbar_wait(smem_addr(&empty[s]), ((u / nst) & 1u) ^ 1u, p.wait_rounds)) {
          ok = false;
          break;
        }
        const CmpRegion r = p.regions[ri];
        const TileInfo ti = tile_info(r, t, TB);
        const uint32_t nb = ti.nsm * 16u;
        const uint32_t fb = smem_addr(&full[s]);
        mbar_arrive_tx(fb, nb * (1 + K));
        if (nb) {
          const uint32_t dst = smem_addr(bufs + (size_t)s * stage_bytes);
          bulk_load(dst, r.ref + ti.off, nb, fb);
          for (uint32_t k = 0; k < K; ++k)
            bulk_load(dst + (1 + k) * TB, p.cands[(size_t)k * p.nregions + ri] + ti.off, nb, fb);
        }
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
    const uint32_t W = kConsumerWarps / K;                  // warps per candidate
    const bool active = warp < W * K;
    const uint32_t k = warp % K, part = warp / K;
    Hot h;
    reset_hot(h);
    Cursor cur;
    cur.u = 0;
    cur.ok = 1;
    uint32_t ri = find_region(p.regions, p.nregions, t0);
    uint64_t t = t0;
    while (t < t1 && cur.ok) {
      while (p.regions[ri + 1].tile0 <= t) ++ri;
      const uint64_t t_end = umin64(t1, p.regions[ri + 1].tile0);
      const CmpRegion r = p.regions[ri];
      const uint64_t cbase = p.cands[(size_t)k * p.nregions + ri];
      h = run_dispatch<NST>(p, r, cbase, t, t_end, bufs, stage_bytes, (1 + k) * TB, full, empty,
                            part, W, active, h, &queues[warp], &cur);
      t = t_end;
      if (active && cur.ok) flush(h, p, k, ri);
    }
    if (!cur.ok && lane == 0) atomicOr(p.err, 1u);
  }
  guard_phase(p, warp, kConsumerWarps + 1);
}

}  // namespace

size_t compare_smem_bytes(uint32_t K, uint32_t tile_bytes, uint32_t nstages) {
  return 128 + kConsumerWarps * sizeof(Queue) + (size_t)nstages * (1 + K) * tile_bytes;
}

// Tiles of a launch group of up to K candidates: 16 KiB for one candidate,
// 8 KiB otherwise, over as many stages as fit (compare_stages).  Larger
// tiles mean fewer per-tile waits and less bookkeeping per chunk.  On a
// 1 GiB fp16 reference (GB/s of reference + candidates read):
//   K            2     3     4     5     6     7     8
//   before    3051  2911  2582  2265  2654  2768  3051   (4 KiB tiles from K = 4, 4 stages)
//   now       3137  2960  3302  3053  3118  3194  3530   (stages: 4 4 4 3 2 2 2)
// and with one candidate, 4 stages of 16 KiB beat 2 stages by a fifth.
// Tiles of whole warp rows (no tail rows) were measured too: better at
// K = 2, worse at K = 3 and 5.
uint32_t compare_tile_bytes(uint32_t K) {
  return K <= 1 ? 16384u : 8192u;
}

// The deepest pipeline (4, 3, else 2 stages) within kCmpSmemBudget of shared
// memory.  The budget stays below the 227 KiB a CTA may take: the rest of
// the SM's 256 KiB is L1, which holds the checking warps' spilled registers
// (about 100 bytes a thread), and deeper pipelines that squeezed it were
// slower (K = 5 at 4 stages and 217 KiB: 2348 GB/s against 3089 at 2 stages).
constexpr size_t kCmpSmemBudget = 192 * 1024;
uint32_t compare_stages(uint32_t K, uint32_t tile_bytes) {
  for (uint32_t n = 4; n > 2; --n)
    if (compare_smem_bytes(K, tile_bytes, n) <= kCmpSmemBudget) return n;
  return 2u;
}

// The dynamic shared memory limit of both instances, raised once per device
// to the most any launch uses (a per-launch call would add its host latency
// to every compare).  0: not yet, 1: done; a failure is returned every time.
namespace {
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
  if ((e = cudaFuncSetAttribute(compare_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kMaxSmemPerCta)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(compare_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kMaxSmemPerCta)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(compare_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kMaxSmemPerCta)) != cudaSuccess)
    return (int)e;
  g_smem_set[dev].store(1, std::memory_order_release);
  return (int)cudaSuccess;
}
}  // namespace

int launch_compare(const CmpParams &p, int grid, void *stream) {
  const size_t smem = compare_smem_bytes(p.K, p.tile_bytes, p.nstages);
  const int rc = prepare_compare(smem);
  if (rc != (int)cudaSuccess) return rc;
  auto kern = p.nstages == 2 ? compare_kernel<2> : p.nstages == 3 ? compare_kernel<3> : compare_kernel<4>;
  kern<<<grid, kCmpThreads, smem, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
