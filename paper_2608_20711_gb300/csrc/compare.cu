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
//  (4) max_rel: a thread keeps its exact maximum Rmax and T <= Rmax(1-2^-19)
//      in fp32.  An element can exceed Rmax only if as > T*|r| (the
//      relative error of as/|r| against d/|r| is below 2^-23), which
//      one fma decides exactly in sign; those elements get the exact
//      RN64(d/|r|).
// The maxima are order-independent (max of exact values), counts are sums
// and first_mismatch a minimum, so any grid gives bit-identical results.
//
// Work split: a CTA's 8 warps are divided among the K candidates (G = 8/K
// warps each).  For K > 1 the reference tile is staged once in shared
// memory and every candidate's warps read it from there, so device memory
// sees the reference once per tile.  Each lane keeps its statistics in
// registers and a warp merges them into the global entries with atomics
// when its CTA moves to the next region.
//
// Roofline: HBM reads of reference + candidate payloads (reference once per
// launch of up to 8 candidates); the screen costs ~10 fp32/integer
// operations per differing element, so dense small differences are also
// ALU-heavy.
#include <float.h>
#include <math_constants.h>
#include "device.cuh"

namespace asmv {
namespace {

struct Hot {
  uint32_t cnt;          // mismatches in the current region (per thread; < 2^32 for any HBM size)
  uint32_t nonfin;       // NaN/Inf-position mismatches
  unsigned long long first;   // lowest mismatching element index seen (~0 if none)
  float m32;             // exact max |c - r| over plain elements (see (3))
  float T;               // relative-error screen threshold
  double dabs;           // exact max |c - r| over exact-path elements
  double drel;           // exact max relative error
};

__device__ __forceinline__ float tfloor(double d) {
  return __fmul_rd(__double2float_rd(d), 0x1.ffffcp-1f);    // <= d (1 - 2^-19)
}

__device__ __forceinline__ void rel_update(Hot &h, double d, double r64) {
  const double ar = fabs(r64);
  const double rel = (ar != 0.0) ? __ddiv_rn(d, ar) : (d == 0.0 ? 0.0 : CUDART_INF);
  if (rel > h.drel) { h.drel = rel; h.T = tfloor(rel); }
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
  h.dabs = fmax(h.dabs, d);
  rel_update(h, d, r64);
  return d > bound ? 1u : 0u;
}

// Exact evaluation of one differing integer pair (always a mismatch).
__device__ __forceinline__ void exact_int(int64_t r, int64_t c, Hot &h) {
  const int64_t dd = c - r;
  const double d = (double)(dd < 0 ? -dd : dd);     // exact: |d| < 2^33
  h.dabs = fmax(h.dabs, d);
  rel_update(h, d, (double)r);
}

// A rare element that the screen decided (definite match or mismatch):
// exact maximum updates.
__device__ __forceinline__ void decided_update(float r, float c, Hot &h) {
  const double r64 = (double)r;
  const double d = fabs(__dsub_rn((double)c, r64));
  h.dabs = fmax(h.dabs, d);
  rel_update(h, d, r64);
}

// Masks of one chunk: bit j for element j.
struct Masks {
  uint32_t bad;    // definite mismatches from the screen
  uint32_t rare;   // elements needing the exact path or a maxima update
};

__device__ __forceinline__ void screen(float r, float c, int j, Hot &h, const TolF &t, Masks &m) {
  const float s = __fsub_rn(c, r);
  const float as = fabsf(s), ar = fabsf(r);
  const float lo = __fmaf_rn(t.rlo, ar, t.alo);
  const float hi = __fmaf_rn(t.rhi, ar, t.ahi);
  const bool ok = as < lo;
  const bool bad = as > hi;                       // Inf/NaN cases are rare below
  const bool plain = __fadd_rn(as, as) < ar;      // c - r exact (Sterbenz)
  const bool rare = !(ok | bad) | !plain | (__fmaf_rn(-h.T, ar, as) > 0.0f);
  if (plain) h.m32 = fmaxf(h.m32, as);
  m.bad |= (uint32_t)bad << j;
  m.rare |= (uint32_t)rare << j;
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

// Element j of a chunk decoded to fp32 (float dtypes; runtime j).
template <uint32_t DT>
__device__ __forceinline__ float elem_f32(const uint4 &v, int j) {
  if (DT == kF32) return __uint_as_float(word_of(v, j));
  if (DT == kBF16) return __uint_as_float(((word_of(v, j >> 1) >> (16 * (j & 1))) & 0xFFFFu) << 16);
  if (DT == kF16) return __half2float(__ushort_as_half((unsigned short)(word_of(v, j >> 1) >> (16 * (j & 1)))));
  const uint32_t b = (word_of(v, j >> 2) >> (8 * (j & 3))) & 0xFFu;
  return f8x2_to_f32(b).x;
}

template <uint32_t DT>
__device__ __forceinline__ int64_t elem_int(const uint4 &v, int j) {
  if (DT == kI32) return (int64_t)(int32_t)word_of(v, j);
  const uint32_t b = (word_of(v, j >> 2) >> (8 * (j & 3))) & 0xFFu;
  if (DT == kI8) return (int64_t)(int8_t)b;
  return (int64_t)b;
}

// Screen one differing 32-bit word of a float chunk.
template <uint32_t DT>
__device__ __forceinline__ void screen_word(uint32_t rw, uint32_t cw, int w, Hot &h,
                                            const TolF &t, Masks &m) {
  if (DT == kF32) {
    screen(__uint_as_float(rw), __uint_as_float(cw), w, h, t, m);
  } else if (DT == kBF16) {
    const uint32_t d = rw ^ cw;
    if (d & 0xFFFFu) screen(__uint_as_float(rw << 16), __uint_as_float(cw << 16), 2 * w, h, t, m);
    if (d >> 16) screen(__uint_as_float(rw & 0xFFFF0000u), __uint_as_float(cw & 0xFFFF0000u), 2 * w + 1, h, t, m);
  } else if (DT == kF16) {
    const uint32_t d = rw ^ cw;
    const float2 rf = f16x2_to_f32(rw), cf = f16x2_to_f32(cw);
    if (d & 0xFFFFu) screen(rf.x, cf.x, 2 * w, h, t, m);
    if (d >> 16) screen(rf.y, cf.y, 2 * w + 1, h, t, m);
  } else {                                      // fp8: four elements
    const uint32_t d = rw ^ cw;
    const float2 r0 = f8x2_to_f32(rw), c0 = f8x2_to_f32(cw);
    const float2 r1 = f8x2_to_f32(rw >> 16), c1 = f8x2_to_f32(cw >> 16);
    if (d & 0xFFu) screen(r0.x, c0.x, 4 * w, h, t, m);
    if (d & 0xFF00u) screen(r0.y, c0.y, 4 * w + 1, h, t, m);
    if (d & 0xFF0000u) screen(r1.x, c1.x, 4 * w + 2, h, t, m);
    if (d >> 24) screen(r1.y, c1.y, 4 * w + 3, h, t, m);
  }
}

// Rare elements are queued per warp in shared memory and evaluated exactly
// once per tile, lane-parallel, instead of diverging inside the screen.
constexpr uint32_t kQueue = 256;          // entries per warp

struct QEntry {
  uint32_t r, c;                          // fp32 bits (floats) or int32 values
  unsigned long long idx;                 // element index in the region
};

struct Queue {
  QEntry e[kQueue];
  uint32_t count;
};

// Exact evaluation of one queued element; returns the mismatch bit.
template <uint32_t DT>
__device__ __forceinline__ uint32_t exact_elem(uint32_t rb, uint32_t cb, Hot &h, const TolF &t) {
  if (DT == kI32 || DT == kI8 || DT == kU8) {
    exact_int((int64_t)(int32_t)rb, (int64_t)(int32_t)cb, h);
    return 1u;
  }
  const float r = __uint_as_float(rb), c = __uint_as_float(cb);
  const float as = fabsf(__fsub_rn(c, r)), ar = fabsf(r);
  const bool ok = as < __fmaf_rn(t.rlo, ar, t.alo);
  const bool definite_bad = (as > __fmaf_rn(t.rhi, ar, t.ahi)) & (as <= FLT_MAX);
  if (ok | definite_bad) {
    decided_update(r, c, h);
    return definite_bad ? 1u : 0u;
  }
  return exact_float(r, c, h, t);
}

template <uint32_t DT>
__device__ __forceinline__ void record(uint32_t bad, unsigned long long idx, Hot &h) {
  if (bad) { h.cnt += 1; h.first = umin64(h.first, idx); }
}

// Drain the warp's queue: lanes take entries in turn; then every lane
// adopts the warp's largest exact relative error (only the overall maximum
// matters, so a shared threshold is as valid as a per-lane one).
template <uint32_t DT>
__device__ __noinline__ Hot drain(Queue *q, Hot h, const TolF t) {
  __syncwarp();
  const uint32_t n = min(q->count, kQueue);
  for (uint32_t j = threadIdx.x & 31; j < n; j += 32) {
    const QEntry e = q->e[j];
    record<DT>(exact_elem<DT>(e.r, e.c, h, t), e.idx, h);
  }
  __syncwarp();
  if ((threadIdx.x & 31) == 0) q->count = 0;
  unsigned long long rb = (unsigned long long)__double_as_longlong(h.drel);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rb = umax64(rb, __shfl_xor_sync(0xFFFFFFFFu, rb, o));
  const double d = __longlong_as_double((long long)rb);
  if (d > h.drel) { h.drel = d; h.T = tfloor(d); }
  __syncwarp();
  return h;
}

template <uint32_t DT>
__device__ __forceinline__ uint32_t elem_bits(const uint4 &v, int j) {
  if (DT == kI32 || DT == kI8 || DT == kU8) return (uint32_t)(int32_t)elem_int<DT>(v, j);
  return __float_as_uint(elem_f32<DT>(v, j));
}

// Queue the flagged elements of one chunk; a full queue falls back to
// evaluating in this lane.
template <uint32_t DT>
__device__ __noinline__ Hot push_rare(const uint4 R, const uint4 C, uint32_t rare,
                                      unsigned long long e0, Queue *q, Hot h, const TolF t) {
  while (rare) {
    const int j = __ffs(rare) - 1;
    rare &= rare - 1;
    const uint32_t rb = elem_bits<DT>(R, j), cb = elem_bits<DT>(C, j);
    const uint32_t slot = atomicAdd(&q->count, 1u);
    if (slot < kQueue) {
      QEntry e;
      e.r = rb; e.c = cb; e.idx = e0 + (unsigned long long)j;
      q->e[slot] = e;
    } else {
      record<DT>(exact_elem<DT>(rb, cb, h, t), e0 + (unsigned long long)j, h);
    }
  }
  return h;
}

// One 16-byte chunk whose first element has index e0.
template <uint32_t DT>
__device__ __forceinline__ void chunk(const uint4 &R, const uint4 &C, uint64_t e0, Hot &h,
                                      const TolF &t, Queue *q) {
  if (R.x == C.x && R.y == C.y && R.z == C.z && R.w == C.w) return;
  uint32_t rare = 0;
  if (DT == kI32 || DT == kI8 || DT == kU8) {
    // integers: every differing element is a mismatch, evaluated exactly
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t d = word_of(R, w) ^ word_of(C, w);
      if (DT == kI32) rare |= (uint32_t)(d != 0) << w;
      else
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) rare |= (uint32_t)(((d >> (8 * qq)) & 0xFFu) != 0) << (4 * w + qq);
    }
  } else {
    Masks m = {0u, 0u};
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t rw = word_of(R, w), cw = word_of(C, w);
      if (rw != cw) screen_word<DT>(rw, cw, w, h, t, m);
    }
    const uint32_t bad = m.bad & ~m.rare;     // decided here; rare ones are decided exactly
    if (bad) {
      h.cnt += __popc(bad);
      h.first = umin64(h.first, e0 + (uint64_t)(__ffs(bad) - 1));
    }
    rare = m.rare;
  }
  if (rare) h = push_rare<DT>(R, C, rare, e0, q, h, t);
}

__device__ __forceinline__ void reset_hot(Hot &h) {
  h.cnt = 0; h.nonfin = 0; h.first = ~0ull;
  h.m32 = 0.0f; h.T = 0.0f; h.dabs = 0.0; h.drel = 0.0;
}

// Merge a warp's statistics for region `ri`, candidate k into the global
// entry with order-independent atomics; then reset.
__device__ __forceinline__ void flush(Hot &h, const CmpParams &p, uint32_t k, uint32_t ri) {
  unsigned long long cnt = h.cnt, nonfin = h.nonfin;
  unsigned long long first = h.first;
  const double a = fmax(h.dabs, (double)h.m32);
  unsigned long long ab = (unsigned long long)__double_as_longlong(a);
  unsigned long long rb = (unsigned long long)__double_as_longlong(h.drel);
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
// kWaitRounds tries of up to kWaitHintNs each, the wait reports failure.
constexpr uint32_t kWaitRounds = 20000;
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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (uint32_t i = 0; i < kWaitRounds; ++i) {
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

// A warp's share of one tile for its candidate: chunks part*32 + lane +
// j*32*W; staged chunks come from shared memory, the rest from global.
template <uint32_t DT>
__device__ __noinline__ Hot tile(const CmpRegion r, uint64_t cbase, TileInfo ti, const uint4 *sref,
                                 const uint4 *scand, uint32_t part, uint32_t W, Hot h, const TolF t,
                                 Queue *q) {
  constexpr int E = Fmt<DT>::E;
  constexpr int U = 2;
  const uint64_t c0 = ti.off >> 4;
  const uint64_t full = r.bytes >> 4;
  const uint32_t stride = 32 * W;
  uint32_t i0 = part * 32 + (threadIdx.x & 31);
  for (; i0 + (U - 1) * stride < ti.nsm; i0 += U * stride) {
    uint4 R[U], C[U];
#pragma unroll
    for (int u = 0; u < U; ++u) { R[u] = sref[i0 + u * stride]; C[u] = scand[i0 + u * stride]; }
#pragma unroll
    for (int u = 0; u < U; ++u) chunk<DT>(R[u], C[u], (c0 + i0 + u * stride) * E, h, t, q);
    __syncwarp();
    if (q->count >= kQueue / 2) h = drain<DT>(q, h, t);
  }
  for (uint32_t i = i0; i < ti.nloc; i += stride) {
    uint4 R, C;
    if (i < ti.nsm) { R = sref[i]; C = scand[i]; }
    else {
      R = load_chunk(r.ref, c0 + i, full, r.bytes, false);
      C = load_chunk(cbase, c0 + i, full, r.bytes, false);
    }
    chunk<DT>(R, C, (c0 + i) * E, h, t, q);
  }
  __syncwarp();
  if (q->count) h = drain<DT>(q, h, t);
  return h;
}

__device__ __forceinline__ Hot tile_dispatch(const CmpParams &p, const CmpRegion &r, uint64_t cbase,
                                             TileInfo ti, const uint4 *sref, const uint4 *scand,
                                             uint32_t part, uint32_t W, Hot h, Queue *q) {
  switch (r.dtype) {
    case kF32: return tile<kF32>(r, cbase, ti, sref, scand, part, W, h, p.tol[kF32], q);
    case kBF16: return tile<kBF16>(r, cbase, ti, sref, scand, part, W, h, p.tol[kBF16], q);
    case kF16: return tile<kF16>(r, cbase, ti, sref, scand, part, W, h, p.tol[kF16], q);
    case kF8: return tile<kF8>(r, cbase, ti, sref, scand, part, W, h, p.tol[kF8], q);
    case kI32: return tile<kI32>(r, cbase, ti, sref, scand, part, W, h, p.tol[0], q);
    case kI8: return tile<kI8>(r, cbase, ti, sref, scand, part, W, h, p.tol[0], q);
    default: return tile<kU8>(r, cbase, ti, sref, scand, part, W, h, p.tol[0], q);
  }
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
__global__ void __launch_bounds__(kCmpThreads, 1) compare_kernel(const CmpParams p) {
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem);
  uint64_t *empty = full + kStages;
  Queue *queues = reinterpret_cast<Queue *>(smem + 128);
  unsigned char *bufs = smem + 128 + kConsumerWarps * sizeof(Queue);
  const uint32_t K = p.K, TB = p.tile_bytes;
  const uint32_t stage_bytes = (1 + K) * TB;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x < kConsumerWarps) queues[threadIdx.x].count = 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
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
        const uint32_t s = u % kStages;
        if (u >= (uint32_t)kStages && !mbar_wait(smem_addr(&empty[s]), ((u / kStages) & 1u) ^ 1u)) {
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
      if (!ok) {
        atomicOr(p.err, 1u);
        // let copies already issued land before the CTA exits
        for (uint32_t v = (u >= (uint32_t)kStages ? u - kStages : 0); v < u; ++v)
          mbar_wait(smem_addr(&full[v % kStages]), (v / kStages) & 1u);
      }
    }
  } else if (t0 < t1) {
    // consumers
    const uint32_t W = kConsumerWarps / K;                  // warps per candidate
    const bool active = warp < W * K;
    const uint32_t k = warp % K, part = warp / K;
    Hot h;
    reset_hot(h);
    uint32_t ri = find_region(p.regions, p.nregions, t0);
    uint32_t u = 0;
    for (uint64_t t = t0; t < t1; ++t, ++u) {
      if (p.regions[ri + 1].tile0 <= t) {
        if (active) flush(h, p, k, ri);
        while (p.regions[ri + 1].tile0 <= t) ++ri;
      }
      const uint32_t s = u % kStages;
      if (!mbar_wait(smem_addr(&full[s]), (u / kStages) & 1u)) {
        ok = false;
        break;
      }
      if (active) {
        const CmpRegion r = p.regions[ri];
        const TileInfo ti = tile_info(r, t, TB);
        const uint4 *sref = reinterpret_cast<const uint4 *>(bufs + (size_t)s * stage_bytes);
        const uint4 *scand = reinterpret_cast<const uint4 *>(bufs + (size_t)s * stage_bytes +
                                                              (size_t)(1 + k) * TB);
        h = tile_dispatch(p, r, p.cands[(size_t)k * p.nregions + ri], ti, sref, scand, part, W, h,
                          &queues[warp]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_addr(&empty[s]));
    }
    if (!ok) {
      if (lane == 0) atomicOr(p.err, 1u);
    } else if (active) {
      flush(h, p, k, ri);
    }
  }
  guard_phase(p, warp, kConsumerWarps + 1);
}

}  // namespace

size_t compare_smem_bytes(uint32_t K, uint32_t tile_bytes) {
  return 128 + kConsumerWarps * sizeof(Queue) + (size_t)kStages * (1 + K) * tile_bytes;
}

uint32_t compare_tile_bytes(uint32_t K) {
  // stage = (1 + K) tiles; keep a stage near 32-36 KiB
  if (K <= 1) return 16384;
  if (K == 2) return 12288;
  if (K == 3) return 8192;
  return 4096;
}

int launch_compare(const CmpParams &p, int grid, void *stream) {
  const size_t smem = compare_smem_bytes(p.K, p.tile_bytes);
  cudaError_t e = cudaFuncSetAttribute(compare_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return (int)e;
  compare_kernel<<<grid, kCmpThreads, smem, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
