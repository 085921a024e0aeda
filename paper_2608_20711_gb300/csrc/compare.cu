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
//  (3) max_abs: RN is monotone, so for as_j < as_k the exact D_j < D_k.
//      Per thread we keep m32 = max as and, over the elements tied at m32,
//      the largest TwoSum residual me (D = m32 + me exactly); the exact
//      maximum is RN64(m32 + me).  Only elements with as >= m32 are touched.
//  (4) max_rel: a thread keeps its exact maximum Rmax and T <= Rmax(1-2^-19)
//      in fp32.  An element can exceed Rmax only if as >= T*|r| (the
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
  uint32_t found;        // first mismatch recorded
  unsigned long long first;
  float m32, me, T;
  double dabs;           // exact max |c - r| over fp64-path elements
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

// A rare element that the screen decided (definite match or mismatch) but
// that may raise max_abs or max_rel.
__device__ __forceinline__ void decided_update(float r, float c, Hot &h) {
  const float s = __fsub_rn(c, r);
  const float as = fabsf(s), ar = fabsf(r);
  if (as >= h.m32) {
    // TwoSum of c and -r: s + e == c - r exactly
    const float bb = __fsub_rn(s, c);
    const float e = __fadd_rn(__fsub_rn(c, __fsub_rn(s, bb)), __fsub_rn(-r, bb));
    const float ep = (s >= 0.0f) ? e : -e;                // |c - r| == as + ep
    if (as > h.m32) { h.m32 = as; h.me = ep; }
    else h.me = fmaxf(h.me, ep);
  }
  if (__fmaf_rn(-h.T, ar, as) >= 0.0f) {
    const double d = fabs(__dsub_rn((double)c, (double)r));
    rel_update(h, d, (double)r);
  }
}

// Masks of one chunk: bit j for element j.
struct Masks {
  uint32_t bad;    // definite mismatches from the screen
  uint32_t rare;   // elements needing the exact path or a maxima update
};

__device__ __forceinline__ void screen(float r, float c, int j, const Hot &h, const TolF &t,
                                       Masks &m) {
  const float s = __fsub_rn(c, r);
  const float as = fabsf(s), ar = fabsf(r);
  const float lo = __fmaf_rn(t.rlo, ar, t.alo);
  const float hi = __fmaf_rn(t.rhi, ar, t.ahi);
  const bool ok = as < lo;
  const bool bad = (as > hi) & (as <= FLT_MAX);
  const bool rare = !(ok | bad) | (as >= h.m32) | (__fmaf_rn(-h.T, ar, as) >= 0.0f);
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
__device__ __forceinline__ void screen_word(uint32_t rw, uint32_t cw, int w, const Hot &h,
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

struct RareOut {
  Hot h;
  uint32_t bad;    // mismatches found on the exact path
};

// Every element of one chunk flagged by the screen (or, for integers,
// every differing element).  Out of line: it is rare, and the fp64
// arithmetic would otherwise inflate the hot loop's register budget.
template <uint32_t DT>
__device__ __noinline__ RareOut rare_chunk(const uint4 R, const uint4 C, uint32_t rare, Hot h,
                                           const TolF t) {
  uint32_t bad = 0;
  while (rare) {
    const int j = __ffs(rare) - 1;
    rare &= rare - 1;
    if (DT == kI32 || DT == kI8 || DT == kU8) {
      exact_int(elem_int<DT>(R, j), elem_int<DT>(C, j), h);
      bad |= 1u << j;
    } else {
      const float r = elem_f32<DT>(R, j), c = elem_f32<DT>(C, j);
      const float as = fabsf(__fsub_rn(c, r)), ar = fabsf(r);
      const bool ok = as < __fmaf_rn(t.rlo, ar, t.alo);
      const bool definite_bad = (as > __fmaf_rn(t.rhi, ar, t.ahi)) & (as <= FLT_MAX);
      if (ok | definite_bad) decided_update(r, c, h);
      else bad |= exact_float(r, c, h, t) << j;
    }
  }
  RareOut o;
  o.h = h;
  o.bad = bad;
  return o;
}

// One 16-byte chunk whose first element has index e0.
template <uint32_t DT>
__device__ __forceinline__ void chunk(const uint4 &R, const uint4 &C, uint64_t e0, Hot &h,
                                      const TolF &t) {
  if (R.x == C.x && R.y == C.y && R.z == C.z && R.w == C.w) return;
  uint32_t allbad = 0, rare = 0;
  if (DT == kI32 || DT == kI8 || DT == kU8) {
    // integers: every differing element is a mismatch, handled exactly
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t d = word_of(R, w) ^ word_of(C, w);
      if (DT == kI32) rare |= (uint32_t)(d != 0) << w;
      else
#pragma unroll
        for (int q = 0; q < 4; ++q) rare |= (uint32_t)(((d >> (8 * q)) & 0xFFu) != 0) << (4 * w + q);
    }
  } else {
    Masks m = {0u, 0u};
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t rw = word_of(R, w), cw = word_of(C, w);
      if (rw != cw) screen_word<DT>(rw, cw, w, h, t, m);
    }
    allbad = m.bad;
    rare = m.rare;
  }
  if (rare) {
    const RareOut o = rare_chunk<DT>(R, C, rare, h, t);
    h = o.h;
    allbad |= o.bad;
  }
  if (allbad) {
    h.cnt += __popc(allbad);
    if (!h.found) { h.found = 1; h.first = e0 + (uint64_t)(__ffs(allbad) - 1); }
  }
}

__device__ __forceinline__ void reset_hot(Hot &h) {
  h.cnt = 0; h.nonfin = 0; h.found = 0; h.first = ~0ull;
  h.m32 = 0.0f; h.me = 0.0f; h.T = 0.0f; h.dabs = 0.0; h.drel = 0.0;
}

// Merge a warp's statistics for region `ri`, candidate k into the global
// entry with order-independent atomics; then reset.
__device__ __forceinline__ void flush(Hot &h, const CmpParams &p, uint32_t k, uint32_t ri) {
  unsigned long long cnt = h.cnt, nonfin = h.nonfin;
  unsigned long long first = h.found ? h.first : ~0ull;
  const double a = fmax(h.dabs, __dadd_rn((double)h.m32, (double)h.me));
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

// A warp's share of one tile for its candidate: chunks part*32 + lane +
// j*32*G of the tile, U at a time.
template <uint32_t DT, bool STAGE>
__device__ __noinline__ Hot tile(const CmpRegion r, uint64_t cbase, uint64_t tile_in_region,
                                 uint32_t part, uint32_t G, Hot h, const TolF t,
                                 const uint4 *ref_tile) {
  constexpr int E = Fmt<DT>::E;
  constexpr int U = 4;
  const uint64_t c0 = tile_in_region * kTileChunks;
  const uint64_t nchunks = (r.bytes + 15) >> 4, full = r.bytes >> 4;
  const uint32_t nloc = (uint32_t)umin64(kTileChunks, nchunks - c0);
  const bool vec = r.vec != 0;
  const uint32_t stride = 32 * G;
  for (uint32_t i0 = part * 32 + (threadIdx.x & 31); i0 < nloc; i0 += U * stride) {
    uint4 R[U], C[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t i = i0 + u * stride;
      if (i < nloc) {
        C[u] = load_chunk(cbase, c0 + i, full, r.bytes, vec);
        R[u] = STAGE ? ref_tile[i] : load_chunk(r.ref, c0 + i, full, r.bytes, vec);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t i = i0 + u * stride;
      if (i < nloc) chunk<DT>(R[u], C[u], (c0 + i) * E, h, t);
    }
  }
  return h;
}

template <bool STAGE>
__device__ __forceinline__ void tile_dispatch(const CmpParams &p, const CmpRegion &r, uint64_t cbase,
                                              uint64_t tr, uint32_t part, uint32_t G, Hot &h,
                                              const uint4 *ref_tile) {
  switch (r.dtype) {
    case kF32: h = tile<kF32, STAGE>(r, cbase, tr, part, G, h, p.tol[kF32], ref_tile); break;
    case kBF16: h = tile<kBF16, STAGE>(r, cbase, tr, part, G, h, p.tol[kBF16], ref_tile); break;
    case kF16: h = tile<kF16, STAGE>(r, cbase, tr, part, G, h, p.tol[kF16], ref_tile); break;
    case kF8: h = tile<kF8, STAGE>(r, cbase, tr, part, G, h, p.tol[kF8], ref_tile); break;
    case kI32: h = tile<kI32, STAGE>(r, cbase, tr, part, G, h, p.tol[0], ref_tile); break;
    case kI8: h = tile<kI8, STAGE>(r, cbase, tr, part, G, h, p.tol[0], ref_tile); break;
    default: h = tile<kU8, STAGE>(r, cbase, tr, part, G, h, p.tol[0], ref_tile); break;
  }
}

// Guard segments: one warp per segment; bad bytes and the first bad offset.
__device__ void guard_phase(const CmpParams &p) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = (uint64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
  const uint64_t nw = (uint64_t)gridDim.x * kWarps;
  for (uint64_t s = warp; s < p.nsegs; s += nw) {
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

// STAGE (K > 1): the reference tile goes through shared memory once.
template <bool STAGE>
__global__ void __launch_bounds__(kThreads, 2) compare_kernel(const CmpParams p) {
  __shared__ __align__(16) uint4 ref_tile[STAGE ? kTileChunks : 1];
  const uint64_t G = gridDim.x, b = blockIdx.x;
  const uint64_t t0 = p.ntiles * b / G, t1 = p.ntiles * (b + 1) / G;
  const uint32_t warp = threadIdx.x >> 5;
  const uint32_t K = p.K, W = kWarps / K;              // warps per candidate
  const bool active = warp < W * K;
  const uint32_t k = warp % K, part = warp / K;
  if (t0 < t1) {
    Hot h;
    reset_hot(h);
    uint32_t ri = find_region(p.regions, p.nregions, t0);
    for (uint64_t t = t0; t < t1; ++t) {
      if (p.regions[ri + 1].tile0 <= t) {
        if (active) flush(h, p, k, ri);
        while (p.regions[ri + 1].tile0 <= t) ++ri;
      }
      const CmpRegion r = p.regions[ri];
      if (STAGE) {
        const uint64_t c0 = (t - r.tile0) * kTileChunks;
        const uint64_t nchunks = (r.bytes + 15) >> 4, full = r.bytes >> 4;
        const uint32_t nloc = (uint32_t)umin64(kTileChunks, nchunks - c0);
        for (uint32_t i = threadIdx.x; i < nloc; i += kThreads)
          ref_tile[i] = load_chunk(r.ref, c0 + i, full, r.bytes, r.vec != 0);
        __syncthreads();
      }
      if (active)
        tile_dispatch<STAGE>(p, r, p.cands[(size_t)k * p.nregions + ri], t - r.tile0, part, W, h,
                             ref_tile);
      if (STAGE) __syncthreads();
    }
    if (active) flush(h, p, k, ri);
  }
  guard_phase(p);
}

}  // namespace

int compare_max_ctas_per_sm(int K) {
  int n = 0;
  const cudaError_t e = (K > 1)
      ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, compare_kernel<true>, kThreads, 0)
      : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, compare_kernel<false>, kThreads, 0);
  if (e != cudaSuccess || n < 1) return 1;
  return n;
}

int launch_compare(const CmpParams &p, int grid, void *stream) {
  if (p.K > 1) compare_kernel<true><<<grid, kThreads, 0, (cudaStream_t)stream>>>(p);
  else compare_kernel<false><<<grid, kThreads, 0, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
