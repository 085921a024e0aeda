// eq64.cu -- the three sums behind the cosine of Eq. 1 (AsmEvo Sec. 3.2)
// for binary64 regions:
//   S_rc = sum r*c over pairs with both values finite,
//   S_rr = sum r*r over finite r,   S_cc = sum c*c over finite c,
// added exactly.
//
// A finite binary64 value is +-m 2^e with m < 2^53 and e >= -1074, read
// straight from its fields, so a product is +-M 2^E with M = m_r m_c below
// 2^106 (one 64x64 -> 128-bit product) and E >= -2148.  With
// t = E - kEq64Base, the product is the five 32-bit words of
// M << (t mod 32) placed at digits q .. q+4, q = t div 32.
//
// Reduction.  A lane handles two values (one 16-byte chunk) per step; the
// products of a warp that share q add their words with one redux per 16-bit
// half (64 halves sum below 2^22) and five lanes add the recombined words to
// the CTA's shared digits; a warp repeats this once per distinct q among its
// products, which is one or two for values of similar magnitude.  The CTA
// adds its shared digits to the region's global digits when it leaves the
// region.  Every element adds less than 2^32 to any one digit and a region
// holds at most 2^31 elements, so no digit, shared or global, leaves the
// int64 range; the host carries and rounds.
//
// Work split: a persistent grid over 16 KiB tiles of the reference payloads
// (2048 values); CTA b takes the contiguous tile range [T b / G,
// T (b+1) / G); within a tile, thread t reads the 16-byte chunks t, t + 256,
// ... of the reference and of each candidate in turn.
#include <cuda_runtime.h>
#include "device.cuh"
#include "eq64.h"

namespace asmv {
namespace {

constexpr uint32_t kFull = 0xFFFFFFFFu;
constexpr int kNloc = 1 + 2 * kMaxCands;
static_assert(kEq64TileBytes % (16 * kThreads) == 0, "eq64 tile split");

struct F64Parts {
  uint64_t m;           // significand (0 for zeros and non-finite values)
  int e;                // weight of its last bit, >= -1074
  uint32_t neg;         // sign bit
  bool fin;
};

__device__ __forceinline__ F64Parts split_f64(uint64_t x) {
  F64Parts v;
  const uint32_t be = (uint32_t)(x >> 52) & 0x7FFu;
  const uint64_t frac = x & ((1ull << 52) - 1ull);
  v.fin = be != 0x7FFu;
  v.m = v.fin ? (be ? (frac | (1ull << 52)) : frac) : 0ull;
  v.e = (int)(be ? be : 1u) - 1075;
  v.neg = (uint32_t)(x >> 63);
  return v;
}

// The five 32-bit words w of M << (t mod 32), M = a.m b.m, returning
// q = t div 32 for t = a.e + b.e - kEq64Base: the product is
// sum_k w[k] 2^(32 (q + k) + kEq64Base).
__device__ __forceinline__ uint32_t product_words(const F64Parts &a, const F64Parts &b,
                                                  uint32_t (&w)[5]) {
  const uint64_t lo = a.m * b.m, hi = __umul64hi(a.m, b.m);       // M = hi:lo < 2^106
  const uint32_t t = (uint32_t)(a.e + b.e - kEq64Base);            // >= 0
  const uint32_t s = t & 31u;
  const uint32_t m0 = (uint32_t)lo, m1 = (uint32_t)(lo >> 32);
  const uint32_t m2 = (uint32_t)hi, m3 = (uint32_t)(hi >> 32);
  w[0] = m0 << s;
  w[1] = __funnelshift_l(m0, m1, s);
  w[2] = __funnelshift_l(m1, m2, s);
  w[3] = __funnelshift_l(m2, m3, s);
  w[4] = __funnelshift_l(m3, 0u, s);
  return t >> 5;
}

// Add the products a0 b0 and a1 b1 (each with sign (-1)^neg when SIGNED,
// and only where ok0 / ok1 hold and both factors are non-zero) to the
// digits acc.  All 32 lanes of the warp call this together.  Each round
// takes the lowest digit index qq still pending in the warp: every lane
// adds the 16-bit halves of its products placed at qq (at most two, so a
// lane's half sums stay below 2^17 and a warp's below 2^22), one redux per
// half sums them over the warp, and lanes 0..4 add the five recombined
// words to digits qq .. qq+4.
template <bool SIGNED>
__device__ __forceinline__ void warp_add_pair(long long *acc, bool ok0, uint32_t neg0, const F64Parts &a0,
                                              const F64Parts &b0, bool ok1, uint32_t neg1,
                                              const F64Parts &a1, const F64Parts &b1) {
  const uint32_t lane = threadIdx.x & 31u;
  uint32_t w0[5] = {0u, 0u, 0u, 0u, 0u}, w1[5] = {0u, 0u, 0u, 0u, 0u};
  uint32_t q0 = 0xFFFFFFFFu, q1 = 0xFFFFFFFFu;                      // 0xFFFFFFFF: nothing pending
  if (ok0 && a0.m != 0ull && b0.m != 0ull) q0 = product_words(a0, b0, w0);
  if (ok1 && a1.m != 0ull && b1.m != 0ull) q1 = product_words(a1, b1, w1);
  while (__any_sync(kFull, (q0 & q1) != 0xFFFFFFFFu)) {
    const uint32_t qq = __reduce_min_sync(kFull, min(q0, q1));
    const bool m0 = q0 == qq, m1 = q1 == qq;
    if (m0) q0 = 0xFFFFFFFFu;
    if (m1) q1 = 0xFFFFFFFFu;
    long long word = 0;
#pragma unroll
    for (int k = 0; k < 5; ++k) {
      int lo = 0, hi = 0;
      if (m0) {
        const int l = (int)(w0[k] & 0xFFFFu), h = (int)(w0[k] >> 16);
        lo += (SIGNED && neg0) ? -l : l;
        hi += (SIGNED && neg0) ? -h : h;
      }
      if (m1) {
        const int l = (int)(w1[k] & 0xFFFFu), h = (int)(w1[k] >> 16);
        lo += (SIGNED && neg1) ? -l : l;
        hi += (SIGNED && neg1) ? -h : h;
      }
      const int slo = (int)__reduce_add_sync(kFull, (uint32_t)lo);
      const int shi = (int)__reduce_add_sync(kFull, (uint32_t)hi);
      if (lane == (uint32_t)k) word = (long long)slo + ((long long)shi << 16);
    }
    if (lane < 5u && word != 0)
      atomicAdd(reinterpret_cast<unsigned long long *>(acc + qq + lane), (unsigned long long)word);
  }
}

__device__ __forceinline__ uint4 load16(uint64_t addr, uint32_t n, uint32_t vec) {
  if (n == 0u) return make_uint4(0u, 0u, 0u, 0u);
  return (vec && n == 16u) ? ldg16(addr) : load_bytes(addr, n);
}

__device__ __forceinline__ uint64_t lo64(const uint4 &v) { return (uint64_t)v.y << 32 | v.x; }
__device__ __forceinline__ uint64_t hi64(const uint4 &v) { return (uint64_t)v.w << 32 | v.z; }

// Add the CTA's shared digits of `region` to its global digits; zero them.
__device__ void cta_flush64(const Eq64Params &p, uint32_t region, long long *sdig) {
  __syncthreads();
  const uint32_t nloc = 1u + 2u * p.K;
  for (uint32_t x = threadIdx.x; x < nloc * kEq64Digits; x += blockDim.x) {
    const long long v = sdig[x];
    if (v != 0) {
      const uint32_t ls = x / kEq64Digits, k = x % kEq64Digits;
      const uint32_t slot = ls == 0u ? 0u : ls + 2u * p.j0;
      long long *g = p.digits + ((size_t)region * p.nslots + slot) * kEq64Digits + k;
      atomicAdd(reinterpret_cast<unsigned long long *>(g), (unsigned long long)v);
      sdig[x] = 0;
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kThreads) eq64_kernel(Eq64Params p) {
  __shared__ long long sdig[kNloc * kEq64Digits];
  for (uint32_t x = threadIdx.x; x < (uint32_t)(kNloc * kEq64Digits); x += blockDim.x) sdig[x] = 0;
  __syncthreads();
  const uint64_t t0 = p.ntiles * blockIdx.x / gridDim.x;
  const uint64_t t1 = p.ntiles * (blockIdx.x + 1) / gridDim.x;
  uint32_t cur = 0xFFFFFFFFu;
  for (uint64_t t = t0; t < t1; ++t) {
    const uint32_t i = find_region(p.regions, p.nregions, t);
    const CmpRegion R = p.regions[i];
    if (i != cur) {
      if (cur != 0xFFFFFFFFu) cta_flush64(p, cur, sdig);
      cur = i;
    }
    const uint64_t a = (t - R.tile0) * kEq64TileBytes;
    const uint32_t nb = (uint32_t)umin64(kEq64TileBytes, R.bytes - a);
#pragma unroll 1
    for (uint32_t c0 = 0; 16u * c0 < nb; c0 += kThreads) {       // the same trip count for every thread
      const uint32_t off = 16u * (c0 + threadIdx.x);
      const uint32_t n = off < nb ? min(16u, nb - off) : 0u;    // bytes past the payload read as zero
      const uint4 rv = load16(R.ref + a + off, n, R.vec);
      const F64Parts r0 = split_f64(lo64(rv)), r1 = split_f64(hi64(rv));
      if (p.do_rr) warp_add_pair<false>(sdig, r0.fin, 0u, r0, r0, r1.fin, 0u, r1, r1);
#pragma unroll 1
      for (uint32_t j = 0; j < p.K; ++j) {
        const uint4 cv = load16(p.cands[(size_t)j * p.nregions + i] + a + off, n, R.vec);
        const F64Parts c0 = split_f64(lo64(cv)), c1 = split_f64(hi64(cv));
        long long *rc = sdig + (1 + 2 * j) * kEq64Digits, *cc = rc + kEq64Digits;
        warp_add_pair<true>(rc, r0.fin && c0.fin, r0.neg ^ c0.neg, r0, c0,
                            r1.fin && c1.fin, r1.neg ^ c1.neg, r1, c1);
        warp_add_pair<false>(cc, c0.fin, 0u, c0, c0, c1.fin, 0u, c1, c1);
      }
    }
  }
  if (cur != 0xFFFFFFFFu) cta_flush64(p, cur, sdig);
}

}  // namespace

int eq64_max_ctas_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, eq64_kernel, kThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return n > 0 ? n : 1;
}

int launch_eq64(const Eq64Params &p, int grid, void *stream) {
  eq64_kernel<<<grid, kThreads, 0, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
