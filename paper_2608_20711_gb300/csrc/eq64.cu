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
// Reduction.  The tile is passed over once for S_rr and once per candidate
// (S_rc and S_cc together; the reference comes from L1 after the first
// pass).  In a pass every lane keeps a window of six 64-bit digits
// qa .. qa+5 per sum, qa the lowest q among the warp's first products; a
// product starting at qa or qa + 1 is added to the window with one select
// and one 64-bit add per digit, and any other product (rare for values of
// one scale) goes to the CTA's shared digits with five atomics.  At the end
// of the pass the warp sums each window digit with three reduxes (two 16-bit
// pieces and the signed rest) and six lanes add the results to the shared
// digits.  The CTA adds its shared digits to the region's global digits when
// it leaves the region.  Every element adds less than 2^32 to any one digit
// and a region holds at most 2^31 elements, so no digit, shared or global,
// leaves the int64 range; the host carries and rounds.
//
// Work split: a persistent grid over 16 KiB tiles of the reference payloads
// (2048 values); CTA b takes the contiguous tile range [T b / G,
// T (b+1) / G); within a pass, thread t reads the 16-byte chunks t, t + 256,
// ... of the tile.
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

constexpr uint32_t kNoAnchor = 0xFFFFFFFFu;

// One product: its words, its digit index q (kNoAnchor when the product is
// zero or skipped) and its sign.
struct Prod {
  uint32_t w[5];
  uint32_t q;
  uint32_t neg;
};

__device__ __forceinline__ Prod make_prod(bool ok, uint32_t neg, const F64Parts &a, const F64Parts &b) {
  Prod P;
  P.neg = neg;
  P.q = kNoAnchor;
#pragma unroll
  for (int k = 0; k < 5; ++k) P.w[k] = 0u;
  if (ok && a.m != 0ull && b.m != 0ull) P.q = product_words(a, b, P.w);
  return P;
}

// A lane's window on one sum: digits qa .. qa+5, each a signed 64-bit sum
// of at most eight words below 2^32 (|d| < 2^35).  qa is the same in every
// lane.
struct Win {
  long long d[6];
  uint32_t qa;
};

__device__ __forceinline__ void win_reset(Win &W) {
#pragma unroll
  for (int j = 0; j < 6; ++j) W.d[j] = 0;
  W.qa = kNoAnchor;
}

// Anchor a window still without one at the lowest digit index among the
// warp's products p0, p1 (all 32 lanes call this together).
__device__ __forceinline__ void win_anchor(Win &W, const Prod &p0, const Prod &p1) {
  if (W.qa == kNoAnchor) W.qa = __reduce_min_sync(kFull, min(p0.q, p1.q));
}

// Add one product: into the window when it starts at digit qa or qa + 1,
// else (rare for values of one scale) straight to the shared digits acc.
template <bool SIGNED>
__device__ __forceinline__ void win_add(Win &W, const Prod &P, long long *acc) {
  if (P.q == kNoAnchor) return;
  const uint32_t o = P.q - W.qa;                  // wraps for q < qa: out of the window
  const bool neg = SIGNED && P.neg;
  if (o <= 1u) {
#pragma unroll
    for (int i = 0; i < 6; ++i) {
      const uint32_t a = i < 5 ? P.w[i] : 0u, b = i >= 1 ? P.w[i - 1] : 0u;
      const long long x = (long long)(o == 0u ? a : b);
      W.d[i] += neg ? -x : x;
    }
  } else {
#pragma unroll
    for (int k = 0; k < 5; ++k)
      if (P.w[k] != 0u)
        atomicAdd(reinterpret_cast<unsigned long long *>(acc + P.q + k),
                  neg ? (unsigned long long)(-(long long)P.w[k]) : (unsigned long long)P.w[k]);
  }
}

// Sum the window over the warp and add its six digits to acc; all 32
// lanes call this together.  A digit (|d| < 2^35) is cut into two 16-bit
// pieces and the signed rest, whose warp sums fit in 32 bits.
__device__ __forceinline__ void win_flush(Win &W, long long *acc) {
  if (W.qa == kNoAnchor) return;                  // warp-uniform
  const uint32_t lane = threadIdx.x & 31u;
  long long word = 0;
#pragma unroll
  for (int i = 0; i < 6; ++i) {
    const long long v = W.d[i];
    const uint32_t s0 = __reduce_add_sync(kFull, (uint32_t)v & 0xFFFFu);
    const uint32_t s1 = __reduce_add_sync(kFull, (uint32_t)(v >> 16) & 0xFFFFu);
    const int s2 = (int)__reduce_add_sync(kFull, (uint32_t)(int)(v >> 32));
    if (lane == (uint32_t)i)
      word = (long long)s0 + ((long long)s1 << 16) + ((long long)s2 << 32);
  }
  if (lane < 6u && word != 0)
    atomicAdd(reinterpret_cast<unsigned long long *>(acc + W.qa + lane), (unsigned long long)word);
}

// 16 bytes (n of them; the rest zero), through L1 when `cached`.
__device__ __forceinline__ uint4 load16(uint64_t addr, uint32_t n, uint32_t vec, bool cached) {
  if (n == 0u) return make_uint4(0u, 0u, 0u, 0u);
  if (!vec || n != 16u) return load_bytes(addr, n);
  return cached ? __ldg(reinterpret_cast<const uint4 *>(addr)) : ldg16(addr);
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
    // one pass over the tile per sum (S_rr), then per candidate (S_rc and
    // S_cc together); the reference tile comes from L1 after the first pass
    if (p.do_rr) {
      Win W;
      win_reset(W);
#pragma unroll 1
      for (uint32_t c0 = 0; 16u * c0 < nb; c0 += kThreads) {     // the same trip count for every thread
        const uint32_t off = 16u * (c0 + threadIdx.x);
        const uint32_t n = off < nb ? min(16u, nb - off) : 0u;  // bytes past the payload read as zero
        const uint4 rv = load16(R.ref + a + off, n, R.vec, true);
        const F64Parts r0 = split_f64(lo64(rv)), r1 = split_f64(hi64(rv));
        const Prod p0 = make_prod(r0.fin, 0u, r0, r0), p1 = make_prod(r1.fin, 0u, r1, r1);
        win_anchor(W, p0, p1);
        win_add<false>(W, p0, sdig);
        win_add<false>(W, p1, sdig);
      }
      win_flush(W, sdig);
    }
#pragma unroll 1
    for (uint32_t j = 0; j < p.K; ++j) {
      const uint64_t cb = p.cands[(size_t)j * p.nregions + i] + a;
      long long *rc = sdig + (1 + 2 * j) * kEq64Digits, *cc = rc + kEq64Digits;
      Win Wrc, Wcc;
      win_reset(Wrc);
      win_reset(Wcc);
#pragma unroll 1
      for (uint32_t c0 = 0; 16u * c0 < nb; c0 += kThreads) {
        const uint32_t off = 16u * (c0 + threadIdx.x);
        const uint32_t n = off < nb ? min(16u, nb - off) : 0u;
        const uint4 rv = load16(R.ref + a + off, n, R.vec, true);
        const uint4 cv = load16(cb + off, n, R.vec, false);
        const F64Parts r0 = split_f64(lo64(rv)), r1 = split_f64(hi64(rv));
        const F64Parts c0v = split_f64(lo64(cv)), c1v = split_f64(hi64(cv));
        const Prod x0 = make_prod(r0.fin && c0v.fin, r0.neg ^ c0v.neg, r0, c0v);
        const Prod x1 = make_prod(r1.fin && c1v.fin, r1.neg ^ c1v.neg, r1, c1v);
        win_anchor(Wrc, x0, x1);
        win_add<true>(Wrc, x0, rc);
        win_add<true>(Wrc, x1, rc);
        const Prod y0 = make_prod(c0v.fin, 0u, c0v, c0v), y1 = make_prod(c1v.fin, 0u, c1v, c1v);
        win_anchor(Wcc, y0, y1);
        win_add<false>(Wcc, y0, cc);
        win_add<false>(Wcc, y1, cc);
      }
      win_flush(Wrc, rc);
      win_flush(Wcc, cc);
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
