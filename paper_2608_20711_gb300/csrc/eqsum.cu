// eqsum.cu -- the three sums behind the cosine of Eq. 1 (AsmEvo Sec. 3.2):
//   S_rc = sum r*c over pairs with both values finite,
//   S_rr = sum r*r over finite r,   S_cc = sum c*c over finite c,
// for every float region of a reference and K candidates, added exactly.
//
// Exactness.  Every sum is kept as integers at a fixed binary point and
// integer additions are exact and commute, so the sums do not depend on the
// order of the elements or on the grid.
//   fp16 and fp8: a finite value is an integer multiple of one quantum, so
//   each product is an integer at 2^-48 (fp16) or 2^-18 (fp8), formed with
//   32x32+64-bit multiply-adds of signed limbs (eq_tile_fixed).
//   bf16 and fp32: a decoded element is +-m 2^e with an integer significand
//   m (< 2^8, 2^24) and e the weight of its last bit; a product is +-P 2^s,
//   P = m_r m_c, s = e_r + e_c.  Each thread adds its products at a binary
//   point 2^L into NACC signed 64-bit accumulators 32 bits apart
//   (accumulator q weighs 2^(L + 32q)):
//     P 2^s = (P << (t & 31)) 2^(L + 32 (t >> 5)),  t = s - L,
//   (fp32 products are split into two 24-bit pieces first).  A product
//   outside the window [L, L + 32 NACC) goes straight to the region's
//   global digits with 64-bit atomics; values between about 2^-24 and 2^24
//   stay in the window.
//
// Reduction.  Every tile, each warp cuts its lanes' accumulated sums into
// 16-bit pieces whose warp sums fit in 32 bits, sums each piece over the
// warp with one redux, and adds the recombined digits to the CTA's shared
// digits; the CTA adds those to the region's global digits when it leaves
// the region.  Three CTAs of 256 threads share an SM (80 registers).  Global digit k of a sum weighs 2^(32k + base), base
// = eq_digit_base(dtype); the host rounds the digits to fp64.
//
// Work split: like the compare, a persistent grid over 16 KiB tiles of the
// reference payloads.  Within a tile, warp w takes a contiguous run of at
// most 128 chunks of 16 bytes (four per lane).  The K candidates are read
// one after another; the reference tile is re-read through L1 for each, so
// it comes from memory once per tile.
#include <cuda_runtime.h>
#include "device.cuh"
#include "plan.h"

namespace asmv {
namespace {

constexpr int kWin = 5;                 // shared digits per sum: NACC + 1 <= 5
constexpr int kMaxRounds = 4;           // chunks per lane per tile (16 KiB / 8 warps / 32 lanes / 16 B)
static_assert(kTileBytes == (uint64_t)kMaxRounds * 16 * 32 * kWarps, "eq tile split");

template <int DT> struct Fmt;
// kL: binary point of the window; kDig: index of the global digit at 2^kL
template <> struct Fmt<kF32>  { static constexpr int kBytes = 4, kNacc = 4, kL = -94, kDig = 7; };
template <> struct Fmt<kBF16> { static constexpr int kBytes = 2, kNacc = 3, kL = -62, kDig = 7; };
template <> struct Fmt<kF16>  { static constexpr int kL = -48, kDig = 2; };   // fixed point, below
template <> struct Fmt<kF8>   { static constexpr int kL = -18, kDig = 2; };

static_assert(Fmt<kF32>::kL - 32 * Fmt<kF32>::kDig == eq_digit_base(kF32), "fp32 digits");
static_assert(Fmt<kBF16>::kL - 32 * Fmt<kBF16>::kDig == eq_digit_base(kBF16), "bf16 digits");
static_assert(Fmt<kF16>::kL - 32 * Fmt<kF16>::kDig == eq_digit_base(kF16), "fp16 digits");
static_assert(Fmt<kF8>::kL - 32 * Fmt<kF8>::kDig == eq_digit_base(kF8), "fp8 digits");

struct Elem {
  uint32_t m;      // significand (integer)
  int e;           // weight of its last bit: |x| = m 2^e
  bool neg, fin;
};

// Element k of a 16-byte chunk.
template <int DT>
__device__ __forceinline__ Elem decode(const uint4 &v, int k) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  Elem x;
  if (DT == kF32) {
    const uint32_t b = w[k];
    const uint32_t E = (b >> 23) & 255u, f = b & 0x7FFFFFu;
    x.fin = E != 255u;
    x.m = E ? (f | 0x800000u) : f;
    x.e = (int)max(E, 1u) - 150;
    x.neg = (b >> 31) != 0;
  } else if (DT == kBF16 || DT == kF16) {
    const uint32_t b = (w[k >> 1] >> (16 * (k & 1))) & 0xFFFFu;
    if (DT == kBF16) {
      const uint32_t E = (b >> 7) & 255u, f = b & 127u;
      x.fin = E != 255u;
      x.m = E ? (f | 128u) : f;
      x.e = (int)max(E, 1u) - 134;
    } else {
      const uint32_t E = (b >> 10) & 31u, f = b & 1023u;
      x.fin = E != 31u;
      x.m = E ? (f | 1024u) : f;
      x.e = (int)max(E, 1u) - 25;
    }
    x.neg = (b >> 15) != 0;
  } else {
    const uint32_t b = (w[k >> 2] >> (8 * (k & 3))) & 0xFFu;
    const uint32_t E = (b >> 3) & 15u, f = b & 7u;
    x.fin = (b & 0x7Fu) != 0x7Fu;
    x.m = E ? (f | 8u) : f;
    x.e = (int)max(E, 1u) - 10;
    x.neg = (b >> 7) != 0;
  }
  return x;
}

// One product outside the window: three digit atomics.  pos = s - base >= 0.
__device__ __noinline__ void rare_add(long long *dig, unsigned long long P, int pos, bool neg) {
  const int q = pos >> 5, b = pos & 31;
  const unsigned long long lo = P << b;
  const unsigned long long hi = b ? (P >> (64 - b)) : 0ull;
  const unsigned long long d[3] = {lo & 0xFFFFFFFFull, lo >> 32, hi};
#pragma unroll
  for (int k = 0; k < 3; ++k)
    if (d[k]) atomicAdd(reinterpret_cast<unsigned long long *>(dig + q + k),
                        neg ? (unsigned long long)(-(long long)d[k]) : d[k]);
}

template <int N>
__device__ __forceinline__ void add_piece(long long (&a)[N], int t, unsigned long long piece, bool neg) {
  long long v = (long long)(piece << (t & 31));
  v = neg ? -v : v;
  const int q = t >> 5;
#pragma unroll
  for (int k = 0; k < N; ++k)
    if (q == k) a[k] += v;
}

// acc += x*y (exact); `dig` is the sum's global digits (for the rare path).
template <int DT>
__device__ __forceinline__ void add_product(long long (&a)[Fmt<DT>::kNacc], const Elem &x,
                                            const Elem &y, long long *dig) {
  using F = Fmt<DT>;
  const unsigned long long P = (unsigned long long)x.m * y.m;
  if (P == 0ull) return;
  const int t = x.e + y.e - F::kL;
  const bool neg = x.neg != y.neg;
  if (DT == kF32) {
    if ((unsigned)t < (unsigned)(32 * F::kNacc - 24)) {
      add_piece(a, t, P & 0xFFFFFFull, neg);
      add_piece(a, t + 24, P >> 24, neg);
    } else {
      rare_add(dig, P, t + 32 * F::kDig, neg);
    }
  } else {
    if ((unsigned)t < (unsigned)(32 * F::kNacc)) add_piece(a, t, P, neg);
    else rare_add(dig, P, t + 32 * F::kDig, neg);
  }
}

// Warp sum of one lane value |v| < 2^32 added to one shared digit: v is
// cut into its low 16 bits and the signed rest (|rest| < 2^16), whose warp
// sums fit in 32 bits and take one redux each.
__device__ __forceinline__ void warp_add_digit(long long v, long long *sd) {
  const uint32_t a = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)v & 0xFFFFu);
  const int b = __reduce_add_sync(0xFFFFFFFFu, (int)(v >> 16));
  if ((threadIdx.x & 31) == 0) {
    const long long s = (long long)a + (long long)b * 65536ll;
    if (s != 0) atomicAdd(reinterpret_cast<unsigned long long *>(sd), (unsigned long long)s);
  }
}

// Carry the lane's accumulators into N+1 digits, sum them over the warp and
// add them to the CTA's shared digits of one sum.  All 32 lanes call this.
template <int N>
__device__ __forceinline__ void warp_flush(long long (&a)[N], long long *sdig) {
  long long d[N + 1];
  long long carry = 0;
#pragma unroll
  for (int k = 0; k < N; ++k) {
    const long long x = a[k] + carry;          // |a| < 2^62, |carry| < 2^31
    d[k] = x & 0xFFFFFFFFll;
    carry = x >> 32;
    a[k] = 0;
  }
  d[N] = carry;
#pragma unroll
  for (int k = 0; k <= N; ++k) warp_add_digit(d[k], sdig + k);
}

__device__ __forceinline__ long long *global_digits(const EqParams &p, uint32_t region, uint32_t slot) {
  return p.digits + ((size_t)region * p.nslots + slot) * kEqDigits;
}

// Global slot of local slot `ls` (0 = S_rr, 1 + 2j = S_rc of candidate j,
// 2 + 2j = S_cc of candidate j).
__device__ __forceinline__ uint32_t global_slot(const EqParams &p, uint32_t ls) {
  return ls == 0 ? 0u : ls + 2u * p.j0;
}

__device__ __forceinline__ uint4 load_chunk(uint64_t addr, uint32_t bytes, bool vec, bool cached) {
  if (!vec || bytes != 16u) return load_bytes(addr, bytes);
  return cached ? __ldg(reinterpret_cast<const uint4 *>(addr)) : ldg16(addr);
}

template <int DT>
__device__ __noinline__ void eq_tile(const EqParams &p, const CmpRegion &R, uint32_t region,
                                     uint64_t a, uint32_t nb, long long *sdig) {
  using F = Fmt<DT>;
  constexpr int kPer = 16 / F::kBytes;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t nchunks = (nb + 15u) >> 4;
  const uint32_t per_warp = (nchunks + kWarps - 1) / kWarps;
  const uint32_t c0 = warp * per_warp;
  const uint32_t c1 = min(c0 + per_warp, nchunks);
  const uint32_t rounds = (per_warp + 31u) >> 5;     // the same for every warp
  if (p.do_rr) {
    long long acc[F::kNacc];
#pragma unroll
    for (int k = 0; k < F::kNacc; ++k) acc[k] = 0;
    long long *dig = global_digits(p, region, 0);
#pragma unroll 1
    for (uint32_t r = 0; r < rounds; ++r) {
      const uint32_t c = c0 + 32u * r + lane;
      uint4 rv = make_uint4(0u, 0u, 0u, 0u);
      if (c < c1) rv = load_chunk(R.ref + a + 16ull * c, min(16u, nb - 16u * c), R.vec, true);
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const Elem x = decode<DT>(rv, k);
        if (x.fin) add_product<DT>(acc, x, x, dig);
      }
    }
    warp_flush(acc, sdig);
  }
  for (uint32_t j = 0; j < p.K; ++j) {
    const uint64_t cbase = p.cands[(size_t)j * p.nregions + region] + a;
    long long rc[F::kNacc], cc[F::kNacc];
#pragma unroll
    for (int k = 0; k < F::kNacc; ++k) { rc[k] = 0; cc[k] = 0; }
    long long *dig_rc = global_digits(p, region, global_slot(p, 1 + 2 * j));
    long long *dig_cc = global_digits(p, region, global_slot(p, 2 + 2 * j));
#pragma unroll 1
    for (uint32_t r = 0; r < rounds; ++r) {
      const uint32_t c = c0 + 32u * r + lane;
      uint4 rv = make_uint4(0u, 0u, 0u, 0u), cv = rv;
      if (c < c1) {
        const uint32_t bytes = min(16u, nb - 16u * c);
        rv = load_chunk(R.ref + a + 16ull * c, bytes, R.vec, true);   // L1 hit after j = 0
        cv = load_chunk(cbase + 16ull * c, bytes, R.vec, false);
      }
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const Elem x = decode<DT>(rv, k);
        const Elem y = decode<DT>(cv, k);
        if (y.fin) {
          add_product<DT>(cc, y, y, dig_cc);
          if (x.fin) add_product<DT>(rc, x, y, dig_rc);
        }
      }
    }
    warp_flush(rc, sdig + (1 + 2 * j) * kWin);
    warp_flush(cc, sdig + (2 + 2 * j) * kWin);
  }
}

// ---------------------------------------------------------------------
// fp16 and fp8: every finite value is an integer multiple of one quantum,
// x = X 2^-24 with |X| < 2^40 (fp16) or x = X 2^-9 with |X| < 2^18 (fp8
// e4m3), so the sums are sums of integer products at one binary point
// (2^-48, 2^-18).  fp16: X = hi 2^20 + lo with signed limbs (|hi| <= 2^20,
// |lo| <= 2^19), and
//   x*y 2^48 = (hi hi') 2^40 + (hi lo' + lo hi') 2^20 + lo lo',
// each partial product at most 2^40 and added with one 32x32+64
// multiply-add; fp8: X X' < 2^36 with one multiply-add.  A non-finite value
// gets X = 0 and drops out of every sum it would enter.
// ---------------------------------------------------------------------
struct Limbs { int hi, lo; };
struct Acc3 { long long s2, s1, s0; };        // s2 2^40 + s1 2^20 + s0

// round(v) for |v| < 2^22: adding 1.5 2^23 leaves the integer in the low
// mantissa bits (one fp32 rounding, to nearest even).
constexpr float kMagic = 12582912.0f;
constexpr int kMagicBits = 0x4B400000;

// fp16 bits -> X = x 2^24 as hi 2^20 + lo, exactly, on the fp32 pipe:
// hi = round(16 x) (|hi| <= 2^20), lo = (x - hi/16) 2^24 (an integer, since
// x is a multiple of 2^-24 and |x - hi/16| <= 2^-5, exact in fp32).
__device__ __forceinline__ Limbs fix_f16(uint32_t b) {
  b = ((b & 0x7C00u) == 0x7C00u) ? 0u : b;                      // NaN, Inf -> 0
  const float x = __half2float(__ushort_as_half((unsigned short)b));
  const float hf = __fmaf_rn(x, 16.0f, kMagic);
  const float l = __fmaf_rn(__fsub_rn(hf, kMagic), -0.0625f, x);
  return {__float_as_int(hf) - kMagicBits,
          __float_as_int(__fmaf_rn(l, 16777216.0f, kMagic)) - kMagicBits};
}

// The limbs of fix_f16, each plus kMagicBits, for the two fp16 values of
// a word (low half first) known to be finite, on packed fp32 (each lane
// rounds exactly as fix_f16's scalar steps).  For a candidate only the
// differences of its limbs from the reference's are used, so the offsets
// cancel and need no subtraction.
__device__ __forceinline__ void fix_f16x2_biased(uint32_t w, Limbs &a, Limbs &b) {
  const float2 x = __half22float2(*reinterpret_cast<const __half2 *>(&w));
  const float2 hf = __ffma2_rn(x, make_float2(16.0f, 16.0f), make_float2(kMagic, kMagic));
  const float2 l = __ffma2_rn(__fadd2_rn(hf, make_float2(-kMagic, -kMagic)), make_float2(-0.0625f, -0.0625f), x);
  const float2 lo = __ffma2_rn(l, make_float2(16777216.0f, 16777216.0f), make_float2(kMagic, kMagic));
  a = {__float_as_int(hf.x), __float_as_int(lo.x)};
  b = {__float_as_int(hf.y), __float_as_int(lo.y)};
}

// A pair of fp16 values with the non-finite ones replaced by zero: x - x is
// zero exactly for finite x and a NaN for an infinity or a NaN.
__device__ __forceinline__ uint32_t finite_f16x2(uint32_t w) {
  const __half2 h = *reinterpret_cast<const __half2 *>(&w);
  return w & __heq2_mask(__hsub2(h, h), __float2half2_rn(0.0f));
}
__device__ __forceinline__ uint4 finite_f16x8(uint4 v) {
  return make_uint4(finite_f16x2(v.x), finite_f16x2(v.y), finite_f16x2(v.z), finite_f16x2(v.w));
}

// fp8 e4m3 bits -> X = x 2^9 (|X| < 2^18), exactly.
__device__ __forceinline__ int fix_f8(uint32_t b) {
  b = ((b & 0x7Fu) == 0x7Fu) ? 0u : b;                          // NaN -> 0
  const __half_raw h = __nv_cvt_fp8_to_halfraw((__nv_fp8_storage_t)b, __NV_E4M3);
  const float x = __half2float(__half(h));
  return __float_as_int(__fmaf_rn(x, 512.0f, kMagic)) - kMagicBits;
}

__device__ __forceinline__ long long mad_wide(int a, int b, long long c) {
  return (long long)a * (long long)b + c;
}

__device__ __forceinline__ void sq(Acc3 &a, const Limbs &x) {
  a.s2 = mad_wide(x.hi, x.hi, a.s2);
  a.s1 = mad_wide(x.hi, 2 * x.lo, a.s1);
  a.s0 = mad_wide(x.lo, x.lo, a.s0);
}

// The difference form: with d = c - r formed exactly on the limbs,
//   S_rc = S_rr + sum r d,   S_cc = S_rr + 2 sum r d + sum d^2,
// so a candidate element adds r*d and d*d.  When |X_d| <= 2^28 (every
// candidate within a few thousand units in the last place of the
// reference) that is 3 multiply-adds instead of 7 (|X_d|^2 <= 2^56 and at
// most 64 adds per flush keep every accumulator below 2^63).  x holds the
// reference's limbs; xo and y the reference's and the candidate's limbs
// with one common offset, which cancels in the differences.
__device__ __forceinline__ void diff_add(Acc3 &rd, Acc3 &dd, const Limbs &x, const Limbs &xo,
                                         const Limbs &y) {
  const int dh = y.hi - xo.hi, dl = y.lo - xo.lo;
  if ((unsigned)(dh + 255) <= 510u) {
    const int xd = dh * (1 << 20) + dl;            // |xd| <= 2^28
    rd.s1 = mad_wide(x.hi, xd, rd.s1);
    rd.s0 = mad_wide(x.lo, xd, rd.s0);
    dd.s0 = mad_wide(xd, xd, dd.s0);
  } else {
    rd.s2 = mad_wide(x.hi, dh, rd.s2);
    rd.s1 = mad_wide(x.hi, dl, rd.s1);
    rd.s1 = mad_wide(x.lo, dh, rd.s1);
    rd.s0 = mad_wide(x.lo, dl, rd.s0);
    dd.s2 = mad_wide(dh, dh, dd.s2);
    dd.s1 = mad_wide(dh, 2 * dl, dd.s1);
    dd.s0 = mad_wide(dl, dl, dd.s0);
  }
}

// Warp sum of one lane value T, |T| < 2^95, added to three of the CTA's
// shared digits (digit k weighs 2^32k).  T is cut into six 16-bit pieces,
// five unsigned and the top one signed:
//   T = p0 + p1 2^16 + p2 2^32 + p3 2^48 + p4 2^64 + p5 2^80,
// so every piece's warp sum fits in 32 bits (below 2^21) and takes one
// redux; lane 0 recombines the sums two by two into the digits.
__device__ __forceinline__ void warp_add_t(__int128 T, long long *sdig) {
  const unsigned long long lo = (unsigned long long)T;
  const long long hi = (long long)(T >> 64);             // |hi| < 2^31
  const uint32_t a0 = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)lo & 0xFFFFu);
  const uint32_t a1 = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)(lo >> 16) & 0xFFFFu);
  const uint32_t a2 = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)(lo >> 32) & 0xFFFFu);
  const uint32_t a3 = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)(lo >> 48));
  const uint32_t a4 = __reduce_add_sync(0xFFFFFFFFu, (uint32_t)hi & 0xFFFFu);
  const int a5 = __reduce_add_sync(0xFFFFFFFFu, (int)(hi >> 16));    // |piece| < 2^15
  if ((threadIdx.x & 31) == 0) {
    const long long d[3] = {(long long)a0 + ((long long)a1 << 16), (long long)a2 + ((long long)a3 << 16),
                            (long long)a4 + ((long long)a5 * 65536ll)};
#pragma unroll
    for (int k = 0; k < 3; ++k)
      if (d[k] != 0) atomicAdd(reinterpret_cast<unsigned long long *>(sdig + k), (unsigned long long)d[k]);
  }
}

// sum = s2 2^40 + s1 2^20 + s0.  Between two flushes a lane adds at most 64
// products (one tile), each |r d|, |d d| <= 2^56 in the short form and each
// partial product <= 2^42 in the limb form, so |s0| < 2^63, |s1| < 2^56,
// |s2| < 2^49 and |sum| < 2^90.
__device__ __forceinline__ void flush3(Acc3 &a, long long *sdig) {
  const __int128 T = (__int128)a.s0 + (__int128)a.s1 * ((__int128)1 << 20) +
                    (__int128)a.s2 * ((__int128)1 << 40);
  warp_add_t(T, sdig);
  a.s2 = a.s1 = a.s0 = 0;
}

// fp8 e4m3 products are below 2^36, so a tile's sum is below 2^42.
__device__ __forceinline__ void flush1(long long &s, long long *sdig) {
  warp_add_t((__int128)s, sdig);
  s = 0;
}

__device__ __forceinline__ uint32_t half_of(const uint4 &v, int k) {
  const uint32_t w = k < 2 ? v.x : k < 4 ? v.y : k < 6 ? v.z : v.w;
  return (k & 1) ? (w >> 16) : (w & 0xFFFFu);
}
__device__ __forceinline__ uint32_t byte_of(const uint4 &v, int k) {
  const uint32_t w = k < 4 ? v.x : k < 8 ? v.y : k < 12 ? v.z : v.w;
  return (w >> (8 * (k & 3))) & 0xFFu;
}
// Element k of a chunk of E5M2 / fnuz fp8 as the bits of its exact fp16 value.
template <uint32_t DT>
__device__ __forceinline__ uint32_t fp8_half(const uint4 &v, int k) {
  return fp8x2_to_half2_bits<DT>(byte_of(v, k)) & 0xFFFFu;
}

// The sums of candidates j and (if TWO) j + 1 over one tile's share of a
// warp, added to the CTA's shared digits sd (slots 1 + 2j .. 4 + 2j), and
// with RR also sum r*r into the reference's slot (sdig0) from the same
// decoded values.  With an odd number of candidates the last call has
// TWO = false and does no work for a second candidate.
template <int DT, bool TWO, bool RR>
__device__ __forceinline__ void pair_sums(const CmpRegion &R, uint64_t ref, uint64_t cb0, uint64_t cb1,
                                          uint32_t c0, uint32_t c1, uint32_t rounds, uint32_t nb,
                                          long long *sd, long long *sdig0) {
  const uint32_t lane = threadIdx.x & 31;
  Acc3 rc0 = {0, 0, 0}, cc0 = {0, 0, 0}, rc1 = {0, 0, 0}, cc1 = {0, 0, 0}, rr = {0, 0, 0};
  long long rc8_0 = 0, cc8_0 = 0, rc8_1 = 0, cc8_1 = 0, r8 = 0;
#pragma unroll 1
  for (uint32_t r = 0; r < rounds; ++r) {
    const uint32_t c = c0 + 32u * r + lane;
    uint4 rv = make_uint4(0u, 0u, 0u, 0u), v0 = rv, v1 = rv;
    if (c < c1) {
      const uint32_t bytes = min(16u, nb - 16u * c);
      rv = load_chunk(ref + 16ull * c, bytes, R.vec, true);     // L1 hit after the first pair
      v0 = load_chunk(cb0 + 16ull * c, bytes, R.vec, false);
      if (TWO) v1 = load_chunk(cb1 + 16ull * c, bytes, R.vec, false);
    }
    if (DT == kF16) {
      rv = finite_f16x8(rv);
      v0 = finite_f16x8(v0);
      if (TWO) v1 = finite_f16x8(v1);
      const uint32_t rw[4] = {rv.x, rv.y, rv.z, rv.w};
      const uint32_t w0[4] = {v0.x, v0.y, v0.z, v0.w};
      const uint32_t w1[4] = {v1.x, v1.y, v1.z, v1.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        Limbs xb[2], y0[2], y1[2];
        fix_f16x2_biased(rw[q], xb[0], xb[1]);
        fix_f16x2_biased(w0[q], y0[0], y0[1]);
        if (TWO) fix_f16x2_biased(w1[q], y1[0], y1[1]);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const Limbs x = {xb[h].hi - kMagicBits, xb[h].lo - kMagicBits};
          if (RR) sq(rr, x);
          diff_add(rc0, cc0, x, xb[h], y0[h]);
          if (TWO) diff_add(rc1, cc1, x, xb[h], y1[h]);
        }
      }
    } else if (DT != kF8) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const Limbs x = fix_f16(fp8_half<DT>(rv, k));
        if (RR) sq(rr, x);
        diff_add(rc0, cc0, x, x, fix_f16(fp8_half<DT>(v0, k)));
        if (TWO) diff_add(rc1, cc1, x, x, fix_f16(fp8_half<DT>(v1, k)));
      }
    } else {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const int x = fix_f8(byte_of(rv, k));
        if (RR) r8 = mad_wide(x, x, r8);
        const int y0 = fix_f8(byte_of(v0, k));
        rc8_0 = mad_wide(x, y0, rc8_0); cc8_0 = mad_wide(y0, y0, cc8_0);
        if (TWO) {
          const int y1 = fix_f8(byte_of(v1, k));
          rc8_1 = mad_wide(x, y1, rc8_1); cc8_1 = mad_wide(y1, y1, cc8_1);
        }
      }
    }
  }
  if (DT != kF8) {
    if (RR) flush3(rr, sdig0);
    flush3(rc0, sd);
    flush3(cc0, sd + kWin);
    if (TWO) { flush3(rc1, sd + 2 * kWin); flush3(cc1, sd + 3 * kWin); }
  } else {
    if (RR) flush1(r8, sdig0);
    flush1(rc8_0, sd);
    flush1(cc8_0, sd + kWin);
    if (TWO) { flush1(rc8_1, sd + 2 * kWin); flush1(cc8_1, sd + 3 * kWin); }
  }
}

// One tile of an fp16 or fp8 region: S_rr, then the candidates two at a
// time (the reference chunk is decoded once per pair).  With a single
// candidate S_rr is added in the candidate's pass, from the same decoded
// reference values (with two candidates per pass the extra accumulator
// costs more than the second decode saves).  E5M2 and the fnuz
// formats go through their exact fp16 values (and fp16's binary point).
// For fp16 and those formats the candidate slots hold the difference-form
// sums sum r d and sum d^2 (diff_add); the host forms S_rc and S_cc.
template <int DT>
__device__ __noinline__ void eq_tile_fixed(const EqParams &p, const CmpRegion &R, uint32_t region,
                                           uint64_t a, uint32_t nb, long long *sdig) {
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t nchunks = (nb + 15u) >> 4;
  const uint32_t per_warp = (nchunks + kWarps - 1) / kWarps;
  const uint32_t c0 = warp * per_warp;
  const uint32_t c1 = min(c0 + per_warp, nchunks);
  const uint32_t rounds = (per_warp + 31u) >> 5;     // the same for every warp
  const uint64_t ref = R.ref + a;
  if (p.do_rr && p.K >= 2) {           // with one candidate S_rr rides on its pass
    Acc3 rr = {0, 0, 0};
    long long r8 = 0;
#pragma unroll 1
    for (uint32_t r = 0; r < rounds; ++r) {
      const uint32_t c = c0 + 32u * r + lane;
      uint4 rv = make_uint4(0u, 0u, 0u, 0u);
      if (c < c1) rv = load_chunk(ref + 16ull * c, min(16u, nb - 16u * c), R.vec, true);
      if (DT == kF16) {
#pragma unroll
        for (int k = 0; k < 8; ++k) sq(rr, fix_f16(half_of(rv, k)));
      } else if (DT != kF8) {
#pragma unroll
        for (int k = 0; k < 16; ++k) sq(rr, fix_f16(fp8_half<DT>(rv, k)));
      } else {
#pragma unroll
        for (int k = 0; k < 16; ++k) { const int x = fix_f8(byte_of(rv, k)); r8 = mad_wide(x, x, r8); }
      }
    }
    if (DT != kF8) flush3(rr, sdig); else flush1(r8, sdig);
  }
  for (uint32_t j = 0; j < p.K; j += 2) {
    const uint64_t cb0 = p.cands[(size_t)j * p.nregions + region] + a;
    long long *sd = sdig + (1 + 2 * j) * kWin;
    const uint64_t cb1 = j + 1 < p.K ? p.cands[(size_t)(j + 1) * p.nregions + region] + a : cb0;
    if (j + 1 < p.K) pair_sums<DT, true, false>(R, ref, cb0, cb1, c0, c1, rounds, nb, sd, sdig);
    else if (p.K == 1 && p.do_rr) pair_sums<DT, false, true>(R, ref, cb0, cb1, c0, c1, rounds, nb, sd, sdig);
    else pair_sums<DT, false, false>(R, ref, cb0, cb1, c0, c1, rounds, nb, sd, sdig);
  }
}

// Add the CTA's shared digits of `region` to its global digits; zero them.
__device__ void cta_flush(const EqParams &p, uint32_t region, uint32_t dtype, long long *sdig) {
  __syncthreads();
  const int dig0 = dtype == kF32 ? Fmt<kF32>::kDig : dtype == kBF16 ? Fmt<kBF16>::kDig
                 : dtype == kF8 ? Fmt<kF8>::kDig : Fmt<kF16>::kDig;   // other fp8: fp16's point
  const uint32_t nloc = 1u + 2u * p.K;
  for (uint32_t x = threadIdx.x; x < nloc * kWin; x += blockDim.x) {
    const long long v = sdig[x];
    if (v != 0) {
      const uint32_t ls = x / kWin, k = x % kWin;
      atomicAdd(reinterpret_cast<unsigned long long *>(global_digits(p, region, global_slot(p, ls)) +
                                                       dig0 + k),
                (unsigned long long)v);
      sdig[x] = 0;
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kThreads, 3) eq_kernel(EqParams p) {   // 3 CTAs per SM
  __shared__ long long sdig[(1 + 2 * kMaxCands) * kWin];
  for (uint32_t x = threadIdx.x; x < (1 + 2 * kMaxCands) * kWin; x += blockDim.x) sdig[x] = 0;
  __syncthreads();
  const uint64_t t0 = p.ntiles * blockIdx.x / gridDim.x;
  const uint64_t t1 = p.ntiles * (blockIdx.x + 1) / gridDim.x;
  uint32_t cur = 0xFFFFFFFFu, cur_dtype = 0;
  for (uint64_t t = t0; t < t1; ++t) {
    const uint32_t i = find_region(p.regions, p.nregions, t);
    const CmpRegion R = p.regions[i];
    if (i != cur) {
      if (cur != 0xFFFFFFFFu) cta_flush(p, cur, cur_dtype, sdig);
      cur = i;
      cur_dtype = R.dtype;
    }
    const uint64_t a = (t - R.tile0) * kTileBytes;
    const uint32_t nb = (uint32_t)umin64(kTileBytes, R.bytes - a);
    switch (R.dtype) {
      case kF32: eq_tile<kF32>(p, R, i, a, nb, sdig); break;
      case kBF16: eq_tile<kBF16>(p, R, i, a, nb, sdig); break;
      case kF16: eq_tile_fixed<kF16>(p, R, i, a, nb, sdig); break;
      case kF8E5M2: eq_tile_fixed<kF8E5M2>(p, R, i, a, nb, sdig); break;
      case kF8E4FNUZ: eq_tile_fixed<kF8E4FNUZ>(p, R, i, a, nb, sdig); break;
      case kF8E5FNUZ: eq_tile_fixed<kF8E5FNUZ>(p, R, i, a, nb, sdig); break;
      default: eq_tile_fixed<kF8>(p, R, i, a, nb, sdig); break;
    }
  }
  if (cur != 0xFFFFFFFFu) cta_flush(p, cur, cur_dtype, sdig);
}

}  // namespace

int eq_max_ctas_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, eq_kernel, kThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return n > 0 ? n : 1;
}

int launch_eq(const EqParams &p, int grid, void *stream) {
  eq_kernel<<<grid, kThreads, 0, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
