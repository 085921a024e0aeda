// device.cuh -- device building blocks shared by the kernels: the exact
// fp16 / fp8 decoders, 64-bit integer helpers, 16-byte loads and stores
// and the tile -> region lookup.
#pragma once
#include <stdint.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <cuda_fp8.h>
#include "plan.h"

namespace asmv {

// ---------------------------------------------------------------- decoders
__device__ __forceinline__ float2 f16x2_to_f32(uint32_t w) {
  return __half22float2(*reinterpret_cast<const __half2 *>(&w));
}
// Two fp8 values (low byte first) as an exact half2, per format.  The fnuz
// formats are half the value of the OCP format with the same bits, finite
// at the top exponent (E4M3: 0x7F is 240; E5M2: exponent 31 holds
// (4..7) * 8192), with 0x80 the NaN.
__device__ __forceinline__ uint32_t half_bits_fnuz(uint32_t b, uint32_t hw, bool e5) {
  const uint32_t sign = (b & 0x80u) << 8;
  if (b == 0x80u) return 0x7E00u;
  if (!e5 && (b & 0x7Fu) == 0x7Fu) return sign | 0x5B80u;                   // 240
  if (e5 && (b & 0x7Cu) == 0x7Cu) return sign | 0x7800u | ((b & 3u) << 8);  // (4+m) 2^13
  const __half h = __hmul(__ushort_as_half((unsigned short)hw), __float2half(0.5f));
  return (uint32_t)__half_as_ushort(h);
}

template <uint32_t DT>
__device__ __forceinline__ uint32_t fp8x2_to_half2_bits(uint32_t w16) {
  const __nv_fp8x2_storage_t s = (__nv_fp8x2_storage_t)(w16 & 0xFFFFu);
  const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2(
      s, (DT == kF8 || DT == kF8E4FNUZ) ? __NV_E4M3 : __NV_E5M2);
  if (DT == kF8 || DT == kF8E5M2) return (uint32_t)h.x | ((uint32_t)h.y << 16);
  const bool e5 = DT == kF8E5FNUZ;
  return half_bits_fnuz(w16 & 0xFFu, h.x, e5) | (half_bits_fnuz((w16 >> 8) & 0xFFu, h.y, e5) << 16);
}

// ---------------------------------------------------------------- integers
__device__ __forceinline__ unsigned long long umin64(unsigned long long a, unsigned long long b) {
  return a < b ? a : b;
}
__device__ __forceinline__ unsigned long long umax64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}

// ---------------------------------------------------------------- memory
__device__ __forceinline__ uint4 ldg16(uint64_t addr) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(addr));
  return v;
}
__device__ __forceinline__ void stg16(uint64_t addr, uint4 v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};"
               :: "l"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}

// Up to 16 bytes at any alignment; bytes past `n` read as zero.
__device__ __forceinline__ uint4 load_bytes(uint64_t addr, uint32_t n) {
  uint32_t w[4] = {0u, 0u, 0u, 0u};
  const uint8_t *p = reinterpret_cast<const uint8_t *>(addr);
#pragma unroll
  for (uint32_t j = 0; j < 16; ++j)
    if (j < n) w[j >> 2] |= (uint32_t)__ldg(p + j) << (8 * (j & 3));
  return make_uint4(w[0], w[1], w[2], w[3]);
}
__device__ __forceinline__ void store_bytes(uint64_t addr, uint4 v, uint32_t n) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint8_t *p = reinterpret_cast<uint8_t *>(addr);
#pragma unroll
  for (uint32_t j = 0; j < 16; ++j)
    if (j < n) p[j] = (uint8_t)(w[j >> 2] >> (8 * (j & 3)));
}

// The debug-bounds build's check of an access [a, a + n) against the
// allocation it belongs to: true when inside; otherwise it sets kErrBounds
// in *err and the caller skips the access.  The normal build always passes.
__device__ __forceinline__ bool in_alloc(const Span &s, uint64_t a, uint64_t n, uint32_t *err) {
#if ASMV_DEBUG_BOUNDS
  if (a >= s.lo && a <= s.hi && n <= s.hi - a) return true;
  atomicOr(err, kErrBounds);
  return false;
#else
  (void)s; (void)a; (void)n; (void)err;
  return true;
#endif
}

// Region owning tile t: the last i with tile0[i] <= t (regions with no
// tiles share their successor's tile0 and are skipped).
template <class R>
__device__ __forceinline__ uint32_t find_region(const R *regs, uint32_t n, uint64_t t) {
  uint32_t lo = 0, hi = n;          // invariant: regs[lo].tile0 <= t < regs[hi].tile0
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (regs[mid].tile0 <= t) lo = mid; else hi = mid;
  }
  return lo;
}

}  // namespace asmv
