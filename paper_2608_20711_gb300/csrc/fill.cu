// fill.cu -- Tier 1 guarded input synthesis (AsmEvo Sec. 3.4, Tier 1):
// every region's payload receives its seeded Philox4x32-10 stream shaped to
// its distribution, and both guard bands receive the region's canary byte.
//
// One 16-byte chunk c of a payload always holds the same bytes, whatever
// the payload's address: RAW chunk c is Philox block c; fp32 UNIFORM and
// NORMAL map element i to word (i mod 4) of block (i div 4) (NORMAL:
// Box-Muller on word pairs (0,1) and (2,3)), binary64 to half of such a
// block; the 16-bit and 8-bit float formats take one block per chunk, so
// that each element draws as many Philox bits as it stores (16-bit: a
// Box-Muller pair per word, UNIFORM a 16-bit fraction per half word; 8-bit:
// a pair per half word, UNIFORM an 8-bit fraction per byte).  Aligned
// payloads are written with 128-bit stores; unaligned payloads and the
// short last chunk with byte stores.
//
// Roofline: HBM writes of payload + guard bytes.  Philox costs 18 wide
// multiplies per block on the FMA-heavy pipe (20, less two formed once per
// tile), so a RAW fill is co-limited by the block rate; NORMAL adds its
// transform, which makes the fill issue-bound for every NORMAL format.  Each
// thread computes two chunks at a time so that the two Philox chains overlap.
#include "fill_math.cuh"
#include "ln_table.h"

namespace asmv {
namespace {

__device__ __forceinline__ float uniform_of(uint32_t w, float lo, float width) {
  const float f = __fmul_rn(__uint2float_rn(w >> 8), 0x1p-24f);
  return __fadd_rn(lo, __fmul_rn(f, width));
}

// v = mean + sd*z for the four normals of a block, two per packed
// instruction: v[0], v[2] from z0 of the two pairs, v[1], v[3] from z1.
__device__ __forceinline__ void normal4(uint4 w, float mean, float sd, uint32_t tab, float v[4]) {
  float2 z0, z1;
  box_muller2(w, tab, z0, z1);
  // multiply, then add, each rounded: scalar _rn operations, which are never
  // contracted (a packed multiply followed by a packed add was fused into
  // one multiply-add whatever their rounding modifiers)
  v[0] = __fadd_rn(mean, __fmul_rn(sd, z0.x));
  v[1] = __fadd_rn(mean, __fmul_rn(sd, z1.x));
  v[2] = __fadd_rn(mean, __fmul_rn(sd, z0.y));
  v[3] = __fadd_rn(mean, __fmul_rn(sd, z1.y));
}

// uniform_of for the four words of a block, two per packed instruction.
__device__ __forceinline__ void uniform4(uint4 w, float lo, float width, float v[4]) {
  const float2 fa = fmul2(make_float2(__uint2float_rn(w.x >> 8), __uint2float_rn(w.y >> 8)), f2(0x1p-24f));
  const float2 fb = fmul2(make_float2(__uint2float_rn(w.z >> 8), __uint2float_rn(w.w >> 8)), f2(0x1p-24f));
  // f (exact) times the width, then plus lo, each rounded (scalar _rn: never contracted)
  v[0] = __fadd_rn(lo, __fmul_rn(fa.x, width));
  v[1] = __fadd_rn(lo, __fmul_rn(fa.y, width));
  v[2] = __fadd_rn(lo, __fmul_rn(fb.x, width));
  v[3] = __fadd_rn(lo, __fmul_rn(fb.y, width));
}

// UNIFORM of the narrow formats: v = lo + (k scale) width, k a 16-bit or
// 8-bit field (k scale is exact).
__device__ __forceinline__ float uniform_frac(uint32_t k, float scale, float lo, float width) {
  return __fadd_rn(lo, __fmul_rn(__fmul_rn(__uint2float_rn(k), scale), width));
}

__device__ __forceinline__ uint32_t int_of(uint32_t w, int64_t lo, uint64_t span) {
  return (uint32_t)(lo + (int64_t)(((uint64_t)w * span) >> 32));
}

// Round keys of a launch and the shared-memory addresses of this lane's
// copies of the tables.
struct Keys {
  const uint32_t *k0, *k1;
  uint32_t ln;              // ln reduction row 0 (fp32 / binary64 NORMAL)
  uint32_t offT;            // angle table entry 0
  uint32_t offR16;          // 16-bit radius chord "entry 1776" (the bias of F' >> 19)
  uint32_t offR8;           // 8-bit radius entry 0
#if ASMV_DEBUG_BOUNDS
  uint32_t *err;
#endif
};

__device__ __forceinline__ uint4 payload_block(const Keys &K, const PhiloxPre &Q, uint64_t b) {
  return philox10_pre((uint32_t)b, Q, K.k0, K.k1);
}
// The first Philox block of chunk c, for the blocks per chunk (1/2, 1, 2 or 4)
// that make_chunk takes.
static_assert((kFillTileChunks & (kFillTileChunks - 1)) == 0, "a tile's Philox blocks share the high word");
template <uint32_t DIST, uint32_t DT>
__device__ __forceinline__ uint64_t first_block(uint64_t c) {
  if (DIST == kRaw) return c;
  if (DIST == kIntRange) return DT == kI64 ? c >> 1 : DT == kI16 ? 2 * c : DT == kI32 ? c : 4 * c;
  return DT == kF64 ? c >> 1 : c;
}

// Four fp32 values of one block (fp32 formats), per float distribution.
template <uint32_t DIST>
__device__ __forceinline__ void float4_of(uint4 w, const FillRegion &r, const Keys &K, float v[4]) {
  if (DIST == kNormal) normal4(w, r.f0, r.f1, K.ln, v);
  else uniform4(w, r.f0, r.f1, v);
}

__device__ __forceinline__ uint32_t pack_fp8(uint32_t DT, const float v[4]) {
  if (DT == kF8) return pack_f8x4(v[0], v[1], v[2], v[3]);
  if (DT == kF8E5M2) return pack_e5m2x4(v[0], v[1], v[2], v[3]);
  if (DT == kF8E4FNUZ)
    return enc_e4m3fnuz(v[0]) | (enc_e4m3fnuz(v[1]) << 8) | (enc_e4m3fnuz(v[2]) << 16) |
           (enc_e4m3fnuz(v[3]) << 24);
  return enc_e5m2fnuz(v[0]) | (enc_e5m2fnuz(v[1]) << 8) | (enc_e5m2fnuz(v[2]) << 16) |
         (enc_e5m2fnuz(v[3]) << 24);
}

// The 16 bytes of chunk c.
template <uint32_t DIST, uint32_t DT>
__device__ __forceinline__ uint4 make_chunk(const FillRegion &r, const Keys &K, const PhiloxPre &Q, uint64_t c) {
  if (DIST == kRaw) return payload_block(K, Q, c);
  if (DIST == kIntRange) {
    if (DT == kI64) {                           // 2 elements: words 2(c mod 2), +1 of block c/2
      const uint4 w = payload_block(K, Q, c >> 1);
      const uint32_t wa = (c & 1) ? w.z : w.x, wb = (c & 1) ? w.w : w.y;
      const int64_t a = r.ilo + (int64_t)(((uint64_t)wa * r.ispan) >> 32);
      const int64_t b = r.ilo + (int64_t)(((uint64_t)wb * r.ispan) >> 32);
      return make_uint4((uint32_t)a, (uint32_t)((uint64_t)a >> 32), (uint32_t)b,
                        (uint32_t)((uint64_t)b >> 32));
    }
    if (DT == kI16) {                           // 8 elements: blocks 2c, 2c+1
      uint32_t out[4];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint4 w = payload_block(K, Q, 2 * c + q);
        out[2 * q] = (int_of(w.x, r.ilo, r.ispan) & 0xFFFFu) | (int_of(w.y, r.ilo, r.ispan) << 16);
        out[2 * q + 1] = (int_of(w.z, r.ilo, r.ispan) & 0xFFFFu) | (int_of(w.w, r.ilo, r.ispan) << 16);
      }
      return make_uint4(out[0], out[1], out[2], out[3]);
    }
    if (DT == kI32) {
      const uint4 w = payload_block(K, Q, c);
      return make_uint4(int_of(w.x, r.ilo, r.ispan), int_of(w.y, r.ilo, r.ispan),
                        int_of(w.z, r.ilo, r.ispan), int_of(w.w, r.ilo, r.ispan));
    } else {                                    // 8-bit: 16 elements, blocks 4c..4c+3
      uint32_t out[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 w = payload_block(K, Q, 4 * c + q);
        out[q] = (int_of(w.x, r.ilo, r.ispan) & 0xFFu) | ((int_of(w.y, r.ilo, r.ispan) & 0xFFu) << 8) |
                 ((int_of(w.z, r.ilo, r.ispan) & 0xFFu) << 16) | (int_of(w.w, r.ilo, r.ispan) << 24);
      }
      return make_uint4(out[0], out[1], out[2], out[3]);
    }
  }
  // UNIFORM / NORMAL on float dtypes
  if (DT == kF64) {                             // 2 elements: words 2(c mod 2), +1 of block c/2
    const uint4 w = payload_block(K, Q, c >> 1);
    float v0, v1;
    if (DIST == kNormal) {
      float z0, z1;
      if (c & 1) box_muller(w.z, w.w, K.ln, z0, z1);
      else box_muller(w.x, w.y, K.ln, z0, z1);
      v0 = __fadd_rn(r.f0, __fmul_rn(r.f1, z0));
      v1 = __fadd_rn(r.f0, __fmul_rn(r.f1, z1));
    } else {
      v0 = uniform_of((c & 1) ? w.z : w.x, r.f0, r.f1);
      v1 = uniform_of((c & 1) ? w.w : w.y, r.f0, r.f1);
    }
    const unsigned long long a = (unsigned long long)__double_as_longlong((double)v0);
    const unsigned long long b = (unsigned long long)__double_as_longlong((double)v1);
    return make_uint4((uint32_t)a, (uint32_t)(a >> 32), (uint32_t)b, (uint32_t)(b >> 32));
  }
  if (DT == kF32) {
    float v[4];
    float4_of<DIST>(payload_block(K, Q, c), r, K, v);
    return make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                      __float_as_uint(v[3]));
  }
  const uint4 w = payload_block(K, Q, c);       // the narrow formats: block c
  const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
  uint32_t out[4];
  if (DT == kBF16 || DT == kF16) {              // 8 elements: a pair (or two fractions) per word
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float a, b;
      if (DIST == kNormal) {
        normal16_pair(ww[q], K.offR16, K.offT, r.f0, r.f1, a, b);
      } else {
        a = uniform_frac(ww[q] & 0xFFFFu, 0x1p-16f, r.f0, r.f1);
        b = uniform_frac(ww[q] >> 16, 0x1p-16f, r.f0, r.f1);
      }
      out[q] = (DT == kBF16) ? pack_bf16x2(a, b) : pack_f16x2(a, b);
    }
  } else {                                      // fp8: 16 elements, four per word
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float v[4];
      if (DIST == kNormal) {
        normal8_word(ww[q], K.offR8, K.offT, r.f0, r.f1, v);
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) v[e] = uniform_frac((ww[q] >> (8 * e)) & 0xFFu, 0x1p-8f, r.f0, r.f1);
      }
      out[q] = pack_fp8(DT, v);
    }
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

// Chunk i of a tile whose first chunk, c0 of the payload, is at `base`: one
// 16-byte store for the tile's chunks below nvec, byte stores for the rest
// (the payload's short last chunk, every chunk of an unaligned payload).
__device__ __forceinline__ void store_chunk(const FillRegion &r, const Keys &K, uint64_t base, uint64_t c0,
                                            uint32_t i, uint32_t nvec, uint4 v) {
  const uint64_t addr = base + 16 * i;
#if ASMV_DEBUG_BOUNDS
  if (!in_alloc(r.alloc, addr, umin64(16, r.bytes - 16 * (c0 + i)), K.err)) return;
#else
  (void)K;
#endif
  if (i < nvec) stg16(addr, v);
  else store_bytes(addr, v, (uint32_t)umin64(16, r.bytes - 16 * (c0 + i)));
}

// Thread t makes chunks t + 2 k kFillThreads and t + (2 k + 1) kFillThreads
// of the tile together, so that their Philox chains overlap; where a thread
// has no second chunk it recomputes its first and stores once.
template <uint32_t DIST, uint32_t DT>
__device__ void fill_tile(const FillRegion &r, const Keys &K, uint64_t tile_in_region) {
  const uint64_t c0 = tile_in_region * kFillTileChunks;
  const uint64_t nchunks = (r.bytes + 15) >> 4;
  const uint64_t full = r.bytes >> 4;
  const uint32_t nloc = (uint32_t)umin64(kFillTileChunks, nchunks - c0);
  // A tile's blocks [first_block(c0), first_block(c0 + kFillTileChunks)) start
  // at a multiple of their count, a power of two below 2^32: one high word.
  const PhiloxPre Q = philox_pre(r.region_id, (uint32_t)(first_block<DIST, DT>(c0) >> 32), K.k0);
  const uint32_t nvec = r.vec ? (uint32_t)umin64(nloc, full > c0 ? full - c0 : 0) : 0u;
  const uint64_t base = r.payload + 16 * c0;
#pragma unroll 1
  for (uint32_t i = threadIdx.x; i < nloc; i += 2 * kFillThreads) {
    const uint32_t i2 = i + kFillThreads;
    const bool two = i2 < nloc;
    const uint4 va = make_chunk<DIST, DT>(r, K, Q, c0 + i);
    const uint4 vb = make_chunk<DIST, DT>(r, K, Q, c0 + (two ? i2 : i));
    store_chunk(r, K, base, c0, i, nvec, va);
    if (two) store_chunk(r, K, base, c0, i2, nvec, vb);
  }
}

__device__ void fill_tile_dispatch(const FillRegion &r, const Keys &K, uint64_t t) {
  switch (r.dist) {
    case kRaw: fill_tile<kRaw, kU8>(r, K, t); break;
    case kIntRange:
      switch (r.dtype) {
        case kI32: fill_tile<kIntRange, kI32>(r, K, t); break;
        case kI16: fill_tile<kIntRange, kI16>(r, K, t); break;
        case kI64: fill_tile<kIntRange, kI64>(r, K, t); break;
        default: fill_tile<kIntRange, kI8>(r, K, t); break;
      }
      break;
    case kUniform:
      switch (r.dtype) {
        case kF32: fill_tile<kUniform, kF32>(r, K, t); break;
        case kBF16: fill_tile<kUniform, kBF16>(r, K, t); break;
        case kF16: fill_tile<kUniform, kF16>(r, K, t); break;
        case kF8E5M2: fill_tile<kUniform, kF8E5M2>(r, K, t); break;
        case kF8E4FNUZ: fill_tile<kUniform, kF8E4FNUZ>(r, K, t); break;
        case kF8E5FNUZ: fill_tile<kUniform, kF8E5FNUZ>(r, K, t); break;
        case kF64: fill_tile<kUniform, kF64>(r, K, t); break;
        default: fill_tile<kUniform, kF8>(r, K, t); break;
      }
      break;
    case kNormal:
      switch (r.dtype) {
        case kF32: fill_tile<kNormal, kF32>(r, K, t); break;
        case kBF16: fill_tile<kNormal, kBF16>(r, K, t); break;
        case kF16: fill_tile<kNormal, kF16>(r, K, t); break;
        case kF8E5M2: fill_tile<kNormal, kF8E5M2>(r, K, t); break;
        case kF8E4FNUZ: fill_tile<kNormal, kF8E4FNUZ>(r, K, t); break;
        case kF8E5FNUZ: fill_tile<kNormal, kF8E5FNUZ>(r, K, t); break;
        case kF64: fill_tile<kNormal, kF64>(r, K, t); break;
        default: fill_tile<kNormal, kF8>(r, K, t); break;
      }
      break;
    default: break;                              // NONE: payload untouched
  }
}

// Copy `entries` table entries of T into shared memory at `off`, `copies`
// copies of each side by side.
template <class T>
__device__ __forceinline__ void load_table(uint8_t *sm, uint32_t off, const T *src, uint32_t entries,
                                           uint32_t copies) {
  for (uint32_t i = threadIdx.x; i < entries * copies; i += kFillThreads)
    *reinterpret_cast<T *>(sm + off + sizeof(T) * i) = src[i / copies];
}

__global__ void __launch_bounds__(kFillThreads) fill_kernel(const __grid_constant__ FillParams p) {
  extern __shared__ __align__(16) uint8_t sm[];
  const FillLayout &L = p.smem;
  if (L.angle != kNoTable) load_table(sm, L.angle, kAngleTable, 256, kAngleCopies);
  if (L.rad16 != kNoTable) load_table(sm, L.rad16, kRadius16Table, 512, kRad16Copies);
  if (L.rad8 != kNoTable) load_table(sm, L.rad8, kRadius8Table, 256, kRad8Copies);
  if (L.ln != kNoTable) load_table(sm, L.ln, kLnTableInit, ASMV_LN_TABLE_ROWS, kLnCopies);
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t G = gridDim.x, b = blockIdx.x;
  // Tiles b, b + G, b + 2G, ...: every CTA gets its share of every region,
  // so regions of very different cost per tile (NORMAL against RAW) spread
  // evenly over the SMs.
  if (b < p.ntiles) {
    const uint32_t sm32 = (uint32_t)__cvta_generic_to_shared(sm);
    Keys K = {p.key0, p.key1, sm32 + L.ln + 16u * (lane % kLnCopies),
              sm32 + L.angle + 8u * (lane % kAngleCopies),
              sm32 + L.rad16 + 8u * (lane % kRad16Copies) - 1776u * 8u * kRad16Copies,
              sm32 + L.rad8 + 4u * (lane % kRad8Copies)};
#if ASMV_DEBUG_BOUNDS
    K.err = p.err;
#endif
    // The region records of the CTA's next kTileBatch tiles: one binary
    // search per thread, all in flight together, copied to shared memory.
    // (A search per tile, with 4096 regions, held every warp of the CTA for
    // a dozen dependent loads each time the CTA stepped into a new region.)
    constexpr uint32_t kTileBatch = 128;
    __shared__ FillRegion tile_region[kTileBatch];
    for (uint64_t t0 = b; t0 < p.ntiles; t0 += G * kTileBatch) {
      const uint64_t tt = t0 + threadIdx.x * G;
      __syncthreads();
      if (threadIdx.x < kTileBatch && tt < p.ntiles)
        tile_region[threadIdx.x] = p.regions[find_region(p.regions, p.nregions, tt)];
      __syncthreads();
      const uint32_t nt = (uint32_t)umin64(kTileBatch, (p.ntiles - t0 + G - 1) / G);
      for (uint32_t j = 0; j < nt; ++j) {
        const FillRegion r = tile_region[j];
        fill_tile_dispatch(r, K, t0 + j * G - r.tile0);
      }
    }
  }
  // guard bands: one warp per segment
  const uint64_t warp = b * kFillWarps + (threadIdx.x >> 5), nw = G * kFillWarps;
  for (uint64_t s = warp; s < p.nsegs; s += nw) {
    const GuardSeg g = p.segs[s];
#if ASMV_DEBUG_BOUNDS
    if (!in_alloc(g.alloc, g.ptr, g.len, p.err)) continue;
#endif
    uint8_t *dst = reinterpret_cast<uint8_t *>(g.ptr);
    for (uint32_t j = lane; j < g.len; j += 32) dst[j] = g.canary;
  }
}

}  // namespace

// CTAs of the fill per SM with `smem_bytes` of tables, on the current device
// (which also receives the kernel's shared-memory opt-in); 0 on an error.
int fill_max_ctas_per_sm(uint32_t smem_bytes) {
  const size_t most = (size_t)kAngleBytes + kRad16Bytes + kRad8Bytes + kLnBytes;
  if (cudaFuncSetAttribute(fill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)most) !=
      cudaSuccess)
    return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fill_kernel, kFillThreads, smem_bytes) !=
      cudaSuccess)
    return 0;
  return n;
}

int launch_fill(const FillParams &p, int grid, void *stream) {
  fill_kernel<<<grid, kFillThreads, p.smem.bytes, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
