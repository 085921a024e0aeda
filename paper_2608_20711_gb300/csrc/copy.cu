// copy.cu -- Tier 2 replay restore (AsmEvo Sec. 3.4, Tier 2): before a
// candidate replays a captured dispatch, every referenced region gets its
// captured pre-dispatch bytes back and its guard bands are rewritten with
// the canary, so each candidate starts from identical memory.  The same
// kernel runs the capture direction (region payload -> snapshot buffer,
// no guard writes).
//
// Work split: the payloads of all regions form one space of 16 KiB tiles; a
// persistent grid gives each CTA a contiguous tile range.  In a tile, thread
// t moves 16-byte chunks t, t+256, t+512, t+768: all four loads are issued
// before the four stores.  A region whose source and destination are both
// 16-byte aligned moves with 128-bit accesses, others byte by byte.  Guard
// bands are written by warps after the tiles.
//
// Roofline: HBM, reads of the source plus writes of the destination
// (2 x payload bytes) and the guard bytes written.
#include "device.cuh"

namespace asmv {
namespace {

__device__ __forceinline__ void copy_tile(const CopyRegion &r, uint64_t t, uint32_t *err) {
  (void)err;
  const uint64_t off = t * kTileBytes;
  const uint64_t nb = umin64(kTileBytes, r.bytes - off);
  const uint32_t nch = (uint32_t)((nb + 15) / 16);
  constexpr int kPer = kTileChunks / kThreads;        // 4
  uint4 v[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const uint32_t c = threadIdx.x + k * kThreads;
    if (c < nch) {
      const uint64_t a = r.src + off + 16ull * c;
      const uint32_t n = (uint32_t)umin64(16, nb - 16ull * c);
#if ASMV_DEBUG_BOUNDS
      if (!in_alloc(r.src_alloc, a, n, err)) { v[k] = make_uint4(0u, 0u, 0u, 0u); continue; }
#endif
      v[k] = (r.vec && n == 16) ? ldg16(a) : load_bytes(a, n);
    }
  }
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const uint32_t c = threadIdx.x + k * kThreads;
    if (c < nch) {
      const uint64_t a = r.dst + off + 16ull * c;
      const uint32_t n = (uint32_t)umin64(16, nb - 16ull * c);
#if ASMV_DEBUG_BOUNDS
      if (!in_alloc(r.dst_alloc, a, n, err)) continue;
#endif
      if (r.vec && n == 16) stg16(a, v[k]);
      else store_bytes(a, v[k], n);
    }
  }
}

__global__ void __launch_bounds__(kThreads) copy_kernel(const CopyParams p) {
  const uint64_t G = gridDim.x, b = blockIdx.x;
  const uint64_t t0 = p.ntiles * b / G, t1 = p.ntiles * (b + 1) / G;
  if (t0 < t1) {
    uint32_t ri = find_region(p.regions, p.nregions, t0);
    for (uint64_t t = t0; t < t1; ++t) {
      while (p.regions[ri + 1].tile0 <= t) ++ri;
      const CopyRegion r = p.regions[ri];
#if ASMV_DEBUG_BOUNDS
      copy_tile(r, t - r.tile0, p.err);
#else
      copy_tile(r, t - r.tile0, nullptr);
#endif
    }
  }
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = b * kWarps + (threadIdx.x >> 5), nw = G * kWarps;
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

int copy_max_ctas_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, copy_kernel, kThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    return 1;
  }
  return n > 0 ? n : 1;
}

int launch_copy(const CopyParams &p, int grid, void *stream) {
  copy_kernel<<<grid, kThreads, 0, (cudaStream_t)stream>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace asmv
