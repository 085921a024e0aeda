// plan.h -- launch descriptors shared by the host ABI layer (abi.cu) and
// the kernels (fill.cu, compare.cu).  Internal to the library.
//
// Work decomposition.  Every region's payload is cut into tiles of
// kFillTileBytes for the fill, kTileBytes for the Eq. 1 sums and the
// restore, and of a per-launch tile size for the compare (the last tile of a
// region may be short).  Tiles of all
// regions form one index space; region i owns tiles [tile0[i], tile0[i+1]).
// A launch runs a persistent grid.  In the compare and the Eq. 1 sums CTA b
// takes the contiguous tile range [T*b/G, T*(b+1)/G), so a CTA crosses few
// region boundaries and flushes its per-region partial statistics once per
// boundary; the fill, which keeps no per-region state, takes tiles b, b+G,
// b+2G, ..., so that regions of very different cost per tile spread evenly
// over the SMs.  Inside a tile, thread t handles 16-byte chunks t, t+T, ...
// for a CTA of T threads (coalesced 128-bit accesses).
//
// Guard bands are cut into segments of at most kGuardSegBytes and handled
// one warp per segment after the payload tiles.
#pragma once
#include <stdint.h>

// The debug-bounds build (compiled with ASMV_DEBUG_BOUNDS=1 into
// libasmv_debug.so) gives every region descriptor and guard segment the
// allocation it lies in, and the fill, compare and restore kernels check
// each global access against it: an access outside is skipped and sets
// kErrBounds in the launch's error word, which the call returns as
// ASMV_EBOUNDS.  The normal build carries none of it.
#ifndef ASMV_DEBUG_BOUNDS
#define ASMV_DEBUG_BOUNDS 0
#endif

namespace asmv {

constexpr uint32_t kErrTimeout = 1u;    // a bounded wait gave up
constexpr uint32_t kErrBounds = 2u;     // an access fell outside its allocation (debug-bounds build)

// [lo, hi) of one allocation (debug-bounds build).
struct Span {
  uint64_t lo, hi;
};

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kChunkBytes = 16;
constexpr int kTileChunks = 1024;
constexpr uint64_t kTileBytes = (uint64_t)kChunkBytes * kTileChunks;  // 16 KiB
constexpr uint32_t kGuardSegBytes = 4096;
constexpr int kMaxCands = 8;            // candidates per batched launch
constexpr int kConsumerWarps = 15;      // compare: checking warps per CTA (+ 1 feeding: 128 registers each)
constexpr int kStages = 4;              // compare: deepest shared-memory pipeline (2 to 4 stages per launch)
constexpr size_t kMaxSmemPerCta = 232448;   // GB300: 227 KiB of shared memory per CTA (opt-in)
constexpr int kCmpThreads = (kConsumerWarps + 1) * 32;   // + one producer warp
constexpr uint32_t kWaitRounds = 20000;  // compare: default bound of a pipeline wait, in tries

enum : uint32_t { kF32 = 0, kBF16 = 1, kF16 = 2, kF8 = 3, kI32 = 4, kI8 = 5, kU8 = 6,
                  kF8E5M2 = 7, kF8E4FNUZ = 8, kF8E5FNUZ = 9, kF64 = 10, kI16 = 11, kI64 = 12,
                  kNDtypes = 13 };

__host__ __device__ constexpr bool is_fp8(uint32_t dt) {
  return dt == kF8 || dt == kF8E5M2 || dt == kF8E4FNUZ || dt == kF8E5FNUZ;
}
__host__ __device__ constexpr bool is_float_dt(uint32_t dt) {
  return dt <= kF8 || (dt >= kF8E5M2 && dt <= kF64);
}
enum : uint32_t { kRaw = 0, kUniform = 1, kNormal = 2, kIntRange = 3, kNone = 4 };
enum : uint32_t { kSegFill = 0, kSegSelf = 1, kSegCand = 2, kSegRef = 3 };

// One region of a fill launch (64 B).
struct FillRegion {
  uint64_t payload;     // device address of element 0
  uint64_t bytes;       // payload bytes
  uint64_t tile0;       // first tile; the table has a sentinel entry after the last region
  uint32_t dtype, dist;
  uint32_t region_id;
  uint32_t vec;         // payload is 16-byte aligned
  float f0, f1;         // UNIFORM: lo, width; NORMAL: mean, std (fp32)
  int64_t ilo;          // INT_RANGE: lo
  uint64_t ispan;       // INT_RANGE: hi - lo
#if ASMV_DEBUG_BOUNDS
  Span alloc;           // the region's allocation
#endif
};

// One region of a compare launch (32 B).  Candidate payload addresses live
// in a separate [K][nregions] array.
struct CmpRegion {
  uint64_t ref;         // reference payload address
  uint64_t bytes;       // payload bytes
  uint64_t tile0;
  uint32_t dtype;
  uint32_t vec;         // reference and every candidate payload 16-byte aligned
#if ASMV_DEBUG_BOUNDS
  Span alloc;           // the reference's allocation
#endif
};

// A guard band segment (32 B).
struct GuardSeg {
  uint64_t ptr;         // first byte of the segment
  uint64_t offset;      // its offset from the allocation start
  uint32_t len;         // bytes (<= kGuardSegBytes)
  uint32_t stats;       // index into the statistics array
  uint8_t canary;
  uint8_t kind;         // kSeg*
  uint8_t pad_[6];
#if ASMV_DEBUG_BOUNDS
  Span alloc;           // the allocation the band belongs to
#endif
};

// fp32 screening thresholds and exact fp64 tolerances of one float dtype.
// alo/rlo bound atol + rtol*|r| from below, ahi/rhi from above, with a
// relative margin of 2^-21 and an absolute slack of 2^-100 (the proof of the
// screen is in compare.cu).
struct TolF {
  float alo, rlo, ahi, rhi;
  double atol, rtol;
};

// Device statistics entry; bit-compatible with asmv_stats (the two maxima
// are non-negative doubles kept as their bit patterns, so that integer
// atomicMax orders them).
struct StatsDev {
  unsigned long long mismatches, first, abs_bits, rel_bits, nonfinite;
  unsigned long long guard_bad, guard_first, ref_guard_bad;
};

// The fill runs CTAs of kFillThreads; each CTA copies into shared memory
// only the tables its launch needs, every entry replicated so that the lanes
// of a warp read distinct banks: the angle table (256 x 8 B, 16 copies) and
// the 16-bit radius chords (512 x 8 B, 8 copies) for 16-bit NORMAL, the
// angle table and the 8-bit radii (256 x 4 B, 16 copies) for 8-bit NORMAL,
// the ln reduction table (129 x 16 B, 8 copies) for fp32 and binary64
// NORMAL.  fill_layout() gives the byte offsets for a set of needs.
constexpr int kFillThreads = 512;
constexpr int kFillWarps = kFillThreads / 32;
// The fill's tiles are 64 KiB (eight chunks per thread, two at a time), so
// the per-tile work (region lookup, dispatch) is spread over more chunks.
constexpr int kFillTileChunks = 4096;
constexpr uint64_t kFillTileBytes = (uint64_t)kChunkBytes * kFillTileChunks;
enum : uint32_t { kNeedN16 = 1, kNeedN8 = 2, kNeedLn = 4 };
constexpr uint32_t kAngleCopies = 16, kRad16Copies = 8, kRad8Copies = 16, kLnCopies = 8;
constexpr uint32_t kNoTable = 0xFFFFFFFFu;
constexpr uint32_t kAngleBytes = 256 * 8 * kAngleCopies;     // 32 KiB
constexpr uint32_t kRad16Bytes = 512 * 8 * kRad16Copies;     // 32 KiB
constexpr uint32_t kRad8Bytes = 256 * 4 * kRad8Copies;       // 16 KiB
constexpr uint32_t kLnBytes = 129 * 16 * kLnCopies;          // 16.1 KiB

struct FillLayout {
  uint32_t angle, rad16, rad8, ln;   // byte offsets in shared memory, kNoTable if absent
  uint32_t bytes;                    // dynamic shared memory of the launch
};

inline FillLayout fill_layout(uint32_t needs) {
  FillLayout L = {kNoTable, kNoTable, kNoTable, kNoTable, 0};
  if (needs & (kNeedN16 | kNeedN8)) { L.angle = L.bytes; L.bytes += kAngleBytes; }
  if (needs & kNeedN16) { L.rad16 = L.bytes; L.bytes += kRad16Bytes; }
  if (needs & kNeedN8) { L.rad8 = L.bytes; L.bytes += kRad8Bytes; }
  if (needs & kNeedLn) { L.ln = L.bytes; L.bytes += kLnBytes; }
  return L;
}

struct FillParams {
  const FillRegion *regions;   // nregions + 1 entries (sentinel)
  const GuardSeg *segs;
  uint64_t ntiles;
  uint64_t seed;
  uint32_t nregions;
  uint32_t nsegs;
  FillLayout smem;             // the tables in shared memory
  // Philox key of each of the 10 rounds: (seed lo, seed hi) advanced by the
  // Weyl increments, precomputed on the host (kernel-parameter operands)
  uint32_t key0[10], key1[10];
#if ASMV_DEBUG_BOUNDS
  uint32_t *err;               // kErrBounds
#endif
};

struct CmpParams {
  const CmpRegion *regions;    // nregions + 1 entries (sentinel)
  const uint64_t *cands;       // [K][nregions] candidate payload addresses
  const GuardSeg *segs;
  StatsDev *stats;             // [K][nregions] (this launch's candidates)
  StatsDev *seg_stats;         // guard segments index from here
  uint32_t *err;               // kErrTimeout when a bounded wait expires (kErrBounds)
  uint64_t ntiles;
  uint32_t nregions;
  uint32_t nsegs;
  uint32_t K;
  uint32_t tile_bytes;         // payload bytes per tile (multiple of 16)
  uint32_t wait_rounds;        // bound of the producer's wait for a free stage (tries)
  uint32_t nstages;            // pipeline depth of this launch: 2, 3 or 4 (compare_stages)
  TolF tol[kNDtypes];
#if ASMV_DEBUG_BOUNDS
  const Span *cand_allocs;     // [K][nregions] the candidates' allocations
#endif
};

// The Eq. 1 sums (eqsum.cu).  Each sum of a region is kept as kEqDigits
// signed 64-bit digits, digit k weighing 2^(32k + eq_digit_base(dtype)); the
// digits of one region are [slot][kEqDigits] with slot 0 = S_rr and slots
// 1 + 2j, 2 + 2j = S_rc, S_cc of candidate j -- or, for the formats of
// eq_difference_form, sum r d and sum d^2 with d = c - r, from which
// S_rc = S_rr + sum r d and S_cc = S_rr + 2 sum r d + sum d^2.
constexpr int kEqDigits = 20;
// fp8 formats other than E4M3 are summed through their exact fp16 value.
constexpr int eq_digit_base(uint32_t dtype) {
  return dtype == kF32 ? -318 : dtype == kBF16 ? -286 : dtype == kF8 ? -82 : -112;
}

constexpr bool eq_difference_form(uint32_t dtype) {
  return dtype == kF16 || dtype == kF8E5M2 || dtype == kF8E4FNUZ || dtype == kF8E5FNUZ;
}

struct EqParams {
  const CmpRegion *regions;    // nregions + 1 entries (sentinel); bytes = 0 for non-float
  const uint64_t *cands;       // [K][nregions] candidate payload addresses (this launch)
  long long *digits;           // [nregions][nslots][kEqDigits]
  uint64_t ntiles;             // tiles of kTileBytes
  uint32_t nregions;
  uint32_t K;                  // candidates in this launch (<= kMaxCands)
  uint32_t j0;                 // index of this launch's first candidate
  uint32_t nslots;             // 1 + 2 * (all candidates)
  uint32_t do_rr;              // this launch also adds S_rr
};

// One region of a restore or capture launch (48 B): move `bytes` from src to
// dst; the table has a sentinel entry after the last region.
struct CopyRegion {
  uint64_t dst, src, bytes, tile0;
  uint32_t vec;         // src and dst both 16-byte aligned
  uint32_t pad_[3];
#if ASMV_DEBUG_BOUNDS
  Span dst_alloc, src_alloc;   // the allocations written and read
#endif
};

struct CopyParams {
  const CopyRegion *regions;   // nregions + 1 entries
  const GuardSeg *segs;        // guard bands to rewrite with the canary (restore only)
  uint64_t ntiles;             // tiles of kTileBytes
  uint32_t nregions;
  uint32_t nsegs;
#if ASMV_DEBUG_BOUNDS
  uint32_t *err;               // kErrBounds
#endif
};

// Launchers (defined in fill.cu / compare.cu / eqsum.cu / copy.cu).  Return a cudaError_t.
int launch_fill(const FillParams &p, int grid, void *stream);
int launch_compare(const CmpParams &p, int grid, void *stream);
int fill_max_ctas_per_sm(uint32_t smem_bytes);
uint32_t compare_tile_bytes(uint32_t K);
uint32_t compare_stages(uint32_t K, uint32_t tile_bytes);
size_t compare_smem_bytes(uint32_t K, uint32_t tile_bytes, uint32_t nstages);
int launch_eq(const EqParams &p, int grid, void *stream);
int eq_max_ctas_per_sm();
int launch_copy(const CopyParams &p, int grid, void *stream);
int copy_max_ctas_per_sm();

}  // namespace asmv
