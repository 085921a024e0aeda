// eq64.h -- launch descriptor of the Eq. 1 sums of binary64 regions
// (eq64.cu).  Internal to the library.
#pragma once
#include <stdint.h>
#include "plan.h"

namespace asmv {

// A binary64 product is +-M 2^E with M < 2^106 and -2148 <= E; its
// magnitude is below 2^2048.  Each sum is kept as kEq64Digits signed 64-bit
// digits, digit k weighing 2^(32k + kEq64Base): 2^-2148 .. 2^2048 and 2^64
// of headroom take 134 digits.
constexpr int kEq64Digits = 136;
constexpr int kEq64Base = -2148;
constexpr uint64_t kEq64TileBytes = 16384;     // 2048 values per tile

struct Eq64Params {
  const CmpRegion *regions;    // the binary64 regions, + a sentinel; tiles of kEq64TileBytes
  const uint64_t *cands;       // [K][nregions] candidate payload addresses (this launch)
  long long *digits;           // [nregions][nslots][kEq64Digits]
  uint64_t ntiles;
  uint32_t nregions;
  uint32_t K;                  // candidates in this launch (<= kMaxCands)
  uint32_t j0;                 // index of this launch's first candidate
  uint32_t nslots;             // 1 + 2 * (all candidates): S_rr, then S_rc and S_cc of each
  uint32_t do_rr;              // this launch also adds S_rr
};

int launch_eq64(const Eq64Params &p, int grid, void *stream);
int eq64_max_ctas_per_sm();

}  // namespace asmv
