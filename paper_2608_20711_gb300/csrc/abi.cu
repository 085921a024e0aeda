// abi.cu -- the C ABI of include/asmv.h: argument validation, device-memory
// checks, launch-plan packing, workspace management and result readback.
//
// Each call packs its plan (region descriptors with tile prefixes, candidate
// addresses, guard segments, initial statistics) into pinned staging,
// copies it to the context's device workspace with one asynchronous copy,
// launches the kernel(s) on the caller's stream and, for the checking
// calls, copies the statistics back and synchronises the stream.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <utility>
#include <vector>

#include <cuda_runtime.h>

#include "asmv.h"
#include "plan.h"
#include "eq64.h"
#include "nvtx_range.h"

using namespace asmv;

static_assert(sizeof(asmv_region) == 56, "asmv_region layout");
static_assert(sizeof(asmv_stats) == 64, "asmv_stats layout");
static_assert(sizeof(asmv_eq) == 40, "asmv_eq layout");
static_assert(sizeof(StatsDev) == sizeof(asmv_stats), "device statistics layout");
static_assert(sizeof(CopyRegion) == 48 + (ASMV_DEBUG_BOUNDS ? 32 : 0), "copy region layout");
static_assert(kWaitRounds == ASMV_WAIT_ROUNDS, "default wait bound");
static_assert(kEqDigits == ASMV_EQ_DIGITS, "Eq. 1 digits");
static_assert(kEq64Digits == ASMV_EQ64_DIGITS, "Eq. 1 digits of binary64");
static_assert(sizeof(FillRegion) == 64 + (ASMV_DEBUG_BOUNDS ? 16 : 0) &&
                  sizeof(CmpRegion) == 32 + (ASMV_DEBUG_BOUNDS ? 16 : 0) &&
                  sizeof(GuardSeg) == 32 + (ASMV_DEBUG_BOUNDS ? 16 : 0),
              "plan layouts");

namespace {

typedef int (*AddrRangeFn)(unsigned long long *base, size_t *size, unsigned long long ptr);

const int kDtypeSize[ASMV_NDTYPES] = {4, 2, 2, 1, 4, 1, 1, 1, 1, 1, 8, 2, 8};
static_assert(ASMV_NDTYPES == kNDtypes && ASMV_F64 == kF64 && ASMV_I64 == kI64, "dtype codes");

bool is_float(uint32_t dt) { return dt < ASMV_NDTYPES && is_float_dt(dt); }

// ------------------------------------------------------------ validation
bool region_extent(const asmv_region &r, uint64_t *payload_bytes, uint64_t *total) {
  if (r.dtype >= ASMV_NDTYPES) return false;
  const uint64_t sz = (uint64_t)kDtypeSize[r.dtype];
  if (r.n_elems > UINT64_MAX / sz) return false;
  const uint64_t pb = r.n_elems * sz;
  const uint64_t t = pb + (uint64_t)r.guard_lo;
  if (t < pb || t + (uint64_t)r.guard_hi < t) return false;
  const uint64_t tot = t + (uint64_t)r.guard_hi;
  if (tot > 0 && r.alloc == 0) return false;
  if (r.alloc + tot < r.alloc) return false;
  *payload_bytes = pb;
  *total = tot;
  return true;
}

bool fits_f32(double x) { return std::isfinite(x) && std::fabs(x) <= (double)3.4028234663852886e38; }

bool dist_ok(const asmv_region &r) {
  switch (r.dist) {
    case ASMV_DIST_RAW:
    case ASMV_DIST_NONE:
      return true;
    case ASMV_DIST_UNIFORM: {
      if (!is_float(r.dtype) || !fits_f32(r.p0) || !fits_f32(r.p1) || !(r.p0 <= r.p1)) return false;
      const float w = (float)r.p1 - (float)r.p0;
      return std::isfinite(w);
    }
    case ASMV_DIST_NORMAL: {
      if (!is_float(r.dtype) || !fits_f32(r.p0) || !fits_f32(r.p1) || !(r.p1 >= 0.0)) return false;
      // |mean| + 6 std bounds mean + std*z (|z| <= 5.8) away from fp32 overflow
      return std::fabs((double)(float)r.p0) + 6.0 * (double)(float)r.p1 <= 3.4e38;
    }
    case ASMV_DIST_INT_RANGE: {
      if (is_float(r.dtype)) return false;
      if (!std::isfinite(r.p0) || !std::isfinite(r.p1)) return false;
      if (r.p0 != std::floor(r.p0) || r.p1 != std::floor(r.p1) || !(r.p0 < r.p1)) return false;
      double lo_lim, hi_lim;
      if (r.dtype == ASMV_I32) { lo_lim = -2147483648.0; hi_lim = 2147483648.0; }
      else if (r.dtype == ASMV_I8) { lo_lim = -128.0; hi_lim = 128.0; }
      else if (r.dtype == ASMV_I16) { lo_lim = -32768.0; hi_lim = 32768.0; }
      else if (r.dtype == ASMV_I64) { lo_lim = -9007199254740992.0; hi_lim = 9007199254740992.0; }
      else { lo_lim = 0.0; hi_lim = 256.0; }
      return r.p0 >= lo_lim && r.p1 <= hi_lim && (r.p1 - r.p0) <= 4294967296.0;
    }
    default:
      return false;
  }
}

int check_table(const asmv_region *regs, size_t n, bool for_fill) {
  if (n > 0 && regs == nullptr) return ASMV_EINVAL;
  if (n > (size_t)0x7FFFFFFF) return ASMV_EINVAL;
  std::vector<std::pair<uint64_t, uint64_t>> spans;
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    if (!region_extent(regs[i], &pb, &tot)) return ASMV_EINVAL;
    if (for_fill) {
      if (!dist_ok(regs[i])) return ASMV_EINVAL;
      if (tot > 0) spans.emplace_back(regs[i].alloc, regs[i].alloc + tot);
    }
  }
  if (for_fill && spans.size() > 1) {
    std::sort(spans.begin(), spans.end());
    for (size_t i = 1; i < spans.size(); ++i)
      if (spans[i].first < spans[i - 1].second) return ASMV_EINVAL;
  }
  return ASMV_OK;
}

bool tol_ok(const asmv_tol *tol) {
  if (tol == nullptr) return false;
  for (int d = 0; d < ASMV_NDTYPES; ++d) {
    if (!is_float((uint32_t)d)) continue;
    if (std::isnan(tol[d].atol) || std::isnan(tol[d].rtol)) return false;
    if (tol[d].atol < 0.0 || tol[d].rtol < 0.0) return false;
  }
  return true;
}

float round_down_f32(double x) {
  float f = (float)x;
  if ((double)f > x) f = std::nextafter(f, -INFINITY);
  return f;
}
float round_up_f32(double x) {
  float f = (float)x;
  if ((double)f < x) f = std::nextafter(f, INFINITY);
  return f;
}

// fp32 screen thresholds bracketing atol + rtol*|r| (see compare.cu).
TolF make_tolf(const asmv_tol &t) {
  TolF f;
  const double lo_scale = 1.0 - 0x1p-21, hi_scale = 1.0 + 0x1p-21;
  f.alo = (t.atol >= 0x1p-100) ? round_down_f32(t.atol * lo_scale) : -0x1p-100f;
  f.rlo = round_down_f32(t.rtol * lo_scale);
  f.ahi = round_up_f32(t.atol * hi_scale + 0x1p-100);
  f.rhi = round_up_f32(t.rtol * hi_scale);
  f.atol = t.atol;
  f.rtol = t.rtol;
  return f;
}

uint64_t tiles_of(uint64_t payload_bytes) { return (payload_bytes + kTileBytes - 1) / kTileBytes; }

void add_guard_segments(std::vector<GuardSeg> &segs, uint64_t ptr, uint64_t offset, uint64_t len,
                        uint8_t canary, uint8_t kind, uint32_t stats, uint64_t alloc, uint64_t total) {
  for (uint64_t o = 0; o < len; o += kGuardSegBytes) {
    GuardSeg g;
    std::memset(&g, 0, sizeof g);
    g.ptr = ptr + o;
    g.offset = offset + o;
    g.len = (uint32_t)std::min<uint64_t>(kGuardSegBytes, len - o);
    g.stats = stats;
    g.canary = canary;
    g.kind = kind;
#if ASMV_DEBUG_BOUNDS
    g.alloc = Span{alloc, alloc + total};
#else
    (void)alloc; (void)total;
#endif
    segs.push_back(g);
  }
}

void add_region_guards(std::vector<GuardSeg> &segs, const asmv_region &r, uint8_t kind, uint32_t stats) {
  uint64_t pb, tot;
  region_extent(r, &pb, &tot);
  if (r.guard_lo) add_guard_segments(segs, r.alloc, 0, r.guard_lo, r.canary, kind, stats, r.alloc, tot);
  if (r.guard_hi)
    add_guard_segments(segs, r.alloc + r.guard_lo + pb, (uint64_t)r.guard_lo + pb, r.guard_hi,
                       r.canary, kind, stats, r.alloc, tot);
}

StatsDev empty_stats() {
  StatsDev s;
  s.mismatches = 0; s.first = ~0ull; s.abs_bits = 0; s.rel_bits = 0; s.nonfinite = 0;
  s.guard_bad = 0; s.guard_first = ~0ull; s.ref_guard_bad = 0;
  return s;
}

// Packs sections into one byte image with 256-byte aligned offsets.
struct Image {
  std::vector<unsigned char> bytes;
  size_t add(const void *p, size_t n) {
    const size_t off = (bytes.size() + 255) & ~(size_t)255;
    bytes.resize(off + n);
    if (n) std::memcpy(bytes.data() + off, p, n);
    return off;
  }
};

struct DeviceScope {
  int prev = -1;
  bool ok = false;
  explicit DeviceScope(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceScope() { if (prev >= 0) cudaSetDevice(prev); }
};

}  // namespace

struct asmv_ctx {
  int device = 0;
  int sms = 0;
  int fill_ctas[8] = {0, 0, 0, 0, 0, 0, 0, 0};   // per set of fill tables (kNeed* mask)
  int eq_ctas = 1;
  int eq64_ctas = 1;
  int copy_ctas = 1;
  void *dws = nullptr;
  size_t dws_cap = 0;
  unsigned char *hst = nullptr;
  size_t hst_cap = 0;
  cudaEvent_t staged = nullptr;   // previous upload of the staging buffer finished
  cudaEvent_t ws_done = nullptr;  // previous kernel using the workspace finished
  bool staged_pending = false, ws_pending = false;
  int timing = 0;
  bool timed = false;
  cudaEvent_t t0 = nullptr, t1 = nullptr;
  int cuda_err = 0;
  uint64_t launches = 0;
  uint32_t wait_rounds = kWaitRounds;
  AddrRangeFn addr_range = nullptr;
  uint64_t debug_widen = 0;       // debug-bounds build: bytes added to each fill's loop bound
  int sm_limit = 0;               // SMs a launch may occupy (0: all of them)
};

namespace {

int fail_cuda(asmv_ctx *ctx, cudaError_t e) {
  ctx->cuda_err = (int)e;
  return (e == cudaErrorMemoryAllocation) ? ASMV_ENOMEM : ASMV_ECUDA;
}

// Every byte [alloc, alloc+total) must be device memory of ctx's device
// inside one allocation.  `last` caches the most recent allocation range.
int check_device_span(asmv_ctx *ctx, uint64_t alloc, uint64_t total,
                      std::pair<uint64_t, uint64_t> &last) {
  if (total == 0) return ASMV_OK;
  if (alloc >= last.first && alloc + total <= last.second) return ASMV_OK;
  cudaPointerAttributes a;
  cudaError_t e = cudaPointerGetAttributes(&a, (const void *)alloc);
  if (e != cudaSuccess) { cudaGetLastError(); return ASMV_EINVAL; }
  if (a.type == cudaMemoryTypeDevice) {
    if (a.device != ctx->device) return ASMV_EINVAL;
  } else if (a.type != cudaMemoryTypeManaged) {
    return ASMV_EINVAL;                              // host or unregistered memory
  }
  if (ctx->addr_range) {
    unsigned long long base = 0;
    size_t size = 0;
    if (ctx->addr_range(&base, &size, alloc) != 0) return ASMV_EINVAL;
    if (alloc + total > base + size) return ASMV_EINVAL;
    last = std::make_pair((uint64_t)base, (uint64_t)(base + size));
  }
  return ASMV_OK;
}

int check_device_table(asmv_ctx *ctx, const asmv_region *regs, size_t n,
                       std::pair<uint64_t, uint64_t> &last) {
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    region_extent(regs[i], &pb, &tot);
    const int rc = check_device_span(ctx, regs[i].alloc, tot, last);
    if (rc != ASMV_OK) return rc;
  }
  return ASMV_OK;
}

// Upload `img` (and reserve `readback` bytes of staging after it) to the
// workspace on `s`; returns the device base in *dev.  `dev_extra` more
// bytes of workspace follow the image (at its size rounded up to 256),
// uninitialised.
int stage(asmv_ctx *ctx, const Image &img, size_t readback, cudaStream_t s, unsigned char **dev,
          size_t dev_extra = 0) {
  const size_t need_dev = std::max<size_t>(((img.bytes.size() + 255) & ~(size_t)255) + dev_extra, 256);
  const size_t need_host = ((img.bytes.size() + 255) & ~(size_t)255) + readback;
  cudaError_t e;
  if (ctx->staged_pending) {
    if ((e = cudaEventSynchronize(ctx->staged)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->staged_pending = false;
  }
  if (need_host > ctx->hst_cap) {
    const size_t cap = std::max(need_host, std::max((size_t)1 << 20, ctx->hst_cap * 2));
    if (ctx->hst) cudaFreeHost(ctx->hst);
    ctx->hst = nullptr;
    ctx->hst_cap = 0;
    if ((e = cudaHostAlloc((void **)&ctx->hst, cap, cudaHostAllocDefault)) != cudaSuccess) {
      ctx->hst = nullptr;
      fail_cuda(ctx, e);
      return ASMV_ENOMEM;
    }
    ctx->hst_cap = cap;
  }
  if (need_dev > ctx->dws_cap) {
    if (ctx->ws_pending) {
      if ((e = cudaEventSynchronize(ctx->ws_done)) != cudaSuccess) return fail_cuda(ctx, e);
      ctx->ws_pending = false;
    }
    const size_t cap = std::max(need_dev, std::max((size_t)1 << 20, ctx->dws_cap * 2));
    if (ctx->dws) cudaFree(ctx->dws);
    ctx->dws = nullptr;
    ctx->dws_cap = 0;
    if ((e = cudaMalloc(&ctx->dws, cap)) != cudaSuccess) {
      ctx->dws = nullptr;
      fail_cuda(ctx, e);
      return ASMV_ENOMEM;
    }
    ctx->dws_cap = cap;
  }
  if (ctx->ws_pending && (e = cudaStreamWaitEvent(s, ctx->ws_done, 0)) != cudaSuccess)
    return fail_cuda(ctx, e);
  std::memcpy(ctx->hst, img.bytes.data(), img.bytes.size());
  if ((e = cudaMemcpyAsync(ctx->dws, ctx->hst, img.bytes.size(), cudaMemcpyHostToDevice, s)) !=
      cudaSuccess)
    return fail_cuda(ctx, e);
  if ((e = cudaEventRecord(ctx->staged, s)) != cudaSuccess) return fail_cuda(ctx, e);
  ctx->staged_pending = true;
  *dev = (unsigned char *)ctx->dws;
  return ASMV_OK;
}

int after_launch(asmv_ctx *ctx, cudaStream_t s) {
  cudaError_t e;
  if ((e = cudaEventRecord(ctx->ws_done, s)) != cudaSuccess) return fail_cuda(ctx, e);
  ctx->ws_pending = true;
  return ASMV_OK;
}

// Host staging a call reserves for reading back its launch's error word:
// only the debug-bounds build has one for the fill and the restore.
constexpr size_t debug_err_bytes() { return ASMV_DEBUG_BOUNDS ? 256 : 0; }

#if ASMV_DEBUG_BOUNDS
// The debug-bounds build finishes a fill or restore by reading its error
// word back (the call then synchronises its stream): ASMV_EBOUNDS if an
// access fell outside its allocation.
int debug_finish(asmv_ctx *ctx, size_t err_off, size_t img_bytes, cudaStream_t s) {
  cudaError_t e;
  unsigned char *host = ctx->hst + ((img_bytes + 255) & ~(size_t)255);
  if ((e = cudaMemcpyAsync(host, (unsigned char *)ctx->dws + err_off, sizeof(uint32_t),
                           cudaMemcpyDeviceToHost, s)) != cudaSuccess)
    return fail_cuda(ctx, e);
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return fail_cuda(ctx, e);
  ctx->staged_pending = false;
  ctx->ws_pending = false;
  uint32_t err;
  std::memcpy(&err, host, sizeof err);
  return (err & kErrBounds) ? ASMV_EBOUNDS : ASMV_OK;
}
#endif

// The SMs a launch of ctx may occupy: all of the device's, or the limit
// set with asmv_ctx_set_sm_limit.
uint64_t sms_of(const asmv_ctx *ctx) {
  return (uint64_t)((ctx->sm_limit > 0 && ctx->sm_limit < ctx->sms) ? ctx->sm_limit : ctx->sms);
}

int grid_for(asmv_ctx *ctx, uint64_t ntiles, size_t nsegs, int ctas_per_sm) {
  const uint64_t cap = sms_of(ctx) * (uint64_t)ctas_per_sm;
  uint64_t g = std::max<uint64_t>(ntiles, (nsegs + kWarps - 1) / kWarps);
  g = std::min<uint64_t>(g, cap);
  return (int)std::max<uint64_t>(g, 1);
}

// Read back k*n statistics from the workspace and finish the call.
int readback(asmv_ctx *ctx, size_t stats_off, size_t img_bytes, size_t count, cudaStream_t s,
             asmv_stats *out, size_t ref_n) {
  cudaError_t e;
  unsigned char *host = ctx->hst + ((img_bytes + 255) & ~(size_t)255);
  if ((e = cudaMemcpyAsync(host, (unsigned char *)ctx->dws + stats_off,
                           (count + 1) * sizeof(StatsDev), cudaMemcpyDeviceToHost, s)) != cudaSuccess)
    return fail_cuda(ctx, e);
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return fail_cuda(ctx, e);
  ctx->staged_pending = false;
  ctx->ws_pending = false;
  uint32_t err;
  std::memcpy(&err, host + count * sizeof(StatsDev), sizeof err);
  if (err & kErrBounds) return ASMV_EBOUNDS;         // an access outside its allocation (debug build)
  if (err) return ASMV_ETIMEOUT;                     // a bounded device wait expired
  std::memcpy(out, host, count * sizeof(asmv_stats));
  if (ref_n) {
    // reference-guard damage was accumulated in the first candidate's entries
    for (size_t j = 1; j < count / ref_n; ++j)
      for (size_t i = 0; i < ref_n; ++i) out[j * ref_n + i].ref_guard_bad_bytes = out[i].ref_guard_bad_bytes;
  }
  return ASMV_OK;
}

// The magnitude and sign of the integer sum_k d[k] 2^(32k): the digits are
// carried into nd + 2 limbs of 32 bits in two's complement, and negated when
// the top carry says the value is negative.  msb is the position of the
// leading one bit, -1 for zero.
constexpr int kMaxExactDigits = kEq64Digits;
struct Magnitude {
  uint32_t L[kMaxExactDigits + 2];
  int nl;
  int msb;
  bool neg;
  uint64_t bit(int pos) const {
    return (pos < 0 || pos >= 32 * nl) ? 0u : (uint64_t)((L[pos >> 5] >> (pos & 31)) & 1u);
  }
  bool any_below(int pos) const {                 // some bit at a position < pos is set
    if (pos <= 0) return false;
    const int lim = std::min(pos >> 5, nl);
    for (int k = 0; k < lim; ++k)
      if (L[k] != 0) return true;
    if (lim == nl || (pos & 31) == 0) return false;
    return (L[lim] & ((1u << (pos & 31)) - 1u)) != 0;
  }
};

void magnitude_of(const int64_t *d, int nd, Magnitude *m) {
  m->nl = nd + 2;
  __int128 c = 0;
  for (int k = 0; k < m->nl; ++k) {
    const __int128 x = c + (k < nd ? (__int128)d[k] : (__int128)0);
    m->L[k] = (uint32_t)(x & 0xFFFFFFFF);
    c = x >> 32;                                   // floor: arithmetic shift
  }
  m->neg = c < 0;                                  // c is 0 or -1 here
  if (m->neg) {
    uint64_t carry = 1;
    for (int k = 0; k < m->nl; ++k) {
      const uint64_t x = (uint64_t)(uint32_t)~m->L[k] + carry;
      m->L[k] = (uint32_t)x;
      carry = x >> 32;
    }
  }
  int top = m->nl - 1;
  while (top >= 0 && m->L[top] == 0) --top;
  m->msb = -1;
  if (top >= 0) {
    m->msb = 32 * top;
    for (uint32_t v = m->L[top]; v > 1; v >>= 1) ++m->msb;
  }
}

// |value| 2^scale rounded to the nearest double, ties to even, with gradual
// underflow (the last kept bit weighs at least 2^-1074) and overflow to
// infinity; the sign is not applied.
double round_magnitude(const Magnitude &m, int scale) {
  if (m.msb < 0) return 0.0;
  if (m.msb + scale >= 1024) return INFINITY;
  const int last = std::max(m.msb - 52, -1074 - scale);   // position of the last kept bit
  uint64_t keep = 0;
  for (int pos = m.msb; pos >= last; --pos) keep = (keep << 1) | m.bit(pos);
  const bool half = m.bit(last - 1) != 0;
  const bool sticky = m.any_below(last - 1);
  if (half && (sticky || (keep & 1u))) keep += 1;
  return std::ldexp((double)keep, last + scale);   // exact; 2^1024 becomes infinity
}

// The integer sum_k d[k] 2^(32k + base) rounded to the nearest double (ties
// to even); EINVAL when the value lies outside the normal double range.
int exact_to_double_impl(const int64_t *d, int nd, int base, double *out) {
  if (d == nullptr || out == nullptr || nd < 1 || nd > 64) return ASMV_EINVAL;
  Magnitude m;
  magnitude_of(d, nd, &m);
  if (m.msb < 0) { *out = 0.0; return ASMV_OK; }
  if (m.msb + base < -1022 || m.msb + base >= 1024) return ASMV_EINVAL;
  const double v = round_magnitude(m, base);
  *out = m.neg ? -v : v;
  return ASMV_OK;
}

// c_x of a binary64 region from its exact sums (value = magnitude 2^base):
// S_rr and S_cc scaled by 2^-2p and 2^-2q into [1, 4) and S_rc by
// 2^-(p+q) before rounding, so no sum overflows or underflows, and the
// cosine of the scaled sums is the cosine of the sums.
double eq_cosine_scaled(const Magnitude &rc, const Magnitude &rr, const Magnitude &cc, int base) {
  if (rr.msb < 0 && cc.msb < 0) return 1.0;
  if (rr.msb < 0 || cc.msb < 0) return 0.0;
  auto half_floor = [](int v) { return v >= 0 ? v / 2 : -((1 - v) / 2); };
  const int p = half_floor(rr.msb + base), q = half_floor(cc.msb + base);
  double x = round_magnitude(rc, base - p - q);
  if (rc.neg) x = -x;
  const double y = round_magnitude(rr, base - 2 * p), z = round_magnitude(cc, base - 2 * q);
  return x / (std::sqrt(y) * std::sqrt(z));
}

double eq_cosine(double rc, double rr, double cc) {
  if (rr == 0.0 && cc == 0.0) return 1.0;
  if (rr == 0.0 || cc == 0.0) return 0.0;
  return rc / (std::sqrt(rr) * std::sqrt(cc));
}

}  // namespace

// ====================================================================== ABI
extern "C" {

int asmv_abi_version(void) { return ASMV_ABI_VERSION; }

const char *asmv_strerror(int status) {
  switch (status) {
    case ASMV_OK: return "ok";
    case ASMV_EINVAL: return "invalid argument or region table";
    case ASMV_ECUDA: return "CUDA runtime error";
    case ASMV_ETIMEOUT: return "bounded device wait expired";
    case ASMV_ENOMEM: return "out of memory (workspace or staging)";
    case ASMV_EBOUNDS: return "a device access fell outside its allocation (debug-bounds build)";
    default: return "unknown status";
  }
}

int asmv_check_regions(const asmv_region *regions, size_t n, int for_fill) {
  return check_table(regions, n, for_fill != 0);
}

// The order in which asmv_fill lays out a table's tiles: the regions grouped
// by the code that fills them (distribution, then dtype; RAW of any dtype is
// one kind), in table order within a kind.  The kernel's CTAs take tiles
// round robin, so a CTA then runs one kind for many tiles in a row instead of
// switching code, and the instruction cache, almost at every tile.  No byte
// depends on the order: a region's Philox stream is addressed by its id and
// its own chunk index.
static void fill_order(const asmv_region *regions, size_t n, uint32_t *ord) {
  for (size_t i = 0; i < n; ++i) ord[i] = (uint32_t)i;
  const auto kind = [&](uint32_t i) {
    const asmv_region &r = regions[i];
    return r.dist * 64u + (r.dist == ASMV_DIST_RAW ? 0u : r.dtype);
  };
  std::stable_sort(ord, ord + n, [&](uint32_t a, uint32_t b) { return kind(a) < kind(b); });
}

int asmv_fill_order(const asmv_region *regions, size_t n, uint32_t *order) {
  if (n != 0 && order == nullptr) return ASMV_EINVAL;
  const int rc = check_table(regions, n, true);
  if (rc != ASMV_OK) return rc;
  fill_order(regions, n, order);
  return ASMV_OK;
}

int asmv_ctx_create(asmv_ctx **out, int device) {
  if (out == nullptr) return ASMV_EINVAL;
  *out = nullptr;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess) { cudaGetLastError(); return ASMV_ECUDA; }
  if (device < 0 || device >= ndev) return ASMV_EINVAL;
  asmv_ctx *ctx = new (std::nothrow) asmv_ctx();
  if (!ctx) return ASMV_ENOMEM;
  ctx->device = device;
  DeviceScope ds(device);
  cudaError_t e = cudaSuccess;
  if (!ds.ok) e = cudaErrorInvalidDevice;
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, device);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->staged, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ws_done, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreate(&ctx->t0);
  if (e == cudaSuccess) e = cudaEventCreate(&ctx->t1);
  if (e != cudaSuccess) {
    asmv_ctx_destroy(ctx);
    return ASMV_ECUDA;
  }
  for (uint32_t m = 0; m < 8 && e == cudaSuccess; ++m) {
    ctx->fill_ctas[m] = fill_max_ctas_per_sm(fill_layout(m).bytes);
    if (ctx->fill_ctas[m] <= 0) e = cudaErrorInvalidConfiguration;
  }
  if (e != cudaSuccess) {
    asmv_ctx_destroy(ctx);
    return ASMV_ECUDA;
  }
  ctx->eq_ctas = eq_max_ctas_per_sm();
  ctx->eq64_ctas = eq64_max_ctas_per_sm();
  ctx->copy_ctas = copy_max_ctas_per_sm();
  void *fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &fn, 12000, cudaEnableDefault, &q) ==
          cudaSuccess && q == cudaDriverEntryPointSuccess)
    ctx->addr_range = (AddrRangeFn)fn;
  else
    cudaGetLastError();
  *out = ctx;
  return ASMV_OK;
}

void asmv_ctx_destroy(asmv_ctx *ctx) {
  if (ctx == nullptr) return;
  DeviceScope ds(ctx->device);
  if (ctx->ws_pending) cudaEventSynchronize(ctx->ws_done);
  if (ctx->staged_pending) cudaEventSynchronize(ctx->staged);
  if (ctx->dws) cudaFree(ctx->dws);
  if (ctx->hst) cudaFreeHost(ctx->hst);
  if (ctx->staged) cudaEventDestroy(ctx->staged);
  if (ctx->ws_done) cudaEventDestroy(ctx->ws_done);
  if (ctx->t0) cudaEventDestroy(ctx->t0);
  if (ctx->t1) cudaEventDestroy(ctx->t1);
  delete ctx;
}

int asmv_ctx_set_timing(asmv_ctx *ctx, int enable) {
  if (ctx == nullptr) return ASMV_EINVAL;
  ctx->timing = enable != 0;
  ctx->timed = false;
  return ASMV_OK;
}

int asmv_ctx_kernel_ms(asmv_ctx *ctx, float *ms) {
  if (ctx == nullptr || ms == nullptr || !ctx->timing || !ctx->timed) return ASMV_EINVAL;
  DeviceScope ds(ctx->device);
  cudaError_t e = cudaEventSynchronize(ctx->t1);
  if (e == cudaSuccess) e = cudaEventElapsedTime(ms, ctx->t0, ctx->t1);
  return e == cudaSuccess ? ASMV_OK : fail_cuda(ctx, e);
}

int asmv_ctx_cuda_error(const asmv_ctx *ctx) { return ctx ? ctx->cuda_err : 0; }

uint64_t asmv_ctx_launches(const asmv_ctx *ctx) { return ctx ? ctx->launches : 0; }

int asmv_ctx_set_wait_rounds(asmv_ctx *ctx, uint32_t rounds) {
  if (ctx == nullptr) return ASMV_EINVAL;
  ctx->wait_rounds = rounds;
  return ASMV_OK;
}

int asmv_ctx_set_sm_limit(asmv_ctx *ctx, int sms) {
  if (ctx == nullptr || sms < 0) return ASMV_EINVAL;
  ctx->sm_limit = sms;
  return ASMV_OK;
}

int asmv_debug_bounds(void) { return ASMV_DEBUG_BOUNDS; }

int asmv_ctx_debug_widen(asmv_ctx *ctx, uint64_t bytes) {
  if (ctx == nullptr || !ASMV_DEBUG_BOUNDS) return ASMV_EINVAL;
  ctx->debug_widen = bytes;
  return ASMV_OK;
}

int asmv_fill(asmv_ctx *ctx, const asmv_region *regions, size_t n, uint64_t seed,
              asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_fill");
  if (ctx == nullptr) return ASMV_EINVAL;
  int rc = check_table(regions, n, true);
  if (rc != ASMV_OK) return rc;
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  std::pair<uint64_t, uint64_t> last(0, 0);
  if ((rc = check_device_table(ctx, regions, n, last)) != ASMV_OK) return rc;

  std::vector<uint32_t> ord(n);              // the tiles' region order (fill_order)
  fill_order(regions, n, ord.data());
  std::vector<FillRegion> fr(n + 1);
  std::vector<GuardSeg> segs;
  uint64_t tile = 0;
  uint32_t needs = 0;   // the shared-memory tables the launch's NORMAL regions use
  for (size_t j = 0; j < n; ++j) {
    const size_t i = ord[j];
    const asmv_region &r = regions[i];
    uint64_t pb, tot;
    region_extent(r, &pb, &tot);
    FillRegion &f = fr[j];
    std::memset(&f, 0, sizeof f);
    f.payload = r.alloc + r.guard_lo;
    f.bytes = (r.dist == ASMV_DIST_NONE) ? 0 : pb;
    f.tile0 = tile;
    f.dtype = r.dtype;
    f.dist = r.dist;
    f.region_id = r.region_id;
    f.vec = (f.payload % 16) == 0;
    if (r.dist == ASMV_DIST_UNIFORM) {
      f.f0 = (float)r.p0;
      f.f1 = (float)r.p1 - f.f0;
    } else if (r.dist == ASMV_DIST_NORMAL) {
      f.f0 = (float)r.p0;
      f.f1 = (float)r.p1;
    } else if (r.dist == ASMV_DIST_INT_RANGE) {
      f.ilo = (int64_t)r.p0;
      f.ispan = (uint64_t)((int64_t)r.p1 - (int64_t)r.p0);
    }
#if ASMV_DEBUG_BOUNDS
    f.alloc = Span{r.alloc, r.alloc + tot};
    if (f.bytes) f.bytes += ctx->debug_widen;       // the test hook: loop past the payload
#endif
    tile += (f.bytes + kFillTileBytes - 1) / kFillTileBytes;
    if (f.bytes != 0 && f.dist == ASMV_DIST_NORMAL) {
      const uint32_t sz = (uint32_t)kDtypeSize[r.dtype];
      needs |= sz == 2 ? kNeedN16 : sz == 1 ? kNeedN8 : kNeedLn;
    }
    add_region_guards(segs, r, kSegFill, (uint32_t)i);
  }
  std::memset(&fr[n], 0, sizeof(FillRegion));
  fr[n].tile0 = tile;
  if (tile == 0 && segs.empty()) return ASMV_OK;

  Image img;
  const size_t o_regs = img.add(fr.data(), fr.size() * sizeof(FillRegion));
  const size_t o_segs = img.add(segs.data(), segs.size() * sizeof(GuardSeg));
#if ASMV_DEBUG_BOUNDS
  const uint32_t zero = 0;
  const size_t o_err = img.add(&zero, sizeof zero);
#endif
  unsigned char *dev = nullptr;
  cudaStream_t s = (cudaStream_t)stream;
  if ((rc = stage(ctx, img, debug_err_bytes(), s, &dev)) != ASMV_OK) return rc;
  FillParams p;
#if ASMV_DEBUG_BOUNDS
  p.err = (uint32_t *)(dev + o_err);
#endif
  p.regions = (const FillRegion *)(dev + o_regs);
  p.segs = (const GuardSeg *)(dev + o_segs);
  p.ntiles = tile;
  p.seed = seed;
  p.nregions = (uint32_t)n;
  p.nsegs = (uint32_t)segs.size();
  p.smem = fill_layout(needs);
  for (uint32_t r = 0; r < 10; ++r) {      // Philox round keys (Weyl sequence from the seed)
    p.key0[r] = (uint32_t)seed + r * 0x9E3779B9u;
    p.key1[r] = (uint32_t)(seed >> 32) + r * 0xBB67AE85u;
  }
  cudaError_t e;
  if (ctx->timing && (e = cudaEventRecord(ctx->t0, s)) != cudaSuccess) return fail_cuda(ctx, e);
  if ((e = (cudaError_t)launch_fill(p, grid_for(ctx, tile, segs.size(), ctx->fill_ctas[needs]), s)) !=
      cudaSuccess)
    return fail_cuda(ctx, e);
  ctx->launches += 1;
  if (ctx->timing) {
    if ((e = cudaEventRecord(ctx->t1, s)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->timed = true;
  }
#if ASMV_DEBUG_BOUNDS
  if ((rc = after_launch(ctx, s)) != ASMV_OK) return rc;
  return debug_finish(ctx, o_err, img.bytes.size(), s);
#else
  return after_launch(ctx, s);
#endif
}

// Shared body of guard_check / compare / compare_batched.
static int run_compare(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                       size_t k, size_t n, const asmv_tol *tol, asmv_stats *out, cudaStream_t s,
                       bool guard_only) {
  std::pair<uint64_t, uint64_t> last(0, 0);
  int rc;
  if ((rc = check_device_table(ctx, ref, n, last)) != ASMV_OK) return rc;
  for (size_t j = 0; j < k && !guard_only; ++j)
    if ((rc = check_device_table(ctx, cands[j], n, last)) != ASMV_OK) return rc;

  std::vector<CmpRegion> cr(n + 1);
  std::vector<uint64_t> caddr(guard_only ? 0 : k * n);
  std::vector<Span> callocs(ASMV_DEBUG_BOUNDS && !guard_only ? k * n : 0);   // debug-bounds build
  std::vector<GuardSeg> segs;
  uint64_t tile = 0;
  const uint32_t tile_bytes = compare_tile_bytes((uint32_t)std::min<size_t>(std::max<size_t>(k, 1), kMaxCands));
  for (size_t i = 0; i < n; ++i) {
    const asmv_region &r = ref[i];
    uint64_t pb, tot;
    region_extent(r, &pb, &tot);
    CmpRegion &c = cr[i];
    std::memset(&c, 0, sizeof c);
    c.ref = r.alloc + r.guard_lo;
    c.bytes = guard_only ? 0 : pb;
    c.tile0 = tile;
    c.dtype = r.dtype;
#if ASMV_DEBUG_BOUNDS
    c.alloc = Span{r.alloc, r.alloc + tot};
#endif
    bool vec = (c.ref % 16) == 0;
    for (size_t j = 0; j < caddr.size() / (n ? n : 1); ++j) {
      const uint64_t a = cands[j][i].alloc + cands[j][i].guard_lo;
      caddr[j * n + i] = a;
      vec = vec && (a % 16) == 0;
      if (!callocs.empty()) {
        uint64_t cpb, ctot;
        region_extent(cands[j][i], &cpb, &ctot);
        callocs[j * n + i] = Span{cands[j][i].alloc, cands[j][i].alloc + ctot};
      }
    }
    c.vec = vec;
    tile += (c.bytes + tile_bytes - 1) / tile_bytes;
    if (guard_only) {
      add_region_guards(segs, r, kSegSelf, (uint32_t)i);
    } else {
      add_region_guards(segs, r, kSegRef, (uint32_t)i);
      for (size_t j = 0; j < k; ++j) add_region_guards(segs, cands[j][i], kSegCand, (uint32_t)(j * n + i));
    }
  }
  std::memset(&cr[n], 0, sizeof(CmpRegion));
  cr[n].tile0 = tile;
  const size_t nstats = guard_only ? n : k * n;
  if (nstats == 0) return ASMV_OK;
  // statistics, then one error word, read back together
  std::vector<StatsDev> st(nstats + 1, empty_stats());
  std::memset(&st[nstats], 0, sizeof(StatsDev));

  Image img;
  const size_t o_regs = img.add(cr.data(), cr.size() * sizeof(CmpRegion));
  const size_t o_cand = img.add(caddr.data(), caddr.size() * sizeof(uint64_t));
  const size_t o_segs = img.add(segs.data(), segs.size() * sizeof(GuardSeg));
  const size_t o_stats = img.add(st.data(), st.size() * sizeof(StatsDev));
  const size_t o_callocs = img.add(callocs.data(), callocs.size() * sizeof(Span));
  (void)o_callocs;
  unsigned char *dev = nullptr;
  if ((rc = stage(ctx, img, st.size() * sizeof(StatsDev), s, &dev)) != ASMV_OK) return rc;

  CmpParams p;
  std::memset(&p, 0, sizeof p);
  p.regions = (const CmpRegion *)(dev + o_regs);
  p.segs = (const GuardSeg *)(dev + o_segs);
  p.seg_stats = (StatsDev *)(dev + o_stats);
  p.err = (uint32_t *)((StatsDev *)(dev + o_stats) + nstats);
  p.ntiles = tile;
  p.nregions = (uint32_t)n;
  p.tile_bytes = tile_bytes;
  p.wait_rounds = ctx->wait_rounds;
  for (int d = 0; d < ASMV_NDTYPES; ++d) {
    if (is_float((uint32_t)d) && tol) p.tol[d] = make_tolf(tol[d]);
  }
  cudaError_t e;
  if (ctx->timing && (e = cudaEventRecord(ctx->t0, s)) != cudaSuccess) return fail_cuda(ctx, e);
  const size_t groups = guard_only ? 1 : (k + kMaxCands - 1) / kMaxCands;
  for (size_t g = 0; g < groups; ++g) {
    const size_t kg = guard_only ? 1 : std::min<size_t>(kMaxCands, k - g * kMaxCands);
    p.K = (uint32_t)kg;
    p.nstages = compare_stages(p.K, tile_bytes);
    p.cands = (const uint64_t *)(dev + o_cand) + g * kMaxCands * n;
#if ASMV_DEBUG_BOUNDS
    p.cand_allocs = (const Span *)(dev + o_callocs) + g * kMaxCands * n;
#endif
    p.stats = (StatsDev *)(dev + o_stats) + g * kMaxCands * n;
    p.nsegs = (g == 0) ? (uint32_t)segs.size() : 0u;
    if (guard_only) p.ntiles = 0;
    // one CTA per SM: the shared-memory pipeline sizes itself to the SM
    const uint64_t segs_per_cta = kConsumerWarps + 1;
    const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(
        std::max<uint64_t>(p.ntiles, (p.nsegs + segs_per_cta - 1) / segs_per_cta), sms_of(ctx)));
    if ((e = (cudaError_t)launch_compare(p, grid, s)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->launches += 1;
  }
  if (ctx->timing) {
    if ((e = cudaEventRecord(ctx->t1, s)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->timed = true;
  }
  if ((rc = after_launch(ctx, s)) != ASMV_OK) return rc;
  return readback(ctx, o_stats, img.bytes.size(), nstats, s, out, guard_only ? 0 : n);
}

int asmv_guard_check(asmv_ctx *ctx, const asmv_region *regions, size_t n, asmv_stats *out_host,
                     asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_guard_check");
  if (ctx == nullptr || (n > 0 && out_host == nullptr)) return ASMV_EINVAL;
  int rc = check_table(regions, n, false);
  if (rc != ASMV_OK) return rc;
  if (n == 0) return ASMV_OK;
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  return run_compare(ctx, regions, nullptr, 0, n, nullptr, out_host, (cudaStream_t)stream, true);
}

static int check_pairs(const asmv_region *ref, const asmv_region *const *cands, size_t k, size_t n) {
  int rc = check_table(ref, n, false);
  if (rc != ASMV_OK) return rc;
  for (size_t j = 0; j < k; ++j) {
    if (n > 0 && cands[j] == nullptr) return ASMV_EINVAL;
    if ((rc = check_table(cands[j], n, false)) != ASMV_OK) return rc;
    for (size_t i = 0; i < n; ++i)
      if (cands[j][i].dtype != ref[i].dtype || cands[j][i].n_elems != ref[i].n_elems)
        return ASMV_EINVAL;
  }
  return ASMV_OK;
}

int asmv_compare(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *cand, size_t n,
                 const asmv_tol *tol, asmv_stats *out_host, asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_compare");
  if (ctx == nullptr || (n > 0 && (out_host == nullptr || cand == nullptr)) || !tol_ok(tol))
    return ASMV_EINVAL;
  const asmv_region *cands[1] = {cand};
  int rc = check_pairs(ref, cands, 1, n);
  if (rc != ASMV_OK) return rc;
  if (n == 0) return ASMV_OK;
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  return run_compare(ctx, ref, cands, 1, n, tol, out_host, (cudaStream_t)stream, false);
}

int asmv_compare_batched(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                         size_t k, size_t n, const asmv_tol *tol, asmv_stats *out_host,
                         asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_compare_batched");
  if (ctx == nullptr || k == 0 || cands == nullptr || (n > 0 && out_host == nullptr) || !tol_ok(tol))
    return ASMV_EINVAL;
  if (k > (size_t)0x7FFFFFFF / (n ? n : 1)) return ASMV_EINVAL;
  int rc = check_pairs(ref, cands, k, n);
  if (rc != ASMV_OK) return rc;
  if (n == 0) return ASMV_OK;
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  return run_compare(ctx, ref, cands, k, n, tol, out_host, (cudaStream_t)stream, false);
}

// The exact Eq. 1 sums of k candidates: fills digits[n][1 + 2k][kEqDigits]
// for the float regions other than binary64, and digits64[m][1 + 2k]
// [kEq64Digits] for the m-th binary64 region of the table.
static int run_eq(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                  size_t k, size_t n, cudaStream_t s, std::vector<long long> &digits,
                  std::vector<long long> &digits64) {
  const size_t nslots = 1 + 2 * k;
  digits.assign(n * nslots * kEqDigits, 0);
  std::vector<CmpRegion> cr(n + 1), cr64;
  std::vector<uint64_t> caddr(k * n), caddr64;
  std::vector<size_t> idx64;                       // table index of each binary64 region
  for (size_t i = 0; i < n; ++i)
    if (ref[i].dtype == ASMV_F64) idx64.push_back(i);
  const size_t n64 = idx64.size();
  digits64.assign(n64 * nslots * kEq64Digits, 0);
  cr64.resize(n64 + 1);
  caddr64.resize(k * n64);
  uint64_t tile64 = 0;
  for (size_t m = 0; m < n64; ++m) {
    const asmv_region &r = ref[idx64[m]];
    uint64_t pb, tot;
    region_extent(r, &pb, &tot);
    CmpRegion &c = cr64[m];
    std::memset(&c, 0, sizeof c);
    c.ref = r.alloc + r.guard_lo;
    c.bytes = pb;
    c.tile0 = tile64;
    c.dtype = r.dtype;
    bool vec = (c.ref % 16) == 0;
    for (size_t j = 0; j < k; ++j) {
      const uint64_t a = cands[j][idx64[m]].alloc + cands[j][idx64[m]].guard_lo;
      caddr64[j * n64 + m] = a;
      vec = vec && (a % 16) == 0;
    }
    c.vec = vec;
    tile64 += (pb + kEq64TileBytes - 1) / kEq64TileBytes;
  }
  std::memset(&cr64[n64], 0, sizeof(CmpRegion));
  cr64[n64].tile0 = tile64;
  uint64_t tile = 0;
  for (size_t i = 0; i < n; ++i) {
    const asmv_region &r = ref[i];
    uint64_t pb, tot;
    region_extent(r, &pb, &tot);
    CmpRegion &c = cr[i];
    std::memset(&c, 0, sizeof c);
    c.ref = r.alloc + r.guard_lo;
    c.bytes = (is_float(r.dtype) && r.dtype != ASMV_F64) ? pb : 0;
    c.tile0 = tile;
    c.dtype = r.dtype;
    bool vec = (c.ref % 16) == 0;
    for (size_t j = 0; j < k; ++j) {
      const uint64_t a = cands[j][i].alloc + cands[j][i].guard_lo;
      caddr[j * n + i] = a;
      vec = vec && (a % 16) == 0;
    }
    c.vec = vec;
    tile += tiles_of(c.bytes);
  }
  std::memset(&cr[n], 0, sizeof(CmpRegion));
  cr[n].tile0 = tile;
  if (tile == 0 && tile64 == 0) return ASMV_OK;     // no float payload: all sums are zero
  const size_t dig_bytes = digits.size() * sizeof(long long);
  const size_t dig64_bytes = digits64.size() * sizeof(long long);
  const size_t o_dig64 = (dig_bytes + 255) & ~(size_t)255;     // from o_dig
  const size_t all_dig = o_dig64 + dig64_bytes;

  Image img;
  const size_t o_regs = img.add(cr.data(), cr.size() * sizeof(CmpRegion));
  const size_t o_cand = img.add(caddr.data(), caddr.size() * sizeof(uint64_t));
  const size_t o_regs64 = img.add(cr64.data(), cr64.size() * sizeof(CmpRegion));
  const size_t o_cand64 = img.add(caddr64.data(), caddr64.size() * sizeof(uint64_t));
  const size_t o_dig = (img.bytes.size() + 255) & ~(size_t)255;
  unsigned char *dev = nullptr;
  int rc;
  if ((rc = stage(ctx, img, all_dig, s, &dev, all_dig)) != ASMV_OK) return rc;
  cudaError_t e;
  if ((e = cudaMemsetAsync(dev + o_dig, 0, all_dig, s)) != cudaSuccess) return fail_cuda(ctx, e);

  EqParams p;
  std::memset(&p, 0, sizeof p);
  p.regions = (const CmpRegion *)(dev + o_regs);
  p.digits = (long long *)(dev + o_dig);
  p.ntiles = tile;
  p.nregions = (uint32_t)n;
  p.nslots = (uint32_t)nslots;
  const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(tile, sms_of(ctx) * ctx->eq_ctas));
  Eq64Params p64;
  std::memset(&p64, 0, sizeof p64);
  p64.regions = (const CmpRegion *)(dev + o_regs64);
  p64.digits = (long long *)(dev + o_dig + o_dig64);
  p64.ntiles = tile64;
  p64.nregions = (uint32_t)n64;
  p64.nslots = (uint32_t)nslots;
  const int grid64 =
      (int)std::max<uint64_t>(1, std::min<uint64_t>(tile64, sms_of(ctx) * ctx->eq64_ctas));
  if (ctx->timing && (e = cudaEventRecord(ctx->t0, s)) != cudaSuccess) return fail_cuda(ctx, e);
  for (size_t g = 0; g * kMaxCands < k; ++g) {
    p.K = p64.K = (uint32_t)std::min<size_t>(kMaxCands, k - g * kMaxCands);
    p.j0 = p64.j0 = (uint32_t)(g * kMaxCands);
    p.do_rr = p64.do_rr = g == 0;
    p.cands = (const uint64_t *)(dev + o_cand) + g * kMaxCands * n;
    p64.cands = (const uint64_t *)(dev + o_cand64) + g * kMaxCands * n64;
    if (tile > 0) {
      if ((e = (cudaError_t)launch_eq(p, grid, s)) != cudaSuccess) return fail_cuda(ctx, e);
      ctx->launches += 1;
    }
    if (tile64 > 0) {
      if ((e = (cudaError_t)launch_eq64(p64, grid64, s)) != cudaSuccess) return fail_cuda(ctx, e);
      ctx->launches += 1;
    }
  }
  if (ctx->timing) {
    if ((e = cudaEventRecord(ctx->t1, s)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->timed = true;
  }
  if ((rc = after_launch(ctx, s)) != ASMV_OK) return rc;
  unsigned char *host = ctx->hst + ((img.bytes.size() + 255) & ~(size_t)255);
  if ((e = cudaMemcpyAsync(host, dev + o_dig, all_dig, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
    return fail_cuda(ctx, e);
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return fail_cuda(ctx, e);
  ctx->staged_pending = false;
  ctx->ws_pending = false;
  std::memcpy(digits.data(), host, dig_bytes);
  if (dig64_bytes) std::memcpy(digits64.data(), host + o_dig64, dig64_bytes);
  return ASMV_OK;
}

}  // extern "C"

namespace {

// Validation shared by asmv_compare_eq and asmv_compare_eq_digits.
int check_eq_call(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands, size_t k,
                  size_t n, const asmv_tol *tol, const void *stats_host, const void *out_host) {
  if (ctx == nullptr || k == 0 || cands == nullptr || !tol_ok(tol) ||
      (n > 0 && (stats_host == nullptr || out_host == nullptr)))
    return ASMV_EINVAL;
  if (k > (size_t)0x7FFFFFFF / (n ? n : 1)) return ASMV_EINVAL;
  int rc = check_pairs(ref, cands, k, n);
  if (rc != ASMV_OK) return rc;
  for (size_t i = 0; i < n; ++i)
    if (is_float(ref[i].dtype) && ref[i].n_elems > ((uint64_t)1 << 31)) return ASMV_EINVAL;
  return ASMV_OK;
}

// The statistics and the digit vectors of the Eq. 1 sums (the kernels).
int run_compare_eq(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands, size_t k,
                   size_t n, const asmv_tol *tol, asmv_stream_t stream, std::vector<asmv_stats> &stats,
                   std::vector<long long> &digits, std::vector<long long> &digits64) {
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  const cudaStream_t s = (cudaStream_t)stream;
  stats.assign(k * n, asmv_stats());
  int rc;
  if ((rc = run_compare(ctx, ref, cands, k, n, tol, stats.data(), s, false)) != ASMV_OK) return rc;
  return run_eq(ctx, ref, cands, k, n, s, digits, digits64);
}

// Eq. 1 of every (candidate, region) from statistics and digit vectors: the
// three sums rounded once each, the cosine and the four terms.  The digit
// vectors of the difference-form dtypes hold sum r d and sum d^2, from which
// S_rc = S_rr + sum r d and S_cc = S_rr + 2 sum r d + sum d^2, digit by
// digit; a digit sum that would leave the int64 range is rejected.
//
// Binary64 regions take their sums from digits64 (the m-th binary64 region
// of the table at [m][1 + 2k][kEq64Digits]): each rounded with gradual
// underflow and overflow to infinity, and the cosine formed from the sums
// scaled by powers of two (eq_cosine_scaled).
int eq_combine(const uint32_t *dtypes, size_t k, size_t n, const asmv_stats *stats,
               const long long *digits, const long long *digits64, double theta, double tau,
               asmv_eq *res) {
  const size_t nslots = 1 + 2 * k;
  std::vector<size_t> m64(n, 0);
  for (size_t i = 0, m = 0; i < n; ++i)
    if (dtypes[i] == ASMV_F64) m64[i] = m++;
  for (size_t j = 0; j < k; ++j) {
    for (size_t i = 0; i < n; ++i) {
      const asmv_stats &st = stats[j * n + i];
      asmv_eq &q = res[j * n + i];
      std::memset(&q, 0, sizeof q);
      const bool flt = is_float(dtypes[i]);
      if (flt && dtypes[i] == ASMV_F64) {
        if (digits64 == nullptr) return ASMV_EINVAL;
        const long long *d = digits64 + m64[i] * nslots * kEq64Digits;
        Magnitude rr, rc, cc;
        magnitude_of((const int64_t *)d, kEq64Digits, &rr);
        magnitude_of((const int64_t *)(d + (1 + 2 * j) * kEq64Digits), kEq64Digits, &rc);
        magnitude_of((const int64_t *)(d + (2 + 2 * j) * kEq64Digits), kEq64Digits, &cc);
        if (rr.neg || cc.neg) return ASMV_EINVAL;           // sums of squares
        q.sum_rr = round_magnitude(rr, kEq64Base);
        q.sum_cc = round_magnitude(cc, kEq64Base);
        q.sum_rc = round_magnitude(rc, kEq64Base);
        if (rc.neg) q.sum_rc = -q.sum_rc;
        q.cos = eq_cosine_scaled(rc, rr, cc, kEq64Base);
      } else if (flt) {
        const long long *d = digits + i * nslots * kEqDigits;
        const int base = eq_digit_base(dtypes[i]);
        int64_t rc[kEqDigits], cc[kEqDigits];
        const long long *rr = d, *s1 = d + (1 + 2 * j) * kEqDigits, *s2 = d + (2 + 2 * j) * kEqDigits;
        const bool diff = eq_difference_form(dtypes[i]);
        for (int m = 0; m < kEqDigits; ++m) {
          if (diff) {
            long long a, b, c;
            if (__builtin_add_overflow(rr[m], s1[m], &a) || __builtin_add_overflow(a, s1[m], &b) ||
                __builtin_add_overflow(b, s2[m], &c))
              return ASMV_EINVAL;
            rc[m] = a;
            cc[m] = c;
          } else {
            rc[m] = s1[m];
            cc[m] = s2[m];
          }
        }
        if (exact_to_double_impl(rc, kEqDigits, base, &q.sum_rc) != ASMV_OK ||
            exact_to_double_impl((const int64_t *)rr, kEqDigits, base, &q.sum_rr) != ASMV_OK ||
            exact_to_double_impl(cc, kEqDigits, base, &q.sum_cc) != ASMV_OK)
          return ASMV_EINVAL;
        q.cos = eq_cosine(q.sum_rc, q.sum_rr, q.sum_cc);
      } else {
        q.cos = NAN;
      }
      uint32_t f = 0;
      if (!flt || q.cos >= theta) f |= ASMV_EQ_COS;
      if (!flt || (st.max_abs_err <= tau && st.nonfinite_mismatches == 0)) f |= ASMV_EQ_LINF;
      if (flt || st.mismatches == 0) f |= ASMV_EQ_INT;
      if (st.guard_bad_bytes == 0) f |= ASMV_EQ_GUARD;
      q.flags = f;
      q.eq = f == (ASMV_EQ_COS | ASMV_EQ_LINF | ASMV_EQ_INT | ASMV_EQ_GUARD);
    }
  }
  return ASMV_OK;
}

bool theta_tau_ok(double theta, double tau) {
  return std::isfinite(theta) && std::isfinite(tau) && tau >= 0.0;
}

}  // namespace

extern "C" {

int asmv_compare_eq(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                    size_t k, size_t n, const asmv_tol *tol, double theta, double tau,
                    asmv_stats *stats_host, asmv_eq *eq_host, asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_compare_eq");
  int rc = check_eq_call(ctx, ref, cands, k, n, tol, stats_host, eq_host);
  if (rc != ASMV_OK) return rc;
  if (!theta_tau_ok(theta, tau)) return ASMV_EINVAL;
  if (n == 0) return ASMV_OK;
  std::vector<asmv_stats> stats;
  std::vector<long long> digits, digits64;
  if ((rc = run_compare_eq(ctx, ref, cands, k, n, tol, stream, stats, digits, digits64)) != ASMV_OK)
    return rc;
  std::vector<uint32_t> dt(n);
  for (size_t i = 0; i < n; ++i) dt[i] = ref[i].dtype;
  std::vector<asmv_eq> res(k * n);
  if (eq_combine(dt.data(), k, n, stats.data(), digits.data(), digits64.data(), theta, tau,
                 res.data()) != ASMV_OK)
    return ASMV_ECUDA;                                // digits out of range: a device fault
  std::memcpy(stats_host, stats.data(), stats.size() * sizeof(asmv_stats));
  std::memcpy(eq_host, res.data(), res.size() * sizeof(asmv_eq));
  return ASMV_OK;
}

int asmv_compare_eq_digits(asmv_ctx *ctx, const asmv_region *ref, const asmv_region *const *cands,
                           size_t k, size_t n, const asmv_tol *tol, asmv_stats *stats_host,
                           int64_t *digits_host, asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_compare_eq_digits");
  int rc = check_eq_call(ctx, ref, cands, k, n, tol, stats_host, digits_host);
  if (rc != ASMV_OK) return rc;
  if (n == 0) return ASMV_OK;
  std::vector<asmv_stats> stats;
  std::vector<long long> digits, digits64;
  if ((rc = run_compare_eq(ctx, ref, cands, k, n, tol, stream, stats, digits, digits64)) != ASMV_OK)
    return rc;
  std::memcpy(stats_host, stats.data(), stats.size() * sizeof(asmv_stats));
  if (digits64.empty()) {
    std::memcpy(digits_host, digits.data(), digits.size() * sizeof(int64_t));
    return ASMV_OK;
  }
  // a table with binary64 regions: every slot takes kEq64Digits digits
  const size_t nslots = 1 + 2 * k;
  size_t m = 0;
  for (size_t i = 0; i < n; ++i) {
    int64_t *dst = digits_host + i * nslots * kEq64Digits;
    if (ref[i].dtype == ASMV_F64) {
      std::memcpy(dst, digits64.data() + m * nslots * kEq64Digits, nslots * kEq64Digits * sizeof(int64_t));
      ++m;
      continue;
    }
    for (size_t sl = 0; sl < nslots; ++sl) {
      std::memcpy(dst + sl * kEq64Digits, digits.data() + (i * nslots + sl) * kEqDigits,
                  kEqDigits * sizeof(int64_t));
      std::memset(dst + sl * kEq64Digits + kEqDigits, 0, (kEq64Digits - kEqDigits) * sizeof(int64_t));
    }
  }
  return ASMV_OK;
}

int asmv_eq_from_digits(const uint32_t *dtypes, size_t k, size_t n, const asmv_stats *stats,
                        const int64_t *digits, double theta, double tau, asmv_eq *eq_out) {
  if (k == 0 || !theta_tau_ok(theta, tau)) return ASMV_EINVAL;
  if (n == 0) return ASMV_OK;
  if (dtypes == nullptr || stats == nullptr || digits == nullptr || eq_out == nullptr) return ASMV_EINVAL;
  if (k > (size_t)0x7FFFFFFF / n) return ASMV_EINVAL;
  size_t n64 = 0;
  for (size_t i = 0; i < n; ++i) {
    if (dtypes[i] >= (uint32_t)ASMV_NDTYPES) return ASMV_EINVAL;
    n64 += dtypes[i] == ASMV_F64;
  }
  std::vector<asmv_eq> res(k * n);
  int rc;
  if (n64 == 0) {
    rc = eq_combine(dtypes, k, n, stats, (const long long *)digits, nullptr, theta, tau, res.data());
  } else {
    // kEq64Digits per slot: split into the two layouts eq_combine reads
    const size_t nslots = 1 + 2 * k;
    std::vector<long long> d20(n * nslots * kEqDigits, 0), d64(n64 * nslots * kEq64Digits);
    for (size_t i = 0, m = 0; i < n; ++i) {
      const int64_t *src = digits + i * nslots * kEq64Digits;
      if (dtypes[i] == ASMV_F64) {
        std::memcpy(d64.data() + m * nslots * kEq64Digits, src, nslots * kEq64Digits * sizeof(int64_t));
        ++m;
        continue;
      }
      // the digits past this format's 20 (all -1 words for a carried negative
      // sum) fold into its top digit, which must stay in int64
      for (size_t sl = 0; sl < nslots; ++sl) {
        const int64_t *x = src + sl * kEq64Digits;
        long long *y = d20.data() + (i * nslots + sl) * kEqDigits;
        __int128 top = 0;
        for (int d = kEq64Digits - 1; d >= kEqDigits - 1; --d) {
          top = top * ((__int128)1 << 32) + x[d];
          if (top > INT64_MAX || top < INT64_MIN) return ASMV_EINVAL;
        }
        std::memcpy(y, x, (kEqDigits - 1) * sizeof(int64_t));
        y[kEqDigits - 1] = (long long)top;
      }
    }
    rc = eq_combine(dtypes, k, n, stats, d20.data(), d64.data(), theta, tau, res.data());
  }
  if (rc != ASMV_OK) return rc;
  std::memcpy(eq_out, res.data(), res.size() * sizeof(asmv_eq));
  return ASMV_OK;
}

int asmv_eq_digit_base(uint32_t dtype, int *base) {
  if (base == nullptr || dtype >= (uint32_t)ASMV_NDTYPES || !is_float(dtype)) return ASMV_EINVAL;
  *base = dtype == ASMV_F64 ? kEq64Base : eq_digit_base(dtype);
  return ASMV_OK;
}

// Shared body of asmv_restore / asmv_capture: move every region's payload
// between the region and the caller's buffer addrs[i] (restore: buffer ->
// region, and guard bands rewritten; capture: region -> buffer).
static int run_copy(asmv_ctx *ctx, const asmv_region *regions, const uint64_t *addrs, size_t n,
                    asmv_stream_t stream, bool restore) {
  if (ctx == nullptr || (n > 0 && addrs == nullptr)) return ASMV_EINVAL;
  int rc = check_table(regions, n, false);
  if (rc != ASMV_OK) return rc;
  // allocations pairwise disjoint; buffers disjoint from every allocation
  // (and, for capture, from one another)
  std::vector<std::pair<std::pair<uint64_t, uint64_t>, int>> spans;   // (range, 0 alloc / 1 buffer)
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    region_extent(regions[i], &pb, &tot);
    if (tot > 0) spans.push_back({{regions[i].alloc, regions[i].alloc + tot}, 0});
    if (pb > 0) {
      if (addrs[i] == 0 || addrs[i] + pb < addrs[i]) return ASMV_EINVAL;
      spans.push_back({{addrs[i], addrs[i] + pb}, 1});
    }
  }
  std::sort(spans.begin(), spans.end());
  for (size_t i = 0; i < spans.size(); ++i)
    for (size_t j = i + 1; j < spans.size() && spans[j].first.first < spans[i].first.second; ++j)
      if (spans[i].second == 0 || spans[j].second == 0 || !restore) return ASMV_EINVAL;
  if (n == 0) return ASMV_OK;
  DeviceScope ds(ctx->device);
  if (!ds.ok) return fail_cuda(ctx, cudaErrorInvalidDevice);
  std::pair<uint64_t, uint64_t> last(0, 0);
  if ((rc = check_device_table(ctx, regions, n, last)) != ASMV_OK) return rc;
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    region_extent(regions[i], &pb, &tot);
    if ((rc = check_device_span(ctx, addrs[i], pb, last)) != ASMV_OK) return rc;
  }
  std::vector<CopyRegion> cr(n + 1);
  std::vector<GuardSeg> segs;
  uint64_t tile = 0;
  for (size_t i = 0; i < n; ++i) {
    const asmv_region &r = regions[i];
    uint64_t pb, tot;
    region_extent(r, &pb, &tot);
    CopyRegion &c = cr[i];
    std::memset(&c, 0, sizeof c);
    const uint64_t payload = r.alloc + r.guard_lo;
    c.dst = restore ? payload : addrs[i];
    c.src = restore ? addrs[i] : payload;
    c.bytes = pb;
    c.tile0 = tile;
    c.vec = (c.dst % 16 == 0) && (c.src % 16 == 0);
#if ASMV_DEBUG_BOUNDS
    // the region's allocation on one side, the caller's buffer [addr, addr + payload) on the other
    const Span region_alloc{r.alloc, r.alloc + tot}, buffer{addrs[i], addrs[i] + pb};
    c.dst_alloc = restore ? region_alloc : buffer;
    c.src_alloc = restore ? buffer : region_alloc;
#endif
    tile += tiles_of(pb);
    if (restore) add_region_guards(segs, r, kSegFill, (uint32_t)i);
  }
  std::memset(&cr[n], 0, sizeof(CopyRegion));
  cr[n].tile0 = tile;
  if (tile == 0 && segs.empty()) return ASMV_OK;
  Image img;
  const size_t o_regs = img.add(cr.data(), cr.size() * sizeof(CopyRegion));
  const size_t o_segs = img.add(segs.data(), segs.size() * sizeof(GuardSeg));
#if ASMV_DEBUG_BOUNDS
  const uint32_t zero = 0;
  const size_t o_err = img.add(&zero, sizeof zero);
#endif
  unsigned char *dev = nullptr;
  const cudaStream_t s = (cudaStream_t)stream;
  if ((rc = stage(ctx, img, debug_err_bytes(), s, &dev)) != ASMV_OK) return rc;
  CopyParams p;
  std::memset(&p, 0, sizeof p);
#if ASMV_DEBUG_BOUNDS
  p.err = (uint32_t *)(dev + o_err);
#endif
  p.regions = (const CopyRegion *)(dev + o_regs);
  p.segs = (const GuardSeg *)(dev + o_segs);
  p.ntiles = tile;
  p.nregions = (uint32_t)n;
  p.nsegs = (uint32_t)segs.size();
  cudaError_t e;
  if (ctx->timing && (e = cudaEventRecord(ctx->t0, s)) != cudaSuccess) return fail_cuda(ctx, e);
  if ((e = (cudaError_t)launch_copy(p, grid_for(ctx, tile, segs.size(), ctx->copy_ctas), s)) !=
      cudaSuccess)
    return fail_cuda(ctx, e);
  ctx->launches += 1;
  if (ctx->timing) {
    if ((e = cudaEventRecord(ctx->t1, s)) != cudaSuccess) return fail_cuda(ctx, e);
    ctx->timed = true;
  }
#if ASMV_DEBUG_BOUNDS
  if ((rc = after_launch(ctx, s)) != ASMV_OK) return rc;
  return debug_finish(ctx, o_err, img.bytes.size(), s);
#else
  return after_launch(ctx, s);
#endif
}

int asmv_restore(asmv_ctx *ctx, const asmv_region *regions, const uint64_t *src, size_t n,
                 asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_restore");
  return run_copy(ctx, regions, src, n, stream, true);
}

int asmv_capture(asmv_ctx *ctx, const asmv_region *regions, const uint64_t *dst, size_t n,
                 asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_capture");
  return run_copy(ctx, regions, dst, n, stream, false);
}

int asmv_exact_to_double(const int64_t *digits, int ndigits, int base_exp, double *out) {
  return exact_to_double_impl(digits, ndigits, base_exp, out);
}

}  // extern "C"

// ==================================================== compare without allocation
// Some callers must not allocate device memory while they check a
// candidate: a differential-testing harness that replays captured
// dispatches restores regions at their original virtual addresses and
// needs the address space it reserved to stay exactly as it was, and a
// harness that times candidate kernels cannot afford the device-wide
// synchronisation an allocation may cause.  asmv_compare_noalloc serves
// them: its scratch (the launch plan and the statistics) lives in the
// file-scope device array below, which every GPU that loads this library
// holds until the process exits, and host-side staging is a static
// buffer.  It calls no allocating routine.
namespace {

constexpr size_t kNoAllocBytes = ASMV_NOALLOC_SCRATCH_BYTES;
constexpr int kNoAllocMaxDevices = 64;

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {

alignas(256) unsigned char g_noalloc_host[kNoAllocBytes];   // host image of the same layout
int g_noalloc_sms[kNoAllocMaxDevices];                       // SM count per device (0: not yet read)
AddrRangeFn g_noalloc_range = nullptr;
bool g_noalloc_range_looked_up = false;
std::mutex g_noalloc_mutex;

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Set-up for the current device (under the mutex): the device address of
// the scratch array in the current context, the SM count and the
// address-range lookup.  The address is looked up on every call, not kept:
// a context that was reset and created again loads the module anew, and the
// array may then sit elsewhere (the lookup allocates nothing).
int noalloc_setup(int dev, unsigned char **scratch) {
  if (dev < 0 || dev >= kNoAllocMaxDevices) return ASMV_EINVAL;
  void *p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess || p == nullptr) { cudaGetLastError(); return ASMV_ECUDA; }
  *scratch = (unsigned char *)p;
  if (g_noalloc_sms[dev]) return ASMV_OK;
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return ASMV_ECUDA;
  }
  if (!g_noalloc_range_looked_up) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_noalloc_range = (AddrRangeFn)fn;
    else
      cudaGetLastError();
    g_noalloc_range_looked_up = true;
  }
  g_noalloc_sms[dev] = sms;
  return ASMV_OK;
}

// Device-memory check of one allocation on the current device (no context).
// `last` is the allocation range the previous region was found in: a region
// inside it needs no driver query.
int noalloc_check_span(int dev, uint64_t alloc, uint64_t total, std::pair<uint64_t, uint64_t> &last) {
  if (total == 0) return ASMV_OK;
  if (alloc >= last.first && alloc + total <= last.second) return ASMV_OK;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, (const void *)alloc) != cudaSuccess) {
    cudaGetLastError();
    return ASMV_EINVAL;
  }
  if (a.type == cudaMemoryTypeDevice) {
    if (a.device != dev) return ASMV_EINVAL;
  } else if (a.type != cudaMemoryTypeManaged) {
    return ASMV_EINVAL;
  }
  if (g_noalloc_range) {
    unsigned long long base = 0;
    size_t size = 0;
    if (g_noalloc_range(&base, &size, alloc) != 0) return ASMV_EINVAL;
    if (alloc + total > base + size) return ASMV_EINVAL;
    last = std::make_pair((uint64_t)base, (uint64_t)(base + size));
  }
  return ASMV_OK;
}

size_t noalloc_segments(const asmv_region &r) {
  return ((size_t)r.guard_lo + kGuardSegBytes - 1) / kGuardSegBytes +
         ((size_t)r.guard_hi + kGuardSegBytes - 1) / kGuardSegBytes;
}

// Guard segments of one region written straight into the image.
size_t noalloc_put_guards(GuardSeg *out, const asmv_region &r, uint8_t kind, uint32_t stats) {
  uint64_t pb, tot;
  region_extent(r, &pb, &tot);
  size_t k = 0;
  const uint64_t starts[2] = {r.alloc, r.alloc + r.guard_lo + pb};
  const uint64_t offs[2] = {0, (uint64_t)r.guard_lo + pb};
  const uint64_t lens[2] = {r.guard_lo, r.guard_hi};
  for (int side = 0; side < 2; ++side) {
    for (uint64_t o = 0; o < lens[side]; o += kGuardSegBytes) {
      GuardSeg &g = out[k++];
      std::memset(&g, 0, sizeof g);
      g.ptr = starts[side] + o;
      g.offset = offs[side] + o;
      g.len = (uint32_t)std::min<uint64_t>(kGuardSegBytes, lens[side] - o);
      g.stats = stats;
      g.canary = r.canary;
      g.kind = kind;
#if ASMV_DEBUG_BOUNDS
      g.alloc = Span{r.alloc, r.alloc + tot};
#endif
    }
  }
  return k;
}

}  // namespace

extern "C" int asmv_compare_noalloc(const asmv_region *ref, const asmv_region *cand, size_t n,
                                    const asmv_tol *tol, asmv_stats *out_host,
                                    asmv_stream_t stream) {
  ASMV_NVTX_RANGE("asmv_compare_noalloc");
  if ((n > 0 && (out_host == nullptr || cand == nullptr)) || !tol_ok(tol)) return ASMV_EINVAL;
  int rc = check_table(ref, n, false);
  if (rc != ASMV_OK) return rc;
  if ((rc = check_table(cand, n, false)) != ASMV_OK) return rc;
  for (size_t i = 0; i < n; ++i)
    if (cand[i].dtype != ref[i].dtype || cand[i].n_elems != ref[i].n_elems) return ASMV_EINVAL;
  if (n == 0) return ASMV_OK;

  // sizes of the image: regions (+ sentinel), candidate addresses, guard
  // segments, statistics (+ the error word)
  size_t nsegs = 0;
  for (size_t i = 0; i < n; ++i) nsegs += noalloc_segments(ref[i]) + noalloc_segments(cand[i]);
  const size_t o_regs = 0;
  const size_t o_cand = align256(o_regs + (n + 1) * sizeof(CmpRegion));
  const size_t o_segs = align256(o_cand + n * sizeof(uint64_t));
  const size_t o_stats = align256(o_segs + nsegs * sizeof(GuardSeg));
  const size_t o_callocs = align256(o_stats + (n + 1) * sizeof(StatsDev));   // debug-bounds build
  const size_t total = ASMV_DEBUG_BOUNDS ? o_callocs + n * sizeof(Span) : o_stats + (n + 1) * sizeof(StatsDev);
  if (total > kNoAllocBytes) return ASMV_EINVAL;      // beyond the fixed scratch

  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return ASMV_ECUDA; }
  unsigned char *dscr = nullptr;
  if ((rc = noalloc_setup(dev, &dscr)) != ASMV_OK) return rc;
  std::pair<uint64_t, uint64_t> last_ref(0, 0), last_cand(0, 0);
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    region_extent(ref[i], &pb, &tot);
    if ((rc = noalloc_check_span(dev, ref[i].alloc, tot, last_ref)) != ASMV_OK) return rc;
    region_extent(cand[i], &pb, &tot);
    if ((rc = noalloc_check_span(dev, cand[i].alloc, tot, last_cand)) != ASMV_OK) return rc;
  }

  const uint32_t tile_bytes = compare_tile_bytes(1);
  CmpRegion *cr = (CmpRegion *)(g_noalloc_host + o_regs);
  uint64_t *caddr = (uint64_t *)(g_noalloc_host + o_cand);
  GuardSeg *segs = (GuardSeg *)(g_noalloc_host + o_segs);
  StatsDev *st = (StatsDev *)(g_noalloc_host + o_stats);
  uint64_t tile = 0;
  size_t ks = 0;
  for (size_t i = 0; i < n; ++i) {
    uint64_t pb, tot;
    region_extent(ref[i], &pb, &tot);
    CmpRegion &c = cr[i];
    std::memset(&c, 0, sizeof c);
    c.ref = ref[i].alloc + ref[i].guard_lo;
    c.bytes = pb;
    c.tile0 = tile;
    c.dtype = ref[i].dtype;
    caddr[i] = cand[i].alloc + cand[i].guard_lo;
#if ASMV_DEBUG_BOUNDS
    c.alloc = Span{ref[i].alloc, ref[i].alloc + tot};
    {
      uint64_t cpb, ctot;
      region_extent(cand[i], &cpb, &ctot);
      ((Span *)(g_noalloc_host + o_callocs))[i] = Span{cand[i].alloc, cand[i].alloc + ctot};
    }
#endif
    c.vec = (c.ref % 16) == 0 && (caddr[i] % 16) == 0;
    tile += (pb + tile_bytes - 1) / tile_bytes;
    ks += noalloc_put_guards(segs + ks, ref[i], kSegRef, (uint32_t)i);
    ks += noalloc_put_guards(segs + ks, cand[i], kSegCand, (uint32_t)i);
    st[i] = empty_stats();
  }
  std::memset(&cr[n], 0, sizeof(CmpRegion));
  cr[n].tile0 = tile;
  std::memset(&st[n], 0, sizeof(StatsDev));          // the error word starts at zero

  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(dscr, g_noalloc_host, total, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return ASMV_ECUDA;
  CmpParams p;
  std::memset(&p, 0, sizeof p);
  p.regions = (const CmpRegion *)(dscr + o_regs);
  p.cands = (const uint64_t *)(dscr + o_cand);
  p.segs = (const GuardSeg *)(dscr + o_segs);
  p.stats = (StatsDev *)(dscr + o_stats);
  p.seg_stats = p.stats;
  p.err = (uint32_t *)(p.stats + n);
#if ASMV_DEBUG_BOUNDS
  p.cand_allocs = (const Span *)(dscr + o_callocs);
#endif
  p.ntiles = tile;
  p.nregions = (uint32_t)n;
  p.nsegs = (uint32_t)ks;
  p.K = 1;
  p.tile_bytes = tile_bytes;
  p.nstages = compare_stages(1, tile_bytes);
  p.wait_rounds = kWaitRounds;
  for (int d = 0; d < ASMV_NDTYPES; ++d)
    if (is_float((uint32_t)d)) p.tol[d] = make_tolf(tol[d]);
  const uint64_t per_cta = kConsumerWarps + 1;
  const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(
      std::max<uint64_t>(tile, (ks + per_cta - 1) / per_cta), (uint64_t)g_noalloc_sms[dev]));
  if ((e = (cudaError_t)launch_compare(p, grid, s)) != cudaSuccess) return ASMV_ECUDA;
  if ((e = cudaMemcpyAsync(st, dscr + o_stats, (n + 1) * sizeof(StatsDev), cudaMemcpyDeviceToHost,
                           s)) != cudaSuccess)
    return ASMV_ECUDA;
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return ASMV_ECUDA;
  uint32_t err;
  std::memcpy(&err, &st[n], sizeof err);
  if (err & kErrBounds) return ASMV_EBOUNDS;
  if (err) return ASMV_ETIMEOUT;
  std::memcpy(out_host, st, n * sizeof(asmv_stats));
  return ASMV_OK;
}
