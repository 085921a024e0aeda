/*
 * asmv_oracle.c -- the CPU oracle for the differential-oracle hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The
 * product path (the CUDA library) never calls it and shares no code with it:
 * no header, constant, table or helper is common to the two.
 *
 * What it computes, in the paper's terms (AsmEvo, Sec. 3.2 Eq. 1 and
 * Sec. 3.4 "Tier 1" / "Tier 2"):
 *   - Tier 1 guarded input synthesis: every allocation is a low guard band,
 *     a payload and a high guard band; the payload receives deterministic
 *     seeded values, the guard bands a canary byte, so that an out-of-bounds
 *     write shows up as a changed guard byte (Sec. 3.4, Tier 1).
 *   - The equivalence check of Eq. 1 restated per element: floating-point
 *     outputs pass a tolerance test, integer buffers, opaque state and guard
 *     bytes must be bit-exact (the iota term of Eq. 1; Sec. 3.4, Tier 2).
 *     Per region it reports the mismatch count, first mismatching index, the
 *     exact fp64 maximum absolute and relative error over finite pairs and
 *     the count of NaN/Inf-position mismatches.
 *
 * Everything is a plain scalar loop.  Floating point follows the stated
 * operation order with -ffp-contract=off; no fast-math.
 *
 * Readings where the paper is silent (each one is also listed in the design
 * notes):
 *   R1 The random source is Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11,
 *      "Parallel random numbers: as easy as 1, 2, 3").  key = (seed lo, seed
 *      hi); counter = (block lo, block hi, region_id, stream tag 0).
 *   R2 Element generation from Philox words, per distribution (see fill).
 *   R3 Normal values use Box-Muller in fp32 with in-house ln / sincos(2 pi u)
 *      routines, so that CPU and GPU produce identical bytes.
 *   R4 Float predicate: d = |c - r| in fp64 (exact inputs), bound =
 *      atol + rtol*|r| (multiply, then add), mismatch iff d > bound; both NaN
 *      match, same-signed Inf match, any other non-finite pair mismatches and
 *      counts as a NaN/Inf-position mismatch and is excluded from the maxima.
 *   R5 rel = d / |r|; for r == 0 it is 0 when d == 0, else +Inf.
 *   R6 Integer and opaque regions: mismatch iff the bits differ; abs error is
 *      |int(c) - int(r)| and rel error abs/|r| (same r == 0 rule).
 *   R7 first_mismatch is the lowest element index; first_guard_bad the lowest
 *      byte offset from the allocation start (low guard before high guard).
 *   R10 Further stored formats (for captured state of other producers):
 *      OCP FP8 E5M2 (bias 15, Inf and NaN at exponent 31); the "fnuz" FP8
 *      formats E4M3FNUZ (bias 8) and E5M2FNUZ (bias 16), finite only, no
 *      negative zero, 0x80 the only NaN; IEEE binary64; int16 and int64.
 *      Encoding from fp32 rounds to nearest even and saturates finite
 *      overflow and infinities at the largest finite value (fnuz results of
 *      magnitude zero are +0); binary64 values are the exact widening of
 *      the fp32 value.  For binary64, d = RN64(|c - r|) is one rounded
 *      subtraction.  For int64, |c - r| is formed exactly and rounded once
 *      to fp64, and rel = RN64(that / RN64(|r|)).
 *   R12 The 16-bit and 8-bit float formats draw as many Philox bits per
 *      element as they store: one Philox block per 16-byte chunk of payload.
 *      UNIFORM takes a 16-bit (8-bit) fraction per element.  NORMAL is
 *      Box-Muller on one pair per 32 bits (16-bit formats: a 16-bit radius
 *      index and a 16-bit angle index) or per 16 bits (8-bit formats: 8 + 8),
 *      with radius and angle taken from tables whose entries are the
 *      correctly rounded fp32 values of their closed forms (see "narrow
 *      formats" below).  fp32 and binary64 keep R3.
 *
 * Parity pins live in tests/test_oracle_*.py.  The stats of the large
 * perturbed workloads (attention outputs, the 4096-region snapshot, the
 * batched GEMM output) are data-determined: beyond invariants, parity of
 * those totals is unpinned, and the oracle's value is the reference.
 */
#include <stdint.h>
#include <string.h>
#include <math.h>
#include <float.h>

/* ---- dtype and distribution codes (the numbering of the public ABI) ---- */
enum { OD_F32 = 0, OD_BF16 = 1, OD_F16 = 2, OD_F8E4M3 = 3, OD_I32 = 4,
       OD_I8 = 5, OD_U8 = 6, OD_F8E5M2 = 7, OD_F8E4M3FNUZ = 8,
       OD_F8E5M2FNUZ = 9, OD_F64 = 10, OD_I16 = 11, OD_I64 = 12,
       OD_NDTYPES = 13 };
enum { OX_RAW = 0, OX_UNIFORM = 1, OX_NORMAL = 2, OX_INT_RANGE = 3,
       OX_NONE = 4 };

int oracle_dtype_size(int dt) {
  switch (dt) {
    case OD_F32: case OD_I32: return 4;
    case OD_BF16: case OD_F16: case OD_I16: return 2;
    case OD_F8E4M3: case OD_I8: case OD_U8: case OD_F8E5M2: case OD_F8E4M3FNUZ:
    case OD_F8E5M2FNUZ: return 1;
    case OD_F64: case OD_I64: return 8;
    default: return 0;
  }
}

static int is_float_dtype(int dt) {
  return dt <= OD_F8E4M3 || (dt >= OD_F8E5M2 && dt <= OD_F64);
}

/* ======================================================================
 * Philox4x32-10, written from Salmon et al. (SC'11), Sec. 3 / Table 2:
 * with Ma = 0xD2511F53 and Mb = 0xCD9E8D57, one round maps (x0,x1,x2,x3)
 * under key (k0,k1) to
 *   (hi(Mb*x2) ^ x1 ^ k0,  lo(Mb*x2),  hi(Ma*x0) ^ x3 ^ k1,  lo(Ma*x0))
 * where hi/lo are the halves of the 64-bit product.  Ten rounds; the key
 * advances by the Weyl constants (golden ratio and sqrt(3)-1 in 0.32 fixed
 * point) between consecutive rounds.
 * ====================================================================== */
#define PHILOX_M_A 0xD2511F53u
#define PHILOX_M_B 0xCD9E8D57u
#define PHILOX_W_0 0x9E3779B9u
#define PHILOX_W_1 0xBB67AE85u

void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                          uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) { k0 += PHILOX_W_0; k1 += PHILOX_W_1; }
    uint64_t pa = (uint64_t)PHILOX_M_A * (uint64_t)x0;
    uint64_t pb = (uint64_t)PHILOX_M_B * (uint64_t)x2;
    uint32_t pa_hi = (uint32_t)(pa >> 32), pa_lo = (uint32_t)pa;
    uint32_t pb_hi = (uint32_t)(pb >> 32), pb_lo = (uint32_t)pb;
    uint32_t y0 = pb_hi ^ x1 ^ k0;
    uint32_t y1 = pb_lo;
    uint32_t y2 = pa_hi ^ x3 ^ k1;
    uint32_t y3 = pa_lo;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The block b of region `region_id` under `seed` (stream tag 0 = payload). */
static void payload_block(uint64_t seed, uint32_t region_id, uint64_t b,
                          uint32_t w[4]) {
  uint32_t ctr[4] = {(uint32_t)b, (uint32_t)(b >> 32), region_id, 0u};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  oracle_philox4x32_10(ctr, key, w);
}

/* ======================================================================
 * Exact decoders of the stored formats to fp64 (all are exact in fp64).
 * ====================================================================== */
static uint32_t f32_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }
static float bits_f32(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

double oracle_decode_bf16(uint16_t h) {
  return (double)bits_f32((uint32_t)h << 16);
}

double oracle_decode_f16(uint16_t h) {
  int sign = (h >> 15) & 1, ex = (h >> 10) & 31, man = h & 1023;
  double v;
  if (ex == 31) v = man ? NAN : INFINITY;
  else if (ex == 0) v = ldexp((double)man, -24);
  else v = ldexp((double)(1024 + man), ex - 25);
  return sign ? -v : v;
}

/* OCP FP8 E4M3 ("fn" variant): bias 7, no infinities, S.1111.111 is NaN. */
double oracle_decode_f8e4m3(uint8_t b) {
  int sign = (b >> 7) & 1, ex = (b >> 3) & 15, man = b & 7;
  double v;
  if (ex == 15 && man == 7) v = NAN;
  else if (ex == 0) v = ldexp((double)man, -9);
  else v = ldexp((double)(8 + man), ex - 10);
  return sign ? -v : v;
}

/* OCP FP8 E5M2: bias 15, the top byte of an IEEE binary16; exponent field
 * 31 holds Inf (mantissa 0) and NaN. */
double oracle_decode_f8e5m2(uint8_t b) {
  int sign = (b >> 7) & 1, ex = (b >> 2) & 31, man = b & 3;
  double v;
  if (ex == 31) v = man ? NAN : INFINITY;
  else if (ex == 0) v = ldexp((double)man, -16);
  else v = ldexp((double)(4 + man), ex - 17);
  return sign ? -v : v;
}

/* The "fnuz" FP8 formats (finite, no negative zero): every exponent field
 * is finite, and the bit pattern 0x80 (negative zero elsewhere) is the one
 * NaN.  E4M3FNUZ: bias 8, max 240; E5M2FNUZ: bias 16, max 57344. */
double oracle_decode_f8e4m3fnuz(uint8_t b) {
  if (b == 0x80u) return NAN;
  int sign = (b >> 7) & 1, ex = (b >> 3) & 15, man = b & 7;
  double v = (ex == 0) ? ldexp((double)man, -10) : ldexp((double)(8 + man), ex - 11);
  return sign ? -v : v;
}

double oracle_decode_f8e5m2fnuz(uint8_t b) {
  if (b == 0x80u) return NAN;
  int sign = (b >> 7) & 1, ex = (b >> 2) & 31, man = b & 3;
  double v = (ex == 0) ? ldexp((double)man, -17) : ldexp((double)(4 + man), ex - 18);
  return sign ? -v : v;
}

/* Decode element i of a payload of dtype dt to fp64.  Integer types give
 * their (signed or unsigned) integer value. */
static double decode_elem(const uint8_t *p, int dt, uint64_t i) {
  switch (dt) {
    case OD_F32: { uint32_t u; memcpy(&u, p + 4 * i, 4); return (double)bits_f32(u); }
    case OD_BF16: { uint16_t h; memcpy(&h, p + 2 * i, 2); return oracle_decode_bf16(h); }
    case OD_F16: { uint16_t h; memcpy(&h, p + 2 * i, 2); return oracle_decode_f16(h); }
    case OD_F8E4M3: return oracle_decode_f8e4m3(p[i]);
    case OD_I32: { int32_t v; memcpy(&v, p + 4 * i, 4); return (double)v; }
    case OD_I8: return (double)(int8_t)p[i];
    case OD_U8: return (double)p[i];
    case OD_F8E5M2: return oracle_decode_f8e5m2(p[i]);
    case OD_F8E4M3FNUZ: return oracle_decode_f8e4m3fnuz(p[i]);
    case OD_F8E5M2FNUZ: return oracle_decode_f8e5m2fnuz(p[i]);
    case OD_F64: { double d; memcpy(&d, p + 8 * i, 8); return d; }
    case OD_I16: { int16_t v; memcpy(&v, p + 2 * i, 2); return (double)v; }
    case OD_I64: { int64_t v; memcpy(&v, p + 8 * i, 8); return (double)v; }   /* rounded above 2^53 */
    default: return NAN;
  }
}

/* ======================================================================
 * Round-to-nearest-even encoders from fp32, written on integer bits.
 * ====================================================================== */
uint16_t oracle_f32_to_bf16(float f) {
  uint32_t u = f32_bits(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((u >> 16) | 0x0040u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;                 /* carries into the exponent as needed */
  return (uint16_t)(u >> 16);
}

/* Round the positive finite fp32 value with biased exponent field `bexp`
 * and fraction `frac` to a multiple of 2^qe (RNE); returns the multiplier. */
static uint32_t rne_to_quantum(uint32_t bexp, uint32_t frac, int qe) {
  /* value = m24 * 2^(e - 23), e = bexp - 127 (normal) */
  uint32_t m24;
  int e;
  if (bexp == 0) { m24 = frac; e = -126; } else { m24 = frac | 0x800000u; e = (int)bexp - 127; }
  int shift = qe - (e - 23);          /* bits of m24 below the quantum */
  if (shift <= 0) return m24 << (-shift);
  if (shift > 25) return 0;
  uint32_t q = m24 >> shift;
  uint32_t rem = m24 & ((1u << shift) - 1u);
  uint32_t half = 1u << (shift - 1);
  if (rem > half || (rem == half && (q & 1u))) q += 1;
  return q;
}

uint16_t oracle_f32_to_f16(float f) {
  uint32_t u = f32_bits(f);
  uint16_t sign = (uint16_t)((u >> 16) & 0x8000u);
  uint32_t a = u & 0x7FFFFFFFu;
  if (a > 0x7F800000u) return (uint16_t)(sign | 0x7E00u);
  if (a == 0x7F800000u) return (uint16_t)(sign | 0x7C00u);
  uint32_t bexp = a >> 23, frac = a & 0x7FFFFFu;
  int e = (bexp == 0) ? -126 : (int)bexp - 127;
  if (e < -25) return sign;                        /* below half the least subnormal */
  int qe = (e - 10 > -24) ? e - 10 : -24;          /* quantum of binary16 at this magnitude */
  uint32_t q = rne_to_quantum(bexp, frac, qe);
  if (qe == -24) return (uint16_t)(sign | q);     /* subnormal, or rounds up to 2^-14 */
  if (q == 2048) { q = 1024; e += 1; }
  if (e + 15 >= 31) return (uint16_t)(sign | 0x7C00u);
  return (uint16_t)(sign | ((uint32_t)(e + 15) << 10) | (q - 1024));
}

/* fp32 -> an 8-bit float with `eb` exponent bits, `mb` mantissa bits and
 * bias `bias`, round to nearest even.  Finite overflow and infinities
 * saturate to the largest finite value `maxmag` (its bit pattern without
 * sign).  fnuz formats have no negative zero (a result of magnitude zero is
 * +0) and encode NaN as 0x80; the others keep the sign of zero and encode
 * NaN as S.1..1 with every mantissa bit set. */
static uint8_t encode_fp8(float f, int eb, int mb, int bias, uint8_t maxmag, int fnuz) {
  uint32_t u = f32_bits(f);
  uint8_t sign = (uint8_t)((u >> 24) & 0x80u);
  uint32_t a = u & 0x7FFFFFFFu;
  if (a > 0x7F800000u) return fnuz ? 0x80u : (uint8_t)(sign | 0x7Fu);
  uint8_t mag;
  if (a == 0x7F800000u) {
    mag = maxmag;
  } else {
    uint32_t bexp = a >> 23, frac = a & 0x7FFFFFu;
    int e = (bexp == 0) ? -126 : (int)bexp - 127;
    int emin = 1 - bias;                             /* exponent of the least normal */
    int qmin = emin - mb;                            /* quantum of the subnormals */
    if (e < qmin - 1) {
      mag = 0;                                       /* below half the least subnormal */
    } else {
      int qe = (e - mb > qmin) ? e - mb : qmin;
      uint32_t q = rne_to_quantum(bexp, frac, qe);
      uint32_t field;
      if (qe == qmin) {
        field = q;                                   /* subnormal, or rounds up to the least normal */
      } else {
        if (q == (2u << mb)) { q = 1u << mb; e += 1; }
        int ef = e + bias;
        field = (ef > (1 << eb) - 1) ? 0xFFu : (((uint32_t)ef << mb) | (q - (1u << mb)));
      }
      mag = (field > maxmag) ? maxmag : (uint8_t)field;
    }
  }
  if (fnuz && mag == 0) return 0;
  return (uint8_t)(sign | mag);
}

uint8_t oracle_f32_to_f8e5m2(float f) { return encode_fp8(f, 5, 2, 15, 0x7Bu, 0); }
uint8_t oracle_f32_to_f8e4m3fnuz(float f) { return encode_fp8(f, 4, 3, 8, 0x7Fu, 1); }
uint8_t oracle_f32_to_f8e5m2fnuz(float f) { return encode_fp8(f, 5, 2, 16, 0x7Fu, 1); }

/* fp32 -> OCP E4M3: RNE, finite overflow and infinities saturate to +-448,
 * NaN maps to S.1111.111. */
uint8_t oracle_f32_to_f8e4m3(float f) {
  uint32_t u = f32_bits(f);
  uint8_t sign = (uint8_t)((u >> 24) & 0x80u);
  uint32_t a = u & 0x7FFFFFFFu;
  if (a > 0x7F800000u) return (uint8_t)(sign | 0x7Fu);
  if (bits_f32(a) >= 448.0f) return (uint8_t)(sign | 0x7Eu);
  uint32_t bexp = a >> 23, frac = a & 0x7FFFFFu;
  int e = (bexp == 0) ? -126 : (int)bexp - 127;
  if (e < -10) return sign;
  int qe = (e - 3 > -9) ? e - 3 : -9;
  uint32_t q = rne_to_quantum(bexp, frac, qe);
  if (qe == -9) return (uint8_t)(sign | q);
  if (q == 16) { q = 8; e += 1; }
  return (uint8_t)(sign | ((uint32_t)(e + 7) << 3) | (q - 8));
}

/* ======================================================================
 * fp32 Box-Muller pieces.  Every step below is one IEEE fp32 operation
 * (fmaf where written).
 *
 * ln(u), u = k 2^-24, is P. T. P. Tang's table-driven logarithm ("Table-
 * driven implementation of the logarithm function in IEEE floating-point
 * arithmetic", ACM TOMS 16, 1990) with this library's table and series:
 * u = m 2^e with m in [1, 2) and j = round(128 (m-1));
 * with inv_j = round(32768/(128+j))/256 (eight significant bits) the
 * reduction r = m*inv_j - 1 is exact in one fma and |r| < 2^-7; then
 *   ln u = e ln2 + (-ln inv_j) + log1p(r),
 * log1p(r) = r + r^2 (-1/2 + r (1/3 - r/4)), ln 2 and -ln inv_j each split
 * into a head that is a multiple of 2^-9 (so e*head + head is exact) and an
 * fp32 tail.  The table is computed here, in extended precision, from that
 * definition.
 * sin/cos: Taylor coefficients of the stated series, rounded once to fp32.
 * ====================================================================== */
static float C_LN2_HI, C_LN2_LO, C_THIRD, C_S[5], C_C[6];
static float T_INV[129], T_HI[129], T_LO[129];
static int consts_ready = 0;

static void init_consts(void) {
  if (consts_ready) return;
  long double ln2 = logl(2.0L);
  /* Cody-Waite split of ln 2: a short head (9 significant bits) and the rest */
  C_LN2_HI = 355.0f / 512.0f;
  C_LN2_LO = (float)(ln2 - 355.0L / 512.0L);
  C_THIRD = (float)(1.0L / 3.0L);
  for (int j = 0; j <= 128; ++j) {
    int den = 128 + j;
    int I = (32768 + den / 2) / den;              /* round(32768/den); never a tie */
    long double nl = logl(256.0L / (long double)I);
    long double hi = nearbyintl(nl * 512.0L) / 512.0L;
    T_INV[j] = (float)I / 256.0f;
    T_HI[j] = (float)hi;
    T_LO[j] = (float)(nl - hi);
  }
  /* sin(pi/2 r) and cos(pi/2 r): coefficient of r^j is +-(pi/2)^j / j! */
  long double h = acosl(-1.0L) / 2.0L, p = 1.0L, fact = 1.0L;
  long double coef[12];
  for (int j = 0; j < 12; ++j) {
    if (j > 0) { p *= h; fact *= (long double)j; }
    long double c = p / fact;
    if ((j / 2) % 2 == 1) c = -c;      /* signs: + (j=0,1), - (2,3), + (4,5) ... */
    coef[j] = c;
  }
  for (int k = 0; k < 5; ++k) C_S[k] = (float)coef[2 * k + 1];   /* r^1 .. r^9 */
  for (int k = 0; k < 6; ++k) C_C[k] = (float)coef[2 * k];       /* r^0 .. r^10 */
  consts_ready = 1;
}

/* [ln2 head, ln2 tail, 1/3, sin r^1..r^9 (5), cos r^0..r^10 (6)] */
void oracle_boxmuller_consts(float out[14]) {
  init_consts();
  out[0] = C_LN2_HI; out[1] = C_LN2_LO; out[2] = C_THIRD;
  for (int k = 0; k < 5; ++k) out[3 + k] = C_S[k];
  for (int k = 0; k < 6; ++k) out[8 + k] = C_C[k];
}

/* The ln reduction table: out[3j + 0..2] = inv_j, head_j, tail_j. */
void oracle_ln_table(float out[387]) {
  init_consts();
  for (int j = 0; j <= 128; ++j) {
    out[3 * j] = T_INV[j]; out[3 * j + 1] = T_HI[j]; out[3 * j + 2] = T_LO[j];
  }
}

/* ln(k * 2^-24) for k in [1, 2^24], in fp32. */
float oracle_ln_u24(uint32_t k) {
  init_consts();
  float u = (float)k * 0x1p-24f;                 /* exact */
  uint32_t b = f32_bits(u);
  int e = (int)(b >> 23) - 127;
  uint32_t mb = b & 0x7FFFFFu;
  float m = bits_f32(mb | 0x3F800000u);          /* [1, 2) */
  uint32_t j = (mb + (1u << 15)) >> 16;          /* round(128 (m - 1)), 0..128 */
  float r = fmaf(m, T_INV[j], -1.0f);            /* exact */
  float r2 = r * r;
  float p = fmaf(r, -0.25f, C_THIRD);
  p = fmaf(r, p, -0.5f);
  float lp = fmaf(r2, p, r);
  float ef = (float)e;
  float hi = fmaf(ef, C_LN2_HI, T_HI[j]);        /* exact */
  float lo = fmaf(ef, C_LN2_LO, T_LO[j]);
  return hi + (lo + lp);
}

/* sin and cos of 2*pi*k*2^-24 for k in [0, 2^24), in fp32. */
void oracle_sincos_2pi_u24(uint32_t k, float *sn_out, float *cs_out) {
  init_consts();
  uint32_t q = (k + (1u << 21)) >> 22;             /* nearest quarter turn, 0..4 */
  int32_t ri = (int32_t)k - (int32_t)(q << 22);    /* [-2^21, 2^21) */
  float r = (float)ri * 0x1p-22f;                  /* angle = (q + r) * pi/2 */
  float r2 = r * r;
  float sp = fmaf(r2, C_S[4], C_S[3]);
  sp = fmaf(r2, sp, C_S[2]);
  sp = fmaf(r2, sp, C_S[1]);
  sp = fmaf(r2, sp, C_S[0]);
  float sn = r * sp;
  float cp = fmaf(r2, C_C[5], C_C[4]);
  cp = fmaf(r2, cp, C_C[3]);
  cp = fmaf(r2, cp, C_C[2]);
  cp = fmaf(r2, cp, C_C[1]);
  float cs = fmaf(r2, cp, C_C[0]);
  switch (q & 3u) {
    case 0: *sn_out = sn;  *cs_out = cs;  break;
    case 1: *sn_out = cs;  *cs_out = -sn; break;
    case 2: *sn_out = -sn; *cs_out = -cs; break;
    default: *sn_out = -cs; *cs_out = sn; break;
  }
}

/* The two standard normals of Box-Muller from two Philox words. */
void oracle_boxmuller(uint32_t w0, uint32_t w1, float *z0, float *z1) {
  float l = oracle_ln_u24((w0 >> 8) + 1u);
  float rho = sqrtf(-2.0f * l);
  float sn, cs;
  oracle_sincos_2pi_u24(w1 >> 8, &sn, &cs);
  *z0 = rho * cs;
  *z1 = rho * sn;
}

/* ======================================================================
 * Narrow formats (reading R12): Box-Muller for the 16-bit and 8-bit floats.
 *
 * 16-bit formats, one pair per 32-bit word w:
 *   radius  k = w mod 2^16, u = (k + 1/2) 2^-16.  With d = 1 when u > 1/2,
 *           x = u (d = 0) or x = 1 - u (d = 1) is K 2^-17 for the odd
 *           K = 2t + 1, t = (k mod 2^15) xor (d ? 2^15 - 1 : 0).  The fp32
 *           value F = K 2^(16 d) is exact; write F = 2^E m with m in [1, 2)
 *           and take cell c = 16 E + floor(16 (m - 1)), 0 <= c < 512.  Then
 *             rho = fma(F, A_c, B_c)
 *           where, for the cell's mantissa interval [m0, m0 + 1/16) and
 *           g(m) = sqrt(-2 ln y(m)), y(m) = m 2^(e-17) (d = 0) or
 *           1 - m 2^(e-17) (d = 1), e = E - 16 d, the secant slope is
 *           S = 16 (g(m0 + 1/16) - g(m0)), A_c = RN32(S 2^-E) and
 *           B_c = RN32(g(m0) - S m0): the chord of rho over the cell.
 *   angle   a = w div 2^16, theta = 2 pi (a + 1/2) / 65536.  With
 *           j = a div 256, n = a mod 256, phi_j = 2 pi (j + 1/2) / 256 and
 *           (S_j, C_j) = (RN32(sin phi_j), RN32(cos phi_j)):
 *             delta = fma(n - 128, c16, c16 / 2),  c16 = RN32(2 pi / 65536)
 *             sin ~ fma(C_j, delta, S_j),  cos ~ fma(-S_j, delta, C_j)
 *           (the first-order rotation of phi_j by delta = theta - phi_j).
 *   values  rs = RN32(rho * std); v0 = fma(rs, cos, mean),
 *           v1 = fma(rs, sin, mean).
 * 8-bit formats, one pair per 16-bit half h of a word (low half first):
 *   rho = R8[h mod 256] = RN32(sqrt(-2 ln((k + 1/2) / 256))) and the angle
 *   table entry j = h div 256 itself, (sin, cos) = (S_j, C_j); the values
 *   as above.
 * ====================================================================== */
static float N16_A[512], N16_B[512], T_SIN[256], T_COS[256], R8_RHO[256];
static float C16_STEP;
static int narrow_ready = 0;

static long double nr_g(long double m, int e, int d) {
  long double y = ldexpl(m, e - 17);
  if (d) y = 1.0L - y;
  return sqrtl(-2.0L * logl(y));
}

static void init_narrow(void) {
  if (narrow_ready) return;
  long double pi = acosl(-1.0L);
  for (int E = 0; E < 32; ++E) {
    int d = E >= 16, e = E - 16 * d;
    for (int i = 0; i < 16; ++i) {
      long double m0 = 1.0L + i / 16.0L, m1 = m0 + 1.0L / 16.0L;
      long double g0 = nr_g(m0, e, d), g1 = nr_g(m1, e, d);
      long double S = 16.0L * (g1 - g0);
      N16_A[16 * E + i] = (float)ldexpl(S, -E);
      N16_B[16 * E + i] = (float)(g0 - S * m0);
    }
  }
  for (int j = 0; j < 256; ++j) {
    long double phi = 2.0L * pi * (j + 0.5L) / 256.0L;
    T_SIN[j] = (float)sinl(phi);
    T_COS[j] = (float)cosl(phi);
    R8_RHO[j] = (float)sqrtl(-2.0L * logl((j + 0.5L) / 256.0L));
  }
  C16_STEP = (float)(2.0L * pi / 65536.0L);
  narrow_ready = 1;
}

/* out: A[512], B[512], sin[256], cos[256], R8[256], c16 */
void oracle_narrow_tables(float *out) {
  init_narrow();
  for (int c = 0; c < 512; ++c) { out[c] = N16_A[c]; out[512 + c] = N16_B[c]; }
  for (int j = 0; j < 256; ++j) {
    out[1024 + j] = T_SIN[j]; out[1280 + j] = T_COS[j]; out[1536 + j] = R8_RHO[j];
  }
  out[1792] = C16_STEP;
}

/* The radius of a 16-bit pair, k in [0, 2^16). */
float oracle_radius16(uint32_t k) {
  init_narrow();
  uint32_t d = (k >> 15) & 1u;
  uint32_t t = (k & 0x7FFFu) ^ (d ? 0x7FFFu : 0u);
  float F = (float)(2u * t + 1u) * (d ? 65536.0f : 1.0f);     /* exact */
  uint32_t b = f32_bits(F);
  int E = (int)(b >> 23) - 127;
  int c = 16 * E + (int)((b >> 19) & 15u);
  return fmaf(F, N16_A[c], N16_B[c]);
}

/* sin and cos of the angle of a 16-bit pair, a in [0, 2^16). */
void oracle_angle16(uint32_t a, float *sn, float *cs) {
  init_narrow();
  uint32_t j = a >> 8, n = a & 255u;
  float delta = fmaf((float)n - 128.0f, C16_STEP, C16_STEP * 0.5f);
  *sn = fmaf(T_COS[j], delta, T_SIN[j]);
  *cs = fmaf(-T_SIN[j], delta, T_COS[j]);
}

/* v0, v1 of the pair drawn from word w (16-bit formats). */
void oracle_normal16(uint32_t w, float mean, float sd, float *v0, float *v1) {
  float rho = oracle_radius16(w & 0xFFFFu);
  float sn, cs;
  oracle_angle16(w >> 16, &sn, &cs);
  float rs = rho * sd;
  *v0 = fmaf(rs, cs, mean);
  *v1 = fmaf(rs, sn, mean);
}

/* v0, v1 of the pair drawn from the 16-bit half h (8-bit formats). */
void oracle_normal8(uint32_t h, float mean, float sd, float *v0, float *v1) {
  init_narrow();
  float rho = R8_RHO[h & 255u];
  uint32_t j = (h >> 8) & 255u;
  float rs = rho * sd;
  *v0 = fmaf(rs, T_COS[j], mean);
  *v1 = fmaf(rs, T_SIN[j], mean);
}

/* ======================================================================
 * Tier 1 fill.
 * Element i of a payload, per distribution:
 *   RAW       payload byte j = byte (j mod 16) of block (j div 16); a block
 *             is its four words in order, each little-endian.
 *   INT_RANGE word (i mod 4) of block (i div 4): lo + ((w * (hi-lo)) >> 32)
 *   UNIFORM   fp32 / binary64: word (i mod 4) of block (i div 4),
 *             f = (w >> 8) 2^-24; 16-bit formats: half (i mod 2) of word
 *             (i mod 8) div 2 of block (i div 8), f = h 2^-16; 8-bit formats:
 *             byte (i mod 4) of word (i mod 16) div 4 of block (i div 16),
 *             f = b 2^-8.  v = lo + f*(hi - lo) in fp32, then RNE
 *   NORMAL    fp32 / binary64: block i div 4 gives two pairs (words 0,1 and
 *             2,3); element 4b+2j+t is z_t of pair j, v = mean + std*z in
 *             fp32, then RNE.  16-bit formats: element i is v_(i mod 2) of
 *             the pair of word (i mod 8) div 2 of block (i div 8); 8-bit
 *             formats: v_(i mod 2) of the pair of half (i mod 4) div 2 of
 *             word (i mod 16) div 4 of block (i div 16) (narrow formats
 *             above)
 *   NONE      payload untouched
 * ====================================================================== */
static void store_float(uint8_t *p, int dt, uint64_t i, float v) {
  switch (dt) {
    case OD_F32: { uint32_t u = f32_bits(v); memcpy(p + 4 * i, &u, 4); break; }
    case OD_BF16: { uint16_t h = oracle_f32_to_bf16(v); memcpy(p + 2 * i, &h, 2); break; }
    case OD_F16: { uint16_t h = oracle_f32_to_f16(v); memcpy(p + 2 * i, &h, 2); break; }
    case OD_F8E4M3: p[i] = oracle_f32_to_f8e4m3(v); break;
    case OD_F8E5M2: p[i] = oracle_f32_to_f8e5m2(v); break;
    case OD_F8E4M3FNUZ: p[i] = oracle_f32_to_f8e4m3fnuz(v); break;
    case OD_F8E5M2FNUZ: p[i] = oracle_f32_to_f8e5m2fnuz(v); break;
    case OD_F64: { double d = (double)v; memcpy(p + 8 * i, &d, 8); break; }   /* exact */
  }
}

static void store_int(uint8_t *p, int dt, uint64_t i, int64_t v) {
  switch (dt) {
    case OD_I32: { int32_t x = (int32_t)v; memcpy(p + 4 * i, &x, 4); break; }
    case OD_I8: case OD_U8: p[i] = (uint8_t)v; break;
    case OD_I16: { int16_t x = (int16_t)v; memcpy(p + 2 * i, &x, 2); break; }
    case OD_I64: memcpy(p + 8 * i, &v, 8); break;
  }
}

/* Fill elements [i0, i1) of the payload starting at `payload`.  Returns 0,
 * or -1 for a distribution that does not apply to the dtype. */
int oracle_fill_payload(uint8_t *payload, int dt, int dist, uint64_t i0,
                        uint64_t i1, uint32_t region_id, double p0, double p1,
                        uint64_t seed) {
  int sz = oracle_dtype_size(dt);
  if (sz == 0) return -1;
  if (dist == OX_NONE) return 0;
  if (dist == OX_RAW) {
    for (uint64_t j = i0 * (uint64_t)sz; j < i1 * (uint64_t)sz; ++j) {
      uint32_t w[4];
      payload_block(seed, region_id, j / 16, w);
      uint32_t word = w[(j % 16) / 4];
      payload[j] = (uint8_t)(word >> (8 * (j % 4)));
    }
    return 0;
  }
  if (dist == OX_INT_RANGE) {
    if (is_float_dtype(dt)) return -1;
    int64_t lo = (int64_t)p0, hi = (int64_t)p1;
    uint64_t span = (uint64_t)(hi - lo);
    for (uint64_t i = i0; i < i1; ++i) {
      uint32_t w[4];
      payload_block(seed, region_id, i / 4, w);
      uint64_t off = ((uint64_t)w[i % 4] * span) >> 32;
      store_int(payload, dt, i, lo + (int64_t)off);
    }
    return 0;
  }
  if (!is_float_dtype(dt)) return -1;
  if (dist == OX_UNIFORM) {
    float lo = (float)p0, hi = (float)p1;
    float width = hi - lo;
    for (uint64_t i = i0; i < i1; ++i) {
      uint32_t w[4];
      float f;
      if (sz == 2) {
        payload_block(seed, region_id, i / 8, w);
        f = (float)((w[(i % 8) / 2] >> (16 * (i % 2))) & 0xFFFFu) * 0x1p-16f;
      } else if (sz == 1) {
        payload_block(seed, region_id, i / 16, w);
        f = (float)((w[(i % 16) / 4] >> (8 * (i % 4))) & 0xFFu) * 0x1p-8f;
      } else {
        payload_block(seed, region_id, i / 4, w);
        f = (float)(w[i % 4] >> 8) * 0x1p-24f;
      }
      float v = lo + f * width;
      store_float(payload, dt, i, v);
    }
    return 0;
  }
  if (dist == OX_NORMAL && sz == 2) {
    float mean = (float)p0, sd = (float)p1;
    for (uint64_t i = i0; i < i1; ++i) {
      uint32_t w[4];
      payload_block(seed, region_id, i / 8, w);
      float v0, v1;
      oracle_normal16(w[(i % 8) / 2], mean, sd, &v0, &v1);
      store_float(payload, dt, i, (i % 2 == 0) ? v0 : v1);
    }
    return 0;
  }
  if (dist == OX_NORMAL && sz == 1) {
    float mean = (float)p0, sd = (float)p1;
    for (uint64_t i = i0; i < i1; ++i) {
      uint32_t w[4];
      payload_block(seed, region_id, i / 16, w);
      uint32_t h = (w[(i % 16) / 4] >> (16 * ((i % 4) / 2))) & 0xFFFFu;
      float v0, v1;
      oracle_normal8(h, mean, sd, &v0, &v1);
      store_float(payload, dt, i, (i % 2 == 0) ? v0 : v1);
    }
    return 0;
  }
  if (dist == OX_NORMAL) {
    float mean = (float)p0, sd = (float)p1;
    for (uint64_t i = i0; i < i1; ++i) {
      uint32_t w[4];
      payload_block(seed, region_id, i / 4, w);
      unsigned pair = (unsigned)((i % 4) / 2);
      float z0, z1;
      oracle_boxmuller(w[2 * pair], w[2 * pair + 1], &z0, &z1);
      float z = (i % 2 == 0) ? z0 : z1;
      float v = mean + sd * z;
      store_float(payload, dt, i, v);
    }
    return 0;
  }
  return -1;
}

/* Guard bands: [alloc, alloc+glo) and [alloc+glo+payload_bytes, +ghi). */
void oracle_fill_guards(uint8_t *alloc, uint64_t payload_bytes, uint32_t glo,
                        uint32_t ghi, uint8_t canary) {
  for (uint64_t j = 0; j < glo; ++j) alloc[j] = canary;
  uint8_t *hi = alloc + glo + payload_bytes;
  for (uint64_t j = 0; j < ghi; ++j) hi[j] = canary;
}

/* Count guard bytes differing from the canary; first bad offset from alloc
 * (UINT64_MAX when none). */
void oracle_guard_check(const uint8_t *alloc, uint64_t payload_bytes,
                        uint32_t glo, uint32_t ghi, uint8_t canary,
                        uint64_t *bad_out, uint64_t *first_out) {
  uint64_t bad = 0, first = UINT64_MAX;
  for (uint64_t j = 0; j < glo; ++j)
    if (alloc[j] != canary) { ++bad; if (first == UINT64_MAX) first = j; }
  uint64_t base = (uint64_t)glo + payload_bytes;
  for (uint64_t j = 0; j < ghi; ++j)
    if (alloc[base + j] != canary) { ++bad; if (first == UINT64_MAX) first = base + j; }
  *bad_out = bad;
  *first_out = first;
}

/* ======================================================================
 * The per-element equivalence predicate and per-region statistics.
 * ====================================================================== */
typedef struct {
  uint64_t mismatches;
  uint64_t first_mismatch;
  double max_abs_err;
  double max_rel_err;
  uint64_t nonfinite_mismatches;
} oracle_stats;

/* Compare elements [i0, i1) of two payloads of dtype dt.  Indices in the
 * result are absolute element indices. */
void oracle_compare_range(const uint8_t *ref, const uint8_t *cand, int dt,
                          uint64_t i0, uint64_t i1, double atol, double rtol,
                          oracle_stats *out) {
  oracle_stats st = {0, UINT64_MAX, 0.0, 0.0, 0};
  int sz = oracle_dtype_size(dt);
  for (uint64_t i = i0; i < i1; ++i) {
    int mismatch;
    double abs_err = 0.0, rel_err = 0.0;
    int finite_pair = 1;
    if (!is_float_dtype(dt) && dt == OD_I64) {
      /* |c - r| formed exactly in 128 bits, then rounded once; |r| rounded once */
      int64_t r, c;
      memcpy(&r, ref + 8 * i, 8);
      memcpy(&c, cand + 8 * i, 8);
      mismatch = r != c;
      __int128 dd = (__int128)c - (__int128)r;
      if (dd < 0) dd = -dd;
      abs_err = (double)(unsigned __int128)dd;
      if (r != 0) rel_err = abs_err / fabs((double)r);
      else rel_err = (abs_err == 0.0) ? 0.0 : INFINITY;
    } else if (!is_float_dtype(dt)) {
      mismatch = memcmp(ref + (uint64_t)sz * i, cand + (uint64_t)sz * i, (size_t)sz) != 0;
      double r = decode_elem(ref, dt, i), c = decode_elem(cand, dt, i);
      abs_err = fabs(c - r);                         /* exact: |c - r| < 2^33 */
      if (r != 0.0) rel_err = abs_err / fabs(r);
      else rel_err = (abs_err == 0.0) ? 0.0 : INFINITY;
    } else {
      double r = decode_elem(ref, dt, i), c = decode_elem(cand, dt, i);
      if (isnan(r) || isnan(c) || isinf(r) || isinf(c)) {
        finite_pair = 0;
        if (isnan(r) && isnan(c)) mismatch = 0;
        else if (isinf(r) && isinf(c) && (signbit(r) == signbit(c))) mismatch = 0;
        else { mismatch = 1; st.nonfinite_mismatches += 1; }
      } else {
        double d = fabs(c - r);
        double bound = atol + rtol * fabs(r);
        mismatch = d > bound;
        abs_err = d;
        if (r != 0.0) rel_err = d / fabs(r);
        else rel_err = (d == 0.0) ? 0.0 : INFINITY;
      }
    }
    if (mismatch) {
      st.mismatches += 1;
      if (st.first_mismatch == UINT64_MAX) st.first_mismatch = i;
    }
    if (finite_pair) {
      if (abs_err > st.max_abs_err) st.max_abs_err = abs_err;
      if (rel_err > st.max_rel_err) st.max_rel_err = rel_err;
    }
  }
  *out = st;
}

/* Per-region result in the 8-field layout: mismatches, first_mismatch,
 * max_abs_err, max_rel_err, nonfinite_mismatches, guard_bad_bytes,
 * first_guard_bad, ref_guard_bad_bytes. */
typedef struct {
  uint64_t mismatches;
  uint64_t first_mismatch;
  double max_abs_err;
  double max_rel_err;
  uint64_t nonfinite_mismatches;
  uint64_t guard_bad_bytes;
  uint64_t first_guard_bad;
  uint64_t ref_guard_bad_bytes;
} oracle_region_stats;

void oracle_compare_region(const uint8_t *ref_alloc, uint32_t ref_glo,
                           uint32_t ref_ghi, uint8_t ref_canary,
                           const uint8_t *cand_alloc, uint32_t cand_glo,
                           uint32_t cand_ghi, uint8_t cand_canary,
                           uint64_t n_elems, int dt, double atol, double rtol,
                           oracle_region_stats *out) {
  uint64_t bytes = n_elems * (uint64_t)oracle_dtype_size(dt);
  oracle_stats st;
  oracle_compare_range(ref_alloc + ref_glo, cand_alloc + cand_glo, dt, 0,
                       n_elems, atol, rtol, &st);
  uint64_t gbad, gfirst, rbad, rfirst;
  oracle_guard_check(cand_alloc, bytes, cand_glo, cand_ghi, cand_canary, &gbad, &gfirst);
  oracle_guard_check(ref_alloc, bytes, ref_glo, ref_ghi, ref_canary, &rbad, &rfirst);
  out->mismatches = st.mismatches;
  out->first_mismatch = st.first_mismatch;
  out->max_abs_err = st.max_abs_err;
  out->max_rel_err = st.max_rel_err;
  out->nonfinite_mismatches = st.nonfinite_mismatches;
  out->guard_bad_bytes = gbad;
  out->first_guard_bad = gfirst;
  out->ref_guard_bad_bytes = rbad;
}

/* ======================================================================
 * Tier 2 replay restore (Sec. 3.4, Tier 2): a region is put back into its
 * captured pre-dispatch state -- the captured payload bytes, and the canary
 * in both guard bands -- before each replay.
 * ====================================================================== */
void oracle_restore_region(uint8_t *alloc, uint64_t payload_bytes, uint32_t glo, uint32_t ghi,
                           uint8_t canary, const uint8_t *captured) {
  oracle_fill_guards(alloc, payload_bytes, glo, ghi, canary);
  memcpy(alloc + glo, captured, payload_bytes);
}

/* ======================================================================
 * Eq. 1 aggregate terms.  The cosine c_x = cos(K'(x), O(x)) of a float
 * region is built from three sums over its elements:
 *   S_rc = sum r*c,   S_rr = sum r*r,   S_cc = sum c*c.
 * Readings (the paper gives the formula only):
 *   R8 Each sum takes the elements whose own term is finite: S_rc the
 *      pairs with both values finite, S_rr the finite r, S_cc the finite c.
 *      (Non-finite values are judged by the NaN/Inf rule R4; wherever their
 *      positions agree, the three index sets coincide.)
 *   R9 The sums are exact, then rounded once to fp64 (nearest, ties to
 *      even): every decoded value has at most 24 significant bits, so each
 *      product is exact in fp64, and the products are added here without
 *      rounding, into a fixed-point integer of OEQ_DIGITS signed 64-bit
 *      digits, digit k weighing 2^(32 k + OEQ_BASE).  The final rounding is
 *      done by the caller from the digits.
 * The range covers every product of two fp32 values (2^-298 .. 2^256) with
 * 2^64 of headroom for the sum.  Binary64 products need 106 bits: those
 * regions are summed by oracle_eq64_sums_range (R11) and return zeros here.
 * ====================================================================== */
#define OEQ_DIGITS 20
#define OEQ_BASE (-320)

/* Carry-propagate: digits 0 .. OEQ_DIGITS-2 end in [0, 2^32), the top digit
 * keeps the sign. */
static void eq_normalize(int64_t *acc) {
  for (int k = 0; k < OEQ_DIGITS - 1; ++k) {
    int64_t carry = acc[k] >> 32;          /* floor division by 2^32 */
    acc[k] -= carry * 4294967296LL;
    acc[k + 1] += carry;
  }
}

/* acc += p, for p an exact fp64 product; returns nothing, exact. */
static void eq_add(int64_t *acc, double p) {
  if (p == 0.0) return;
  int e;
  double f = frexp(fabs(p), &e);                   /* |p| = f 2^e, f in [0.5, 1) */
  uint64_t m = (uint64_t)ldexp(f, 53);             /* exact: 53-bit integer */
  int lsb = e - 53;                                /* |p| = m 2^lsb */
  while ((m & 1u) == 0) { m >>= 1; ++lsb; }
  int pos = lsb - OEQ_BASE;                        /* >= 22 for any fp32 product */
  int q = pos / 32, b = pos % 32;
  /* m 2^b spans at most three 32-bit digits */
  uint64_t lo = (m << b) & 0xFFFFFFFFu;
  uint64_t mid = (b == 0) ? (m >> 32) : ((m >> (32 - b)) & 0xFFFFFFFFu);
  uint64_t hi = (b == 0) ? 0 : (m >> (64 - b));
  int64_t sg = (p < 0.0) ? -1 : 1;
  acc[q] += sg * (int64_t)lo;
  acc[q + 1] += sg * (int64_t)mid;
  acc[q + 2] += sg * (int64_t)hi;
}

/* The three sums over elements [i0, i1) of two payloads of float dtype dt,
 * as normalized digits: out[0..D) = S_rc, out[D..2D) = S_rr,
 * out[2D..3D) = S_cc.  Integer and opaque dtypes give zeros. */
void oracle_eq_sums_range(const uint8_t *ref, const uint8_t *cand, int dt,
                          uint64_t i0, uint64_t i1, int64_t *out) {
  int64_t *rc = out, *rr = out + OEQ_DIGITS, *cc = out + 2 * OEQ_DIGITS;
  for (int k = 0; k < 3 * OEQ_DIGITS; ++k) out[k] = 0;
  if (!is_float_dtype(dt) || dt == OD_F64) return;   /* fp64 products are not exact in fp64 */
  uint64_t since = 0;
  for (uint64_t i = i0; i < i1; ++i) {
    double r = decode_elem(ref, dt, i), c = decode_elem(cand, dt, i);
    if (isfinite(r) && isfinite(c)) eq_add(rc, r * c);
    if (isfinite(r)) eq_add(rr, r * r);
    if (isfinite(c)) eq_add(cc, c * c);
    if (++since == (1u << 20)) {     /* each digit grows by < 2^32 per add */
      eq_normalize(rc); eq_normalize(rr); eq_normalize(cc);
      since = 0;
    }
  }
  eq_normalize(rc); eq_normalize(rr); eq_normalize(cc);
}

int oracle_eq_digits(void) { return OEQ_DIGITS; }
int oracle_eq_base(void) { return OEQ_BASE; }

/* ======================================================================
 * Eq. 1 sums of binary64 regions (R9 widened to binary64).
 *   R11 A finite binary64 value is +-m 2^e with m an integer below 2^53
 *       and e >= -1074, so a product of two is +-M 2^E with M = m_r m_c
 *       below 2^106 and E >= -2148, and its magnitude is below 2^2048.
 *       The sums are kept exactly in O64_DIGITS signed 64-bit digits, digit
 *       k weighing 2^(32 k + O64_BASE): 2^-2148 .. 2^2048 and 2^64 of
 *       headroom need 134 digits.  The caller rounds them (gradual
 *       underflow and overflow to infinity included) and forms the cosine.
 * ====================================================================== */
#define O64_DIGITS 136
#define O64_BASE (-2148)

static void eq64_normalize(int64_t *acc) {
  for (int k = 0; k < O64_DIGITS - 1; ++k) {
    int64_t carry = acc[k] >> 32;          /* floor division by 2^32 */
    acc[k] -= carry * 4294967296LL;
    acc[k + 1] += carry;
  }
}

/* |x| = m 2^e with m odd, for finite non-zero x; m = 0 for zeros and
 * non-finite x. */
static void eq64_split(double x, uint64_t *m, int *e) {
  *m = 0;
  *e = 0;
  if (x == 0.0 || !isfinite(x)) return;
  int ex;
  double f = frexp(fabs(x), &ex);                  /* |x| = f 2^ex, f in [0.5, 1) */
  uint64_t mm = (uint64_t)ldexp(f, 53);            /* exact: 53-bit integer */
  int ee = ex - 53;
  while ((mm & 1u) == 0) { mm >>= 1; ++ee; }       /* now ee >= -1074 */
  *m = mm;
  *e = ee;
}

/* Bits lo .. lo + 31 of M as an integer (lo may be negative: low bits 0). */
static uint64_t eq64_bits(unsigned __int128 M, int lo) {
  if (lo >= 128) return 0;
  if (lo < 0) return (uint64_t)((M << -lo) & 0xFFFFFFFFu);
  return (uint64_t)((M >> lo) & 0xFFFFFFFFu);
}

/* acc += (-1)^neg m1 m2 2^(e1 + e2), exactly. */
static void eq64_add(int64_t *acc, int neg, uint64_t m1, int e1, uint64_t m2, int e2) {
  if (m1 == 0 || m2 == 0) return;
  unsigned __int128 M = (unsigned __int128)m1 * m2;      /* < 2^106 */
  int pos = e1 + e2 - O64_BASE;                          /* >= 0 */
  int q = pos / 32, b = pos % 32;
  /* M 2^pos = sum over k of (bits 32k - b .. 32k - b + 31 of M) 2^(32 (q + k)) */
  for (int k = 0; k < 5; ++k) {
    int64_t dig = (int64_t)eq64_bits(M, 32 * k - b);
    acc[q + k] += neg ? -dig : dig;
  }
}

/* The three sums over elements [i0, i1) of two binary64 payloads, as
 * normalized digits: out[0..D) = S_rc, out[D..2D) = S_rr, out[2D..3D) =
 * S_cc, D = O64_DIGITS. */
void oracle_eq64_sums_range(const uint8_t *ref, const uint8_t *cand, uint64_t i0, uint64_t i1,
                            int64_t *out) {
  int64_t *rc = out, *rr = out + O64_DIGITS, *cc = out + 2 * O64_DIGITS;
  for (int k = 0; k < 3 * O64_DIGITS; ++k) out[k] = 0;
  uint64_t since = 0;
  for (uint64_t i = i0; i < i1; ++i) {
    double r = decode_elem(ref, OD_F64, i), c = decode_elem(cand, OD_F64, i);
    uint64_t mr, mc;
    int er, ec;
    eq64_split(r, &mr, &er);
    eq64_split(c, &mc, &ec);
    int nr = signbit(r) != 0, nc = signbit(c) != 0;
    if (isfinite(r) && isfinite(c)) eq64_add(rc, nr != nc, mr, er, mc, ec);
    if (isfinite(r)) eq64_add(rr, 0, mr, er, mr, er);
    if (isfinite(c)) eq64_add(cc, 0, mc, ec, mc, ec);
    if (++since == (1u << 20)) {     /* each digit grows by < 2^32 per add */
      eq64_normalize(rc); eq64_normalize(rr); eq64_normalize(cc);
      since = 0;
    }
  }
  eq64_normalize(rc); eq64_normalize(rr); eq64_normalize(cc);
}

int oracle_eq64_digits(void) { return O64_DIGITS; }
int oracle_eq64_base(void) { return O64_BASE; }

/* ======================================================================
 * Batch entry points for the tests (plain loops over the functions above).
 * ====================================================================== */
void oracle_philox_many(const uint32_t *ctr, const uint32_t *key, uint64_t n,
                        uint32_t *out) {
  for (uint64_t i = 0; i < n; ++i)
    oracle_philox4x32_10(ctr + 4 * i, key + 2 * i, out + 4 * i);
}

void oracle_ln_u24_many(const uint32_t *k, uint64_t n, float *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_ln_u24(k[i]);
}

void oracle_sincos_2pi_u24_many(const uint32_t *k, uint64_t n, float *sn,
                                float *cs) {
  for (uint64_t i = 0; i < n; ++i) oracle_sincos_2pi_u24(k[i], sn + i, cs + i);
}

void oracle_boxmuller_many(const uint32_t *w0, const uint32_t *w1, uint64_t n,
                           float *z0, float *z1) {
  for (uint64_t i = 0; i < n; ++i) oracle_boxmuller(w0[i], w1[i], z0 + i, z1 + i);
}

void oracle_radius16_many(const uint32_t *k, uint64_t n, float *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = oracle_radius16(k[i]);
}

void oracle_angle16_many(const uint32_t *a, uint64_t n, float *sn, float *cs) {
  for (uint64_t i = 0; i < n; ++i) oracle_angle16(a[i], &sn[i], &cs[i]);
}

void oracle_normal16_many(const uint32_t *w, uint64_t n, float mean, float sd, float *v0,
                          float *v1) {
  for (uint64_t i = 0; i < n; ++i) oracle_normal16(w[i], mean, sd, &v0[i], &v1[i]);
}

void oracle_normal8_many(const uint32_t *h, uint64_t n, float mean, float sd, float *v0,
                         float *v1) {
  for (uint64_t i = 0; i < n; ++i) oracle_normal8(h[i], mean, sd, &v0[i], &v1[i]);
}

void oracle_encode_many(const float *x, uint64_t n, int dt, uint8_t *out) {
  for (uint64_t i = 0; i < n; ++i) store_float(out, dt, i, x[i]);
}

void oracle_decode_many(const uint8_t *p, uint64_t n, int dt, double *out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = decode_elem(p, dt, i);
}
