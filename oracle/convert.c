/*
 * convert.c -- CPU oracle of the dtype-correct value conversion applied when
 * test data are loaded (scaffold helpers of Sec. 4.1.2; the float-only
 * loading defect of Sec. 5.2.3).  TEST INFRASTRUCTURE ONLY (see oracle.h).
 *
 * Written from the definitions, one element at a time: each source element
 * is decoded into an exact value (sign, integer magnitude, power of two), and
 * that value is rounded once, to nearest with ties to even, on the grid of
 * the target format -- the textbook IEEE-754 conversion.  No floating-point
 * instruction takes part in the rounding, so the result does not depend on
 * the host's conversion instructions.
 */
#include <string.h>

#include "oracle.h"

typedef unsigned __int128 u128;

int or_dtype_bytes(int dtype) {
  switch (dtype) {
    case OR_F32: case OR_I32: case OR_U32: return 4;
    case OR_F16: case OR_BF16: case OR_I16: case OR_U16: return 2;
    case OR_I64: case OR_U64: case OR_F64: return 8;
    case OR_U8: case OR_I8: return 1;
    default: return 0;
  }
}

static int is_float(int t) { return t == OR_F32 || t == OR_F16 || t == OR_BF16 || t == OR_F64; }

/* IEEE binary formats: precision p (with the hidden bit), exponent bits, bias */
typedef struct { int p, ebits, bias; } fmt;

static fmt format_of(int t) {
  switch (t) {
    case OR_F16: return (fmt){11, 5, 15};
    case OR_BF16: return (fmt){8, 8, 127};
    case OR_F32: return (fmt){24, 8, 127};
    default: return (fmt){53, 11, 1023}; /* OR_F64 */
  }
}

/* An exact value: NaN, +-Inf, or (-1)^neg * mag * 2^exp. */
typedef struct {
  int nan, inf, neg;
  uint64_t mag;
  int exp;
} value;

static uint64_t load_bits(const uint8_t* p, int bytes) {
  uint64_t v = 0;
  memcpy(&v, p, (size_t)bytes); /* little-endian hosts only (x86-64, aarch64) */
  return v;
}

static value decode(int t, uint64_t bits) {
  value v = {0, 0, 0, 0, 0};
  if (!is_float(t)) {
    int64_t s = 0;
    switch (t) {
      case OR_U8: v.mag = (uint8_t)bits; return v;
      case OR_U16: v.mag = (uint16_t)bits; return v;
      case OR_U32: v.mag = (uint32_t)bits; return v;
      case OR_U64: v.mag = bits; return v;
      case OR_I8: s = (int8_t)(uint8_t)bits; break;
      case OR_I16: s = (int16_t)(uint16_t)bits; break;
      case OR_I32: s = (int32_t)(uint32_t)bits; break;
      default: s = (int64_t)bits; break; /* OR_I64 */
    }
    v.neg = s < 0;
    v.mag = v.neg ? (uint64_t)0 - (uint64_t)s : (uint64_t)s; /* |INT64_MIN| = 2^63 */
    return v;
  }
  fmt f = format_of(t);
  int width = f.p + f.ebits; /* total bits: 1 + ebits + (p - 1) */
  uint64_t frac_mask = ((uint64_t)1 << (f.p - 1)) - 1;
  uint64_t emax_field = ((uint64_t)1 << f.ebits) - 1;
  uint64_t frac = bits & frac_mask;
  uint64_t efield = (bits >> (f.p - 1)) & emax_field;
  v.neg = (int)((bits >> (width - 1)) & 1);
  if (efield == emax_field) {
    if (frac) v.nan = 1; else v.inf = 1;
    return v;
  }
  if (efield == 0) { /* zero or subnormal: frac * 2^(1 - bias - (p - 1)) */
    v.mag = frac;
    v.exp = 1 - f.bias - (f.p - 1);
  } else {
    v.mag = frac | ((uint64_t)1 << (f.p - 1));
    v.exp = (int)efield - f.bias - (f.p - 1);
  }
  return v;
}

static int top_bit(uint64_t x) { /* x != 0 */
  int b = 63;
  while (!((x >> b) & 1)) b--;
  return b;
}

/* Round the exact value v to format f (to nearest, ties to even); returns the
 * encoding and sets *overflow when a finite value becomes infinite. */
static uint64_t encode_float(value v, fmt f, int* overflow) {
  int width = f.p + f.ebits;
  uint64_t sign = (uint64_t)v.neg << (width - 1);
  uint64_t emax_field = ((uint64_t)1 << f.ebits) - 1;
  uint64_t hidden = (uint64_t)1 << (f.p - 1);
  *overflow = 0;
  if (v.nan) return (emax_field << (f.p - 1)) | (hidden >> 1); /* canonical quiet NaN, positive */
  if (v.inf) return sign | (emax_field << (f.p - 1));
  if (v.mag == 0) return sign;
  int E = top_bit(v.mag) + v.exp; /* exponent of the leading bit */
  int emin = 1 - f.bias;          /* smallest normal exponent */
  int qe = (E > emin ? E : emin) - (f.p - 1); /* exponent of one unit in the last place */
  int shift = qe - v.exp;                     /* bits of mag below that unit */
  uint64_t q;
  if (shift <= 0) {
    q = v.mag << (-shift); /* exact; at most p bits */
  } else if (shift >= 128) {
    q = 0; /* below half a unit: rounds to zero */
  } else {
    u128 m = v.mag;
    u128 qq = m >> shift;
    u128 rem = m - (qq << shift);
    u128 half = (u128)1 << (shift - 1);
    if (rem > half || (rem == half && (qq & 1))) qq++;
    q = (uint64_t)qq;
  }
  if (q == (hidden << 1)) { /* carried into the next binade */
    q = hidden;
    qe++;
  }
  if (q == 0) return sign;
  if (q < hidden) return sign | q; /* subnormal: biased exponent 0 */
  int64_t efield = (int64_t)qe + (f.p - 1) + f.bias;
  if (efield >= (int64_t)emax_field) {
    *overflow = 1;
    return sign | (emax_field << (f.p - 1));
  }
  return sign | ((uint64_t)efield << (f.p - 1)) | (q - hidden);
}

/* Integer target: the value, clamped to [lo, hi] (*clamped set when it was). */
static uint64_t encode_int(value v, int t, int* clamped) {
  int64_t lo = 0;
  uint64_t hi = 0;
  switch (t) {
    case OR_U8: hi = 0xFF; break;
    case OR_U16: hi = 0xFFFF; break;
    case OR_U32: hi = 0xFFFFFFFFull; break;
    case OR_U64: hi = UINT64_MAX; break;
    case OR_I8: lo = -128; hi = 127; break;
    case OR_I16: lo = -32768; hi = 32767; break;
    case OR_I32: lo = -2147483647 - 1; hi = 2147483647; break;
    default: lo = INT64_MIN; hi = INT64_MAX; break; /* OR_I64 */
  }
  *clamped = 0;
  if (v.neg && v.mag != 0) {
    uint64_t lo_mag = (uint64_t)0 - (uint64_t)lo; /* |lo| as unsigned (0 for unsigned types) */
    if (v.mag > lo_mag) { *clamped = 1; return (uint64_t)lo; }
    return (uint64_t)0 - v.mag; /* two's complement of -mag */
  }
  if (v.mag > hi) { *clamped = 1; return hi; }
  return v.mag;
}

int or_convert(int src_dtype, const void* src, uint64_t n, int dst_dtype, void* dst, uint64_t* n_bad) {
  int sb = or_dtype_bytes(src_dtype), db = or_dtype_bytes(dst_dtype);
  if (n_bad) *n_bad = 0;
  if (!sb || !db) return -1;
  if (is_float(src_dtype) && !is_float(dst_dtype)) return -1;
  if (n && (!src || !dst)) return -1;
  const uint8_t* s = (const uint8_t*)src;
  uint8_t* d = (uint8_t*)dst;
  if (src_dtype == dst_dtype) {
    memmove(d, s, (size_t)(n * (uint64_t)sb));
    return 0;
  }
  uint64_t bad = 0;
  for (uint64_t i = 0; i < n; i++) {
    value v = decode(src_dtype, load_bits(s + i * (uint64_t)sb, sb));
    uint64_t out;
    int lost = 0;
    if (is_float(dst_dtype)) out = encode_float(v, format_of(dst_dtype), &lost);
    else out = encode_int(v, dst_dtype, &lost);
    bad += (uint64_t)lost;
    memcpy(d + i * (uint64_t)db, &out, (size_t)db); /* little-endian: the low bytes */
  }
  if (n_bad) *n_bad = bad;
  return 0;
}
