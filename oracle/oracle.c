/*
 * oracle.c -- plain, slow, single-threaded CPU oracle (test infrastructure).
 *
 * TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the bench's CPU
 * baseline may call it; the product path never does.  Shares no code with the
 * CUDA library.  Compiled with -ffp-contract=off -fno-fast-math.
 *
 * Layout of this file follows the steps of Synthesis-Based Verification
 * (CUDA-Harness, Sec. 4.2): synthesis of test data (Sec. 4.2.1), the
 * functional-validation rule (Eq. 1) and progressive validation (Sec. 4.2.2).
 * The paper names no generator, value map or float semantics; the readings
 * taken here are stated beside each function.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as  */
/* easy as 1, 2, 3", SC'11).  Each round multiplies counter words 0 and 2 by */
/* the two round multipliers; the high halves are xored with the other two   */
/* words and the key, the low halves move across.  The key is advanced by    */
/* the two Weyl increments between rounds.                                   */
/* ------------------------------------------------------------------------ */
#define PHILOX_M4x32_0 0xD2511F53u
#define PHILOX_M4x32_1 0xCD9E8D57u
#define PHILOX_W32_0 0x9E3779B9u
#define PHILOX_W32_1 0xBB67AE85u

static const double TWO_PI = 6.283185307179586476925286766559;

void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += PHILOX_W32_0;
      k1 += PHILOX_W32_1;
    }
    uint64_t prod0 = (uint64_t)PHILOX_M4x32_0 * (uint64_t)x0;
    uint64_t prod1 = (uint64_t)PHILOX_M4x32_1 * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t n0 = hi1 ^ x1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ x3 ^ k1;
    uint32_t n3 = lo0;
    x0 = n0; x1 = n1; x2 = n2; x3 = n3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* One 128-bit draw.  Counter = (block lo, block hi, stream, purpose); key =  */
/* the 64-bit seed.  Every quantity the synthesis needs has its own purpose, */
/* so changing one (say, a special-value rate) never moves another.          */
void or_draw(uint64_t seed, uint32_t stream, uint32_t purpose, uint64_t block, uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)block, (uint32_t)(block >> 32), stream, purpose};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  or_philox4x32_10(ctr, key, out);
}

static uint64_t mulhi64(uint64_t a, uint64_t b) {
  return (uint64_t)(((unsigned __int128)a * (unsigned __int128)b) >> 64);
}

/* ------------------------------------------------------------------------ */
/* element storage                                                          */
/* ------------------------------------------------------------------------ */
static int is_float_dtype(uint32_t dt) { return dt == OR_F32 || dt == OR_F16 || dt == OR_BF16; }
static int is_int_dtype(uint32_t dt) { return dt == OR_I32 || dt == OR_I64 || dt == OR_U32; }

static uint64_t elem_bytes(uint32_t dt) {
  switch (dt) {
    case OR_F32: return 4;
    case OR_F16: return 2;
    case OR_BF16: return 2;
    case OR_I32: return 4;
    case OR_I64: return 8;
    case OR_U32: return 4;
    default: return 0;
  }
}

static uint64_t width_mask(uint32_t dt) {
  uint64_t b = elem_bytes(dt);
  return b == 8 ? ~(uint64_t)0 : (((uint64_t)1 << (8 * b)) - 1);
}

static uint32_t f32_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

static float bits_f32(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* fp32 -> bf16, round to nearest, ties to even, on the 16 dropped bits.     */
/* NaN -> canonical quiet NaN 0x7FC0.  A carry out of the mantissa moves the */
/* exponent up, which is the correct rounding (also to +-Inf).               */
uint16_t or_f32_to_bf16(float f) {
  if (isnan(f)) return 0x7FC0;
  uint32_t u = f32_bits(f);
  uint32_t hi = u >> 16, lo = u & 0xFFFFu;
  if (lo > 0x8000u || (lo == 0x8000u && (hi & 1u))) hi += 1;
  return (uint16_t)hi;
}

float or_bf16_to_f32(uint16_t h) { return bits_f32((uint32_t)h << 16); }

/* fp32 -> IEEE binary16, round to nearest, ties to even, written from the   */
/* value: |f| = q * ulp with ulp the binary16 spacing at |f|'s binade (or    */
/* 2^-24 below the normal range); q is rounded to an integer, ties to even. */
/* Values at or above 65520 (the midpoint above 65504) overflow to Inf.     */
/* NaN -> canonical quiet NaN 0x7E00.                                       */
uint16_t or_f32_to_f16(float f) {
  if (isnan(f)) return 0x7E00;
  uint16_t sign = signbit(f) ? 0x8000 : 0;
  double a = fabs((double)f);
  if (a >= 65520.0) return sign | 0x7C00;
  if (a == 0.0) return sign;
  int ex;
  frexp(a, &ex);          /* a = m * 2^ex, m in [0.5, 1): floor(log2 a) = ex - 1 */
  int e = ex - 1;
  if (e < -14) e = -14;   /* denormal range shares the spacing of binade -14 */
  double ulp = ldexp(1.0, e - 10);
  double q = a / ulp;     /* exact: a has 24 significant bits, ulp is a power of 2 */
  double fl = floor(q);
  double frac = q - fl;
  if (frac > 0.5 || (frac == 0.5 && fmod(fl, 2.0) != 0.0)) fl += 1.0;
  uint32_t mant = (uint32_t)fl; /* in [0, 2048] */
  uint32_t bits;
  if (a < ldexp(1.0, -14) && mant <= 1024) {
    bits = mant; /* denormal; mant == 1024 is the smallest normal 0x0400 */
  } else {
    bits = (uint32_t)(e + 15) * 1024u + (mant - 1024u); /* mant == 2048 carries */
  }
  return (uint16_t)(sign | bits);
}

float or_f16_to_f32(uint16_t h) {
  uint32_t sign = h >> 15, ex = (h >> 10) & 31u, mant = h & 1023u;
  double v;
  if (ex == 0) {
    v = ldexp((double)mant, -24);
  } else if (ex == 31) {
    v = mant ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024u + mant), (int)ex - 25);
  }
  return (float)(sign ? -v : v);
}

static float load_f32(uint32_t dt, uint64_t bits) {
  switch (dt) {
    case OR_F32: return bits_f32((uint32_t)bits);
    case OR_F16: return or_f16_to_f32((uint16_t)bits);
    default: return or_bf16_to_f32((uint16_t)bits);
  }
}

/* float value -> storage bits; every NaN is stored as the canonical quiet NaN */
static uint64_t store_f32(uint32_t dt, float x) {
  switch (dt) {
    case OR_F32: return isnan(x) ? 0x7FC00000u : f32_bits(x);
    case OR_F16: return or_f32_to_f16(x);
    default: return or_f32_to_bf16(x);
  }
}

static int64_t bits_to_int(uint32_t dt, uint64_t bits) {
  switch (dt) {
    case OR_I32: return (int64_t)(int32_t)(uint32_t)bits;
    case OR_U32: return (int64_t)(uint32_t)bits;
    default: return (int64_t)bits;
  }
}

static uint64_t read_bits(const uint8_t* base, uint32_t dt, uint64_t i) {
  uint64_t sz = elem_bytes(dt);
  uint64_t v = 0;
  memcpy(&v, base + i * sz, sz); /* little-endian hosts only (x86_64, aarch64) */
  return v;
}

static void write_bits(uint8_t* base, uint32_t dt, uint64_t i, uint64_t v) {
  uint64_t sz = elem_bytes(dt);
  memcpy(base + i * sz, &v, sz);
}

/* ------------------------------------------------------------------------ */
/* value maps                                                               */
/* ------------------------------------------------------------------------ */

/* U[a, b): u = (w >> 8) * 2^-24 in [0, 1), x = a + (b - a) * u, each        */
/* operation one fp32 rounding (a, b and b - a taken in fp32).               */
float or_uniform_map(float a, float b, uint32_t w) {
  float width = b - a;
  float u = (float)(w >> 8) * 0x1p-24f;
  float t = width * u;
  return a + t;
}

/* Box-Muller on one pair of words, computed in fp64 and rounded once to     */
/* fp32.  u1 = ((wa >> 8) + 1) * 2^-24 in (0, 1]; the angle is               */
/* 2*pi*m/2^24 with m = wb >> 8.  The quarter turn is split off on the       */
/* integer m, so angles on the axes give exactly 0 and +-1 before scaling.   */
/* z0 = r cos(angle), z1 = r sin(angle), r = sqrt(-2 ln u1); |z| <= 5.77.    */
void or_box_muller(uint32_t wa, uint32_t wb, float* z0, float* z1) {
  double u1 = ((double)(wa >> 8) + 1.0) * 0x1p-24;
  double r = sqrt(-2.0 * log(u1));
  uint32_t m = wb >> 8;
  uint32_t quarter = m >> 22;
  uint32_t rem = m & 0x3FFFFFu;
  double t = (double)rem * (TWO_PI / 16777216.0);
  double c = cos(t), s = sin(t);
  double cq, sq;
  switch (quarter) {
    case 0: cq = c; sq = s; break;
    case 1: cq = -s; sq = c; break;
    case 2: cq = -c; sq = -s; break;
    default: cq = s; sq = -c; break;
  }
  *z0 = (float)(r * cq);
  *z1 = (float)(r * sq);
}

/* [lo, lo + r) with r <= 2^32: lo + floor(w * r / 2^32).  No rejection, so  */
/* the map from counter to value is fixed; bucket sizes differ by at most 1. */
int64_t or_int_range_map32(int64_t lo, uint64_t r, uint32_t w) {
  uint64_t off = ((uint64_t)w * r) >> 32;
  return (int64_t)((uint64_t)lo + off);
}

/* Keyed bijection of [0, N).  k = bits of N - 1; four rounds of             */
/* x <- (x * m_r + a_r) mod 2^k, x <- x xor (x >> ceil(k/2)), with m_r odd   */
/* and a_r drawn from the PERM purpose; each step is invertible mod 2^k.     */
/* Values >= N are walked again through the same map until they land in     */
/* [0, N) (cycle walking), which keeps the map a bijection of [0, N).        */
uint64_t or_perm_value(uint64_t N, uint64_t seed, uint32_t stream, uint64_t g) {
  if (N <= 1 || g >= N) return 0; /* defined on [0, N) only */
  int k = 0;
  while (k < 64 && ((uint64_t)1 << k) < N) ++k;
  uint64_t mask = (k >= 64) ? ~(uint64_t)0 : (((uint64_t)1 << k) - 1);
  uint64_t mul[4], add[4];
  for (int r = 0; r < 4; ++r) {
    uint32_t w[4];
    or_draw(seed, stream, OR_P_PERM, (uint64_t)r, w);
    mul[r] = ((((uint64_t)w[0] << 32) | w[1]) | 1u) & mask;
    add[r] = (((uint64_t)w[2] << 32) | w[3]) & mask;
  }
  int shift = (k + 1) / 2;
  uint64_t x = g;
  do {
    for (int r = 0; r < 4; ++r) {
      x = (x * mul[r] + add[r]) & mask;
      x ^= x >> shift;
    }
  } while (x >= N);
  return x;
}

/* Exact-count index selection: [0, N) is cut into k strata                */
/* [floor(s N / k), floor((s+1) N / k)); stratum s contributes one index     */
/* drawn uniformly inside it (INDEX purpose, block s).  k distinct indices.  */
static uint64_t stratum_index_purpose(uint64_t N, uint64_t k, uint64_t seed, uint32_t stream, uint32_t purpose,
                                      uint64_t s) {
  uint64_t start = (uint64_t)(((unsigned __int128)s * N) / k);
  uint64_t end = (uint64_t)(((unsigned __int128)(s + 1) * N) / k);
  uint32_t w[4];
  or_draw(seed, stream, purpose, s, w);
  uint64_t x = ((uint64_t)w[0] << 32) | w[1];
  return start + mulhi64(x, end - start);
}

uint64_t or_stratum_index(uint64_t N, uint64_t k, uint64_t seed, uint32_t stream, uint64_t s) {
  return stratum_index_purpose(N, k, seed, stream, OR_P_INDEX, s);
}

/* The stratum holding g: stratum s covers [floor(sN/k), floor((s+1)N/k)),   */
/* so s is the largest value with floor(sN/k) <= g, i.e. with sN < (g+1)k:    */
/* s = ceil((g+1)k/N) - 1 = floor(((g+1)k - 1)/N), at most k - 1.             */
uint64_t or_stratum_of(uint64_t g, uint64_t k, uint64_t N) {
  unsigned __int128 s = (((unsigned __int128)(g + 1) * k) - 1) / N;
  return s < k ? (uint64_t)s : k - 1;
}

/* Reading of "0.01% injected" as an exact count (the paper asks only for     */
/* broad, special-laden inputs, Sec. 4.2.1): round(rate N) specials, at most  */
/* N, placed one per stratum like the exact-count perturbations but drawn on  */
/* the SPECIAL_SEL purpose of the spec's own stream.                          */
uint64_t or_special_count(double rate, uint64_t N) {
  if (!(rate > 0.0)) return 0;
  double k = floor(rate * (double)N + 0.5);
  return k >= (double)N ? N : (uint64_t)k;
}

uint64_t or_special_index(uint64_t N, uint64_t k, uint64_t seed, uint32_t stream, uint64_t s) {
  return stratum_index_purpose(N, k, seed, stream, OR_P_SPECIAL_SEL, s);
}

static uint64_t rate_threshold(double rate) {
  if (!(rate > 0.0)) return 0;
  if (rate >= 1.0) return (uint64_t)1 << 32;
  return (uint64_t)floor(rate * 4294967296.0);
}

static uint64_t logical_len(const or_spec* s) {
  return s->logical_n ? s->logical_n : s->elem_offset + s->n;
}

/* ------------------------------------------------------------------------ */
/* synthesis: base value -> special values -> element-wise perturbation ->  */
/* exact-count perturbation.  The clean output is the value after specials, */
/* the perturbed twin the value after all four steps.                       */
/* ------------------------------------------------------------------------ */

/* the words of 32-bit-or-narrower element g: block g/4, lane g%4;          */
/* 64-bit elements use two words: block g/2, lanes 2(g%2), 2(g%2)+1.         */
static uint64_t base_value(const or_spec* s, const uint8_t* arena, uint64_t g) {
  uint32_t dt = s->dtype;
  uint32_t w[4];
  switch (s->dist) {
    case OR_UNIFORM: {
      or_draw(s->seed, s->stream, OR_P_VALUE, g >> 2, w);
      return store_f32(dt, or_uniform_map((float)s->p0, (float)s->p1, w[g & 3]));
    }
    case OR_NORMAL: {
      or_draw(s->seed, s->stream, OR_P_VALUE, g >> 2, w);
      uint32_t lane = (uint32_t)(g & 3);
      float z0, z1;
      or_box_muller(w[lane & 2u], w[(lane & 2u) + 1], &z0, &z1);
      float z = (lane & 1u) ? z1 : z0;
      float mu = (float)s->p0, sigma = (float)s->p1;
      float t = sigma * z;
      return store_f32(dt, mu + t);
    }
    case OR_INT_RANGE: {
      uint64_t r = (uint64_t)s->i1 - (uint64_t)s->i0 + 1u; /* 0 means 2^64 */
      if (dt == OR_I64) {
        or_draw(s->seed, s->stream, OR_P_VALUE, g >> 1, w);
        uint32_t j = (uint32_t)(g & 1) * 2u;
        uint64_t x = ((uint64_t)w[j] << 32) | w[j + 1];
        uint64_t off = (r == 0) ? x : mulhi64(x, r);
        return (uint64_t)s->i0 + off;
      }
      or_draw(s->seed, s->stream, OR_P_VALUE, g >> 2, w);
      return (uint64_t)or_int_range_map32(s->i0, r, w[g & 3]) & width_mask(dt);
    }
    case OR_PERMUTATION:
      return or_perm_value(logical_len(s), s->seed, s->stream, g) & width_mask(dt);
    case OR_DOTLIKE: {
      uint64_t i = g / s->cols, j = g % s->cols;
      const uint8_t* A = arena + s->a_offset;
      const uint8_t* B = arena + s->b_offset;
      float acc = 0.0f;
      for (uint64_t k = 0; k < s->dot_k; ++k) {
        float a, b;
        memcpy(&a, A + 4 * (i * s->dot_k + k), 4);
        memcpy(&b, B + 4 * (k * s->cols + j), 4);
        acc = fmaf(a, b, acc);
      }
      return store_f32(dt, acc);
    }
    case OR_RAW_BITS: {
      if (dt == OR_I64) {
        or_draw(s->seed, s->stream, OR_P_VALUE, g >> 1, w);
        uint32_t j = (uint32_t)(g & 1) * 2u;
        return ((uint64_t)w[j] << 32) | w[j + 1];
      }
      or_draw(s->seed, s->stream, OR_P_VALUE, g >> 2, w);
      if (elem_bytes(dt) == 2) return w[g & 3] >> 16;
      return w[g & 3];
    }
    case OR_FROM_ARENA: {
      /* element g of the existing array at a_offset (same element type) */
      uint64_t bits = 0;
      memcpy(&bits, arena + s->a_offset + g * elem_bytes(dt), elem_bytes(dt)); /* little-endian */
      return bits;
    }
    case OR_CONSTANT:
    default:
      if (is_float_dtype(dt)) return store_f32(dt, (float)s->p0);
      return (uint64_t)s->i0 & width_mask(dt);
  }
}

/* special values: element g is special iff its SPECIAL_SEL word is below   */
/* floor(rate * 2^32); its kind is the j-th set bit of the mask with        */
/* j = floor(w0 * popcount / 2^32), w0..w3 from SPECIAL_KIND block g.       */
/* Selection: with OR_SP_EXACT, g is special iff it is the index drawn in    */
/* its own stratum (only that stratum's draw can land on g); otherwise iff   */
/* its SPECIAL_SEL word is below floor(rate * 2^32).                          */
static int is_special(const or_spec* s, uint64_t g) {
  if ((s->special_mask & OR_SP_KINDS) == 0) return 0;
  if (s->special_mask & OR_SP_EXACT) {
    uint64_t N = logical_len(s), k = or_special_count(s->special_rate, N);
    if (k == 0) return 0;
    return or_special_index(N, k, s->seed, s->stream, or_stratum_of(g, k, N)) == g;
  }
  uint64_t thr = rate_threshold(s->special_rate);
  if (thr == 0) return 0;
  uint32_t w[4];
  or_draw(s->seed, s->stream, OR_P_SPECIAL_SEL, g >> 2, w);
  return (uint64_t)w[g & 3] < thr;
}

static uint64_t clean_value(const or_spec* s, const uint8_t* arena, uint64_t g) {
  uint64_t v0 = base_value(s, arena, g);
  if (!is_special(s, g)) return v0;
  uint32_t kinds = s->special_mask & OR_SP_KINDS;
  uint32_t kw[4];
  or_draw(s->seed, s->stream, OR_P_SPECIAL_KIND, g, kw);
  uint32_t nkinds = 0;
  for (int b = 0; b < 32; ++b) nkinds += (kinds >> b) & 1u;
  uint32_t pick = (uint32_t)(((uint64_t)kw[0] * nkinds) >> 32);
  uint32_t kind = 0;
  for (int b = 0, seen = 0; b < 32; ++b) {
    if ((kinds >> b) & 1u) {
      if ((uint32_t)seen == pick) { kind = 1u << b; break; }
      ++seen;
    }
  }
  uint32_t dt = s->dtype;
  switch (kind) {
    case OR_SP_NAN: return store_f32(dt, NAN);
    case OR_SP_PINF: return store_f32(dt, INFINITY);
    case OR_SP_NINF: return store_f32(dt, -INFINITY);
    case OR_SP_DENORM: {
      /* random sign, random nonzero fraction, zero exponent */
      uint32_t neg = kw[1] >> 31;
      if (dt == OR_F32) return ((uint64_t)neg << 31) | ((kw[1] & 0x7FFFFFu) | 1u);
      if (dt == OR_F16) return ((uint64_t)neg << 15) | ((kw[1] & 0x3FFu) | 1u);
      return ((uint64_t)neg << 15) | ((kw[1] & 0x7Fu) | 1u);
    }
    case OR_SP_ZERO: return 0;
    case OR_SP_IMIN:
      if (dt == OR_I32) return 0x80000000u;
      if (dt == OR_I64) return (uint64_t)1 << 63;
      return 0;
    case OR_SP_IMAX:
      if (dt == OR_I32) return 0x7FFFFFFFu;
      if (dt == OR_I64) return ~((uint64_t)1 << 63);
      return 0xFFFFFFFFu;
    case OR_SP_DUP: {
      /* a copy of the base value at a uniformly drawn index of the array */
      uint64_t x = ((uint64_t)kw[2] << 32) | kw[3];
      uint64_t j = mulhi64(x, logical_len(s));
      return base_value(s, arena, j);
    }
    default: return v0;
  }
}

/* element-wise candidate perturbation, applied to the clean value          */
static uint64_t elementwise_perturbed(const or_spec* s, uint64_t g, uint64_t v1) {
  const or_perturb* p = &s->pelem;
  uint32_t dt = s->dtype;
  uint32_t w[4];
  if (p->kind == OR_PERT_RATE_ADD_PM) {
    /* Bernoulli(rate) selection, then +-value with the sign drawn per element */
    or_draw(s->seed, p->stream, OR_P_PERT_SEL, g >> 2, w);
    if (!((uint64_t)w[g & 3] < rate_threshold(p->rate))) return v1;
    or_draw(s->seed, p->stream, OR_P_PERT_VAL, g, w);
    int neg = (int)(w[0] >> 31);
    if (is_float_dtype(dt)) {
      float x = load_f32(dt, v1);
      if (!isfinite(x)) return v1;
      float d = (float)p->value;
      float y = neg ? x - d : x + d;
      return store_f32(dt, y);
    }
    uint64_t delta = neg ? (uint64_t)0 - (uint64_t)p->ivalue : (uint64_t)p->ivalue;
    return (v1 + delta) & width_mask(dt);
  }
  if (p->kind == OR_PERT_REL_NOISE) {
    /* y = x + (c |x|) z, z ~ N(0,1) by Box-Muller on the NOISE purpose */
    float x = load_f32(dt, v1);
    if (!isfinite(x)) return v1;
    or_draw(s->seed, p->stream, OR_P_NOISE, g >> 2, w);
    uint32_t lane = (uint32_t)(g & 3);
    float z0, z1;
    or_box_muller(w[lane & 2u], w[(lane & 2u) + 1], &z0, &z1);
    float z = (lane & 1u) ? z1 : z0;
    float c = (float)p->value;
    float t = c * fabsf(x);
    float u = t * z;
    return store_f32(dt, x + u);
  }
  return v1;
}

static uint64_t pre_count_value(const or_spec* s, const uint8_t* arena, uint64_t g) {
  return elementwise_perturbed(s, g, clean_value(s, arena, g));
}

/* exact-count perturbation of one selected element whose value is v2       */
static uint64_t count_applied(const or_spec* s, uint64_t v2) {
  const or_perturb* p = &s->pcount;
  uint32_t dt = s->dtype;
  if (p->kind == OR_PERT_COUNT_SET) {
    if (is_float_dtype(dt)) return store_f32(dt, (float)p->value);
    return (uint64_t)p->ivalue & width_mask(dt);
  }
  /* OR_PERT_COUNT_ADD: finite values move by value, non-finite become value */
  if (is_float_dtype(dt)) {
    float x = load_f32(dt, v2);
    float d = (float)p->value;
    return store_f32(dt, isfinite(x) ? x + d : d);
  }
  return (v2 + (uint64_t)p->ivalue) & width_mask(dt);
}

static uint64_t count_strata(const or_spec* s) {
  return s->pcount.kind == OR_PERT_SWAP_PAIRS ? 2 * s->pcount.count : s->pcount.count;
}

uint64_t or_value_at(const or_spec* s, const uint8_t* arena, uint64_t g, int role) {
  if (role == 0) return clean_value(s, arena, g);
  uint64_t v2 = pre_count_value(s, arena, g);
  const or_perturb* p = &s->pcount;
  if (p->kind == OR_PERT_NONE) return v2;
  uint64_t N = logical_len(s), k = count_strata(s);
  for (uint64_t st = 0; st < k; ++st) {
    if (or_stratum_index(N, k, s->seed, p->stream, st) != g) continue;
    if (p->kind == OR_PERT_SWAP_PAIRS) {
      uint64_t partner = or_stratum_index(N, k, s->seed, p->stream, st ^ 1u);
      return pre_count_value(s, arena, partner);
    }
    return count_applied(s, v2);
  }
  return v2;
}

int or_check_spec(const or_spec* s, uint64_t arena_bytes) {
  uint32_t dt = s->dtype;
  if (elem_bytes(dt) == 0) return -1;
  int fl = is_float_dtype(dt);
  switch (s->dist) {
    case OR_UNIFORM: case OR_NORMAL: case OR_DOTLIKE: if (!fl) return -1; break;
    case OR_INT_RANGE: case OR_PERMUTATION: if (!is_int_dtype(dt)) return -1; break;
    case OR_RAW_BITS: case OR_CONSTANT: case OR_FROM_ARENA: break;
    default: return -1;
  }
  if (s->ref_offset == OR_ABSENT && s->cand_offset == OR_ABSENT) return -1;
  uint64_t N = logical_len(s);
  if (N < s->elem_offset + s->n) return -1;
  uint64_t bytes = s->n * elem_bytes(dt);
  if (s->ref_offset != OR_ABSENT && (s->ref_offset > arena_bytes || bytes > arena_bytes - s->ref_offset)) return -1;
  if (s->cand_offset != OR_ABSENT && (s->cand_offset > arena_bytes || bytes > arena_bytes - s->cand_offset)) return -1;
  if (s->dist == OR_INT_RANGE) {
    if (s->i1 < s->i0) return -1;
    if (dt == OR_I32 && (s->i0 < INT32_MIN || s->i1 > INT32_MAX)) return -1;
    if (dt == OR_U32 && (s->i0 < 0 || s->i1 > (int64_t)UINT32_MAX)) return -1;
  }
  if (s->dist == OR_DOTLIKE) {
    if (s->cols == 0 || s->rows * s->cols != N || s->dot_k == 0) return -1;
    if (s->a_offset + 4 * s->rows * s->dot_k > arena_bytes) return -1;
    if (s->b_offset + 4 * s->dot_k * s->cols > arena_bytes) return -1;
  }
  if (s->dist == OR_FROM_ARENA) {
    /* the source is the whole logical array; it must lie in the arena, away from the outputs */
    uint64_t src = N * elem_bytes(dt);
    if (s->a_offset % 16 || s->a_offset > arena_bytes || src > arena_bytes - s->a_offset) return -1;
    if (s->ref_offset != OR_ABSENT && bytes && s->ref_offset < s->a_offset + src && s->a_offset < s->ref_offset + bytes)
      return -1;
    if (s->cand_offset != OR_ABSENT && bytes && s->cand_offset < s->a_offset + src &&
        s->a_offset < s->cand_offset + bytes)
      return -1;
  }
  uint32_t fmask = OR_SP_NAN | OR_SP_PINF | OR_SP_NINF | OR_SP_DENORM | OR_SP_ZERO | OR_SP_DUP | OR_SP_EXACT;
  uint32_t imask = OR_SP_ZERO | OR_SP_IMIN | OR_SP_IMAX | OR_SP_DUP | OR_SP_EXACT;
  if (s->special_mask & ~(fl ? fmask : imask)) return -1;
  uint32_t ek = s->pelem.kind, ck = s->pcount.kind;
  if (ek != OR_PERT_NONE && ek != OR_PERT_RATE_ADD_PM && ek != OR_PERT_REL_NOISE) return -1;
  if (ek == OR_PERT_REL_NOISE && !fl) return -1;
  if (ck != OR_PERT_NONE && ck != OR_PERT_COUNT_SET && ck != OR_PERT_COUNT_ADD && ck != OR_PERT_SWAP_PAIRS) return -1;
  if (ck != OR_PERT_NONE && (count_strata(s) == 0 || count_strata(s) > N)) return -1;
  return 0;
}

int or_generate(const or_spec* specs, int n_specs, uint8_t* arena, uint64_t arena_bytes) {
  int status = 0;
  for (int si = 0; si < n_specs; ++si) {
    const or_spec* s = &specs[si];
    if (or_check_spec(s, arena_bytes) != 0) { status = -1; continue; }
    uint32_t dt = s->dtype;
    uint8_t* ref = s->ref_offset == OR_ABSENT ? NULL : arena + s->ref_offset;
    uint8_t* cand = s->cand_offset == OR_ABSENT ? NULL : arena + s->cand_offset;
    /* steps 1-3 for every element of this chunk */
    for (uint64_t i = 0; i < s->n; ++i) {
      uint64_t g = s->elem_offset + i;
      uint64_t v1 = clean_value(s, arena, g);
      if (ref) write_bits(ref, dt, i, v1);
      if (cand) write_bits(cand, dt, i, elementwise_perturbed(s, g, v1));
    }
    /* step 4: the exact-count edits that fall inside this chunk */
    const or_perturb* p = &s->pcount;
    if (!cand || p->kind == OR_PERT_NONE) continue;
    uint64_t N = logical_len(s), k = count_strata(s);
    uint64_t lo = s->elem_offset, hi = s->elem_offset + s->n;
    if (p->kind == OR_PERT_SWAP_PAIRS) {
      for (uint64_t t = 0; t < p->count; ++t) {
        uint64_t a = or_stratum_index(N, k, s->seed, p->stream, 2 * t);
        uint64_t b = or_stratum_index(N, k, s->seed, p->stream, 2 * t + 1);
        uint64_t va = pre_count_value(s, arena, a), vb = pre_count_value(s, arena, b);
        if (a >= lo && a < hi) write_bits(cand, dt, a - lo, vb);
        if (b >= lo && b < hi) write_bits(cand, dt, b - lo, va);
      }
    } else {
      for (uint64_t st = 0; st < k; ++st) {
        uint64_t idx = or_stratum_index(N, k, s->seed, p->stream, st);
        if (idx >= lo && idx < hi)
          write_bits(cand, dt, idx - lo, count_applied(s, pre_count_value(s, arena, idx)));
      }
    }
  }
  return status;
}

/* ------------------------------------------------------------------------ */
/* functional validation, Eq. 1: |K(x) - y| <= atol + rtol |y|, y = the      */
/* reference.  Readings: the rule is evaluated in fp32 (tolerances rounded   */
/* once to fp32, 16-bit values widened exactly, no fused operations); it is  */
/* applied only where both values are finite; equal values (same infinity,  */
/* +0/-0) always match; two NaNs match when OR_EQUAL_NAN is set.  Integer    */
/* types are compared exactly.                                               */
/* ------------------------------------------------------------------------ */
static int check_pair(const or_pair* p, uint64_t cand_bytes, uint64_t ref_bytes) {
  uint64_t sz = elem_bytes(p->dtype);
  if (sz == 0) return -1;
  if (p->n > UINT64_MAX / sz) return -1;
  uint64_t bytes = p->n * sz;
  if (p->cand_offset > cand_bytes || bytes > cand_bytes - p->cand_offset) return -1;
  if (p->ref_offset > ref_bytes || bytes > ref_bytes - p->ref_offset) return -1;
  if (is_float_dtype(p->dtype) && !(p->atol >= 0.0 && p->rtol >= 0.0)) return -1;
  return 0;
}

int or_check_pair(const or_pair* p, uint64_t cand_bytes, uint64_t ref_bytes) {
  return check_pair(p, cand_bytes, ref_bytes);
}

/* one segment by the rule above; *sumsq_out receives the sum of squared     */
/* differences behind r->rms (so chunked drivers can combine exact sums)     */
static void compare_one_sum(const or_pair* p, const uint8_t* cand, const uint8_t* ref, or_result* r,
                            double* sumsq_out) {
  memset(r, 0, sizeof(*r));
  r->first_mismatch = -1;
  r->state = OR_STAGE_RUN;
  uint32_t dt = p->dtype;
  const uint8_t* xb = cand + p->cand_offset;
  const uint8_t* yb = ref + p->ref_offset;
  if (is_float_dtype(dt)) {
    float atol = (float)p->atol, rtol = (float)p->rtol;
    float max_abs = 0.0f, max_rel = 0.0f;
    double sumsq = 0.0;
    for (uint64_t i = 0; i < p->n; ++i) {
      float x = load_f32(dt, read_bits(xb, dt, i));
      float y = load_f32(dt, read_bits(yb, dt, i));
      int xnan = isnan(x), ynan = isnan(y);
      int xinf = isinf(x), yinf = isinf(y);
      int both_finite = !xnan && !ynan && !xinf && !yinf;
      float d = fabsf(x - y);
      float tol = atol + rtol * fabsf(y);
      int match;
      if (x == y) match = 1;
      else if (both_finite && d <= tol) match = 1;
      else if (xnan && ynan && (p->flags & OR_EQUAL_NAN)) match = 1;
      else match = 0;
      if (!match) {
        r->mismatches++;
        if (r->first_mismatch < 0) r->first_mismatch = (int64_t)i;
        if (xnan != ynan) r->nan_disagree++;
        else if (!xnan && (xinf || yinf)) r->inf_disagree++;
      }
      if (both_finite) {
        r->n_finite++;
        if (d > max_abs) max_abs = d;
        sumsq += (double)d * (double)d;
        if (y != 0.0f) {
          float q = d / fabsf(y);
          if (q > max_rel) max_rel = q;
        }
      }
    }
    r->max_abs = max_abs;
    r->max_rel = max_rel;
    r->rms = r->n_finite ? sqrt(sumsq / (double)r->n_finite) : 0.0;
    *sumsq_out = sumsq;
  } else {
    double sumsq = 0.0, max_rel = 0.0;
    for (uint64_t i = 0; i < p->n; ++i) {
      int64_t x = bits_to_int(dt, read_bits(xb, dt, i));
      int64_t y = bits_to_int(dt, read_bits(yb, dt, i));
      if (x != y) {
        r->mismatches++;
        if (r->first_mismatch < 0) r->first_mismatch = (int64_t)i;
      }
      /* |x - y| as an unsigned 64-bit number: never negates INT64_MIN */
      uint64_t d = x >= y ? (uint64_t)x - (uint64_t)y : (uint64_t)y - (uint64_t)x;
      if (d > r->max_abs_u64) r->max_abs_u64 = d;
      double dd = (double)d;
      sumsq += dd * dd;
      if (y != 0) {
        double q = dd / fabs((double)y);
        if (q > max_rel) max_rel = q;
      }
    }
    r->n_finite = p->n;
    r->max_abs = (double)r->max_abs_u64;
    r->max_rel = max_rel;
    r->rms = p->n ? sqrt(sumsq / (double)p->n) : 0.0;
    *sumsq_out = sumsq;
  }
  r->pass = r->mismatches == 0;
}

static void compare_one(const or_pair* p, const uint8_t* cand, const uint8_t* ref, or_result* r) {
  double sumsq;
  compare_one_sum(p, cand, ref, r, &sumsq);
}

int or_compare(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
               const uint8_t* ref, uint64_t ref_bytes, or_result* out) {
  for (int i = 0; i < n_pairs; ++i)
    if (check_pair(&pairs[i], cand_bytes, ref_bytes) != 0) return -1;
  for (int i = 0; i < n_pairs; ++i) compare_one(&pairs[i], cand, ref, &out[i]);
  return 0;
}

int or_compare_sums(const or_pair* pairs, int n_pairs, const uint8_t* cand, uint64_t cand_bytes,
                    const uint8_t* ref, uint64_t ref_bytes, or_result* out, double* sumsq) {
  for (int i = 0; i < n_pairs; ++i)
    if (check_pair(&pairs[i], cand_bytes, ref_bytes) != 0) return -1;
  for (int i = 0; i < n_pairs; ++i) compare_one_sum(&pairs[i], cand, ref, &out[i], &sumsq[i]);
  return 0;
}

/* shaped outputs: a rows x cols output (row-major, row pitches in elements) */
/* compared tile by tile.  Each tile's elements are gathered in row-major   */
/* order into dense buffers and compared as one segment by the rule above;  */
/* its first mismatch is reported as the output-wide index row * cols + col.*/
int or_compare_tiles(const or_tiles* t, const uint8_t* cand, uint64_t cand_bytes, const uint8_t* ref,
                     uint64_t ref_bytes, or_result* out) {
  uint64_t sz = elem_bytes(t->dtype);
  if (sz == 0 || t->tile_rows == 0 || t->tile_cols == 0) return -1;
  if (t->cand_pitch < t->cols || t->ref_pitch < t->cols) return -1;
  if (is_float_dtype(t->dtype) && !(t->atol >= 0.0 && t->rtol >= 0.0)) return -1;
  if (t->rows && t->cols) { /* the last element of each operand lies inside its buffer */
    uint64_t xe = t->cand_offset + ((t->rows - 1) * t->cand_pitch + t->cols) * sz;
    uint64_t ye = t->ref_offset + ((t->rows - 1) * t->ref_pitch + t->cols) * sz;
    if (xe > cand_bytes || ye > ref_bytes) return -1;
  }
  uint64_t ntr = (t->rows + t->tile_rows - 1) / t->tile_rows, ntc = (t->cols + t->tile_cols - 1) / t->tile_cols;
  uint8_t* xt = (uint8_t*)malloc(t->tile_rows * t->tile_cols * sz + 1);
  uint8_t* yt = (uint8_t*)malloc(t->tile_rows * t->tile_cols * sz + 1);
  if (!xt || !yt) { free(xt); free(yt); return -1; }
  for (uint64_t i = 0; i < ntr; ++i) {
    for (uint64_t j = 0; j < ntc; ++j) {
      uint64_t r0 = i * t->tile_rows, r1 = r0 + t->tile_rows < t->rows ? r0 + t->tile_rows : t->rows;
      uint64_t c0 = j * t->tile_cols, c1 = c0 + t->tile_cols < t->cols ? c0 + t->tile_cols : t->cols;
      uint64_t w = c1 - c0, k = 0;
      for (uint64_t r = r0; r < r1; ++r, k += w) {
        memcpy(xt + k * sz, cand + t->cand_offset + (r * t->cand_pitch + c0) * sz, w * sz);
        memcpy(yt + k * sz, ref + t->ref_offset + (r * t->ref_pitch + c0) * sz, w * sz);
      }
      or_pair p = {t->dtype, t->flags, (r1 - r0) * w, 0, 0, t->atol, t->rtol};
      or_result* r = &out[i * ntc + j];
      compare_one(&p, xt, yt, r);
      if (r->first_mismatch >= 0) {
        uint64_t f = (uint64_t)r->first_mismatch;
        r->first_mismatch = (int64_t)((r0 + f / w) * t->cols + c0 + f % w);
      }
    }
  }
  free(xt);
  free(yt);
  return 0;
}

/* progressive validation (Sec. 4.2.2): stages in the given order, stop at   */
/* the first failing stage; later stages are reported as not run.            */
int or_progressive(const or_pair* stages, int n_stages, const uint8_t* cand, uint64_t cand_bytes,
                   const uint8_t* ref, uint64_t ref_bytes, or_result* out, int32_t* first_failed) {
  for (int i = 0; i < n_stages; ++i)
    if (check_pair(&stages[i], cand_bytes, ref_bytes) != 0) return -1;
  *first_failed = -1;
  for (int i = 0; i < n_stages; ++i) {
    if (*first_failed >= 0) {
      memset(&out[i], 0, sizeof(out[i]));
      out[i].first_mismatch = -1;
      out[i].state = OR_STAGE_SKIPPED;
      continue;
    }
    compare_one(&stages[i], cand, ref, &out[i]);
    if (!out[i].pass) *first_failed = i;
  }
  return 0;
}

/* ------------------------------------------------------------------------ */
/* bulk maps used by the exhaustive pins                                    */
/* ------------------------------------------------------------------------ */
void or_map_uniform(float a, float b, const uint32_t* w, uint64_t n, float* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = or_uniform_map(a, b, w[i]);
}

void or_map_box_muller(const uint32_t* w, uint64_t n_pairs, float* z) {
  for (uint64_t i = 0; i < n_pairs; ++i) or_box_muller(w[2 * i], w[2 * i + 1], &z[2 * i], &z[2 * i + 1]);
}

void or_map_f32_to_bf16(const float* x, uint64_t n, uint16_t* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = or_f32_to_bf16(x[i]);
}

void or_map_f32_to_f16(const float* x, uint64_t n, uint16_t* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = or_f32_to_f16(x[i]);
}

void or_map_perm(uint64_t N, uint64_t seed, uint32_t stream, uint64_t g0, uint64_t n, uint64_t* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = or_perm_value(N, seed, stream, g0 + i);
}

/* bucket counts of the [0, r) map over all 2^32 words */
void or_int_range_histogram(uint64_t r, uint64_t* counts) {
  for (uint64_t i = 0; i < r; ++i) counts[i] = 0;
  uint32_t w = 0;
  do {
    counts[or_int_range_map32(0, r, w)]++;
    ++w;
  } while (w != 0);
}
