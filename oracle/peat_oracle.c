/*
 * peat_oracle.c -- TEST INFRASTRUCTURE ONLY (the oracle).
 *
 * A plain, slow, sequential and exact CPU statement of what the PEAT
 * error-signature path computes.  Only tests/, __graft_entry__.smoke() and
 * bench.py's cpu_baseline leg may call it.  It shares no code, header,
 * table or constant generator with the CUDA library.
 *
 * What the paper fixes (Section IV-B-3, "FI Assessment Scores"; Alg. 1 and
 * Alg. 2, the final Err step): the error between a golden output g and a
 * fault-injected output c is their absolute difference, and a recorded
 * tensor is scored by the maximum, the mean and the variance of that error
 * (the mean of the top 10 % is a separate score, not part of this pass).
 *
 * What the paper leaves open, and the reading taken here (all quantities are
 * evaluated exactly over the reals, then rounded once to nearest-even):
 *  - non-finite pairs: both NaN, or both infinite with equal sign, are EXACT;
 *    any other pair with a NaN or an infinity is NAN_INF_ASYM.  Non-finite
 *    pairs never enter the sums or the abs/rel maxima.
 *  - finite pairs: d = c - g, a = |d|.  EXACT iff a = 0 (so +0 vs -0 is
 *    EXACT).  WITHIN_TOL iff 0 < a <= atol + rtol*|g| with rtol, atol the
 *    float32 roundings of the requested tolerances (the torch.isclose form
 *    used in Section III-A, golden as the reference).  SIGN_FLIP iff not yet
 *    classified, g != 0, c != 0 and their sign bits differ.  MISMATCH
 *    otherwise.
 *  - rel = a/|g| (0 if a = 0; +inf if g = 0 < a).  Rel histogram bin 0 holds
 *    a = 0 (and equal non-finite pairs); bins 1..62 hold
 *    k = floor(log2(a/|g|)) at bin clamp(k + 48, 1, 62); bin 63 holds g = 0 < a
 *    and every NAN_INF_ASYM pair.
 *  - ULP distance u = |key(c) - key(g)| with key(x) = +mag or -mag by the
 *    sign bit (mag = bit pattern without the sign), so +0 and -0 both map to
 *    0 and +-Inf sit one step past the largest finite value.  ULP bin
 *    min(u, 63); a pair with a NaN has no ULP distance: it goes to bin 63
 *    (bin 0 when both are NaN) and is left out of max_ulp.
 *  - maxima take the lowest index on ties, decided by exact comparison.
 *  - sums run over finite pairs: sum |d|, sum d^2 and sum d, accumulated in a
 *    fixed-point integer wide enough to hold every term exactly.
 *
 * Floating-point model: IEEE binary64 with round-to-nearest-even and no
 * contraction (build with -ffp-contract=off); every float32 operation in the
 * injector is written out explicitly so the order of roundings is the one
 * stated in its comments.
 */
#include "peat_oracle.h"

#include <float.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Exact fixed-point accumulator (Kulisch's long accumulator): a two's       */
/* complement integer of ACC_W 64-bit words whose bit 0 weighs 2^ACC_LSB.    */
/* It holds every double (down to 2^-1074), every product of two doubles     */
/* (down to 2^-2148, up to 2^2048 with the factor 4 of a scaled difference)  */
/* and sums of up to 2^60 such products.                                     */
/* ------------------------------------------------------------------------ */
#define ACC_W ORC_ACC_WORDS
#define ACC_LSB ORC_ACC_LSB

typedef struct {
  uint64_t w[ACC_W];
} acc_t;

typedef unsigned __int128 u128;

static void acc_zero(acc_t* a) { memset(a, 0, sizeof(*a)); }

/* a += (neg ? -1 : +1) * mag * 2^e */
static void acc_add_mag(acc_t* a, u128 mag, int e, int neg) {
  if (mag == 0) return;
  int p = e - ACC_LSB;
  if (p < 0 || p + 128 > (ACC_W - 1) * 64) abort(); /* outside the exact range */
  int limb = p / 64, off = p % 64;
  uint64_t lo = (uint64_t)mag, hi = (uint64_t)(mag >> 64);
  uint64_t part[3];
  if (off == 0) {
    part[0] = lo;
    part[1] = hi;
    part[2] = 0;
  } else {
    part[0] = lo << off;
    part[1] = (hi << off) | (lo >> (64 - off));
    part[2] = hi >> (64 - off);
  }
  if (!neg) {
    uint64_t carry = 0;
    for (int j = limb; j < ACC_W; j++) {
      u128 add = (j - limb < 3 ? part[j - limb] : 0);
      u128 s = (u128)a->w[j] + add + carry;
      a->w[j] = (uint64_t)s;
      carry = (uint64_t)(s >> 64);
      if (j - limb >= 2 && carry == 0) break;
    }
  } else {
    uint64_t borrow = 0;
    for (int j = limb; j < ACC_W; j++) {
      u128 sub = (u128)(j - limb < 3 ? part[j - limb] : 0) + borrow;
      borrow = ((u128)a->w[j] < sub) ? 1 : 0;
      a->w[j] = (uint64_t)((u128)a->w[j] - sub);
      if (j - limb >= 2 && borrow == 0) break;
    }
  }
}

/* split a finite nonzero double into x = m * 2^e with m a 53-bit integer */
static uint64_t dbl_split(double x, int* e) {
  int ex;
  double m = frexp(fabs(x), &ex); /* m in [0.5, 1) */
  *e = ex - 53;
  return (uint64_t)ldexp(m, 53);
}

static void acc_add_double(acc_t* a, double x, int neg) {
  if (x == 0.0) return;
  int e;
  uint64_t m = dbl_split(x, &e);
  acc_add_mag(a, (u128)m, e, neg ^ (x < 0));
}

/* a += (neg ? -1 : 1) * x * y, exactly */
static void acc_add_product(acc_t* a, double x, double y, int neg) {
  if (x == 0.0 || y == 0.0) return;
  int ex, ey;
  uint64_t mx = dbl_split(x, &ex), my = dbl_split(y, &ey);
  acc_add_mag(a, (u128)mx * (u128)my, ex + ey, neg ^ (x < 0) ^ (y < 0));
}

static int acc_sign(const acc_t* a) {
  if (a->w[ACC_W - 1] >> 63) return -1;
  for (int j = 0; j < ACC_W; j++)
    if (a->w[j]) return 1;
  return 0;
}

static void acc_negate(acc_t* a) {
  uint64_t carry = 1;
  for (int j = 0; j < ACC_W; j++) {
    u128 s = (u128)(~a->w[j]) + carry;
    a->w[j] = (uint64_t)s;
    carry = (uint64_t)(s >> 64);
  }
}

static int acc_bit(const acc_t* a, int k) {
  if (k < 0) return 0;
  return (int)((a->w[k / 64] >> (k % 64)) & 1u);
}

/* round-to-nearest-even double of the exact value */
static double acc_to_double(const acc_t* in) {
  acc_t a = *in;
  int neg = acc_sign(&a) < 0;
  if (neg) acc_negate(&a);
  int top = -1;
  for (int j = ACC_W - 1; j >= 0 && top < 0; j--)
    if (a.w[j]) top = j * 64 + 63 - __builtin_clzll(a.w[j]);
  if (top < 0) return 0.0;
  /* the last kept bit: 53 significant bits, but none below 2^-1074 */
  int low = top - 52;
  if (low + ACC_LSB < -1074) low = -1074 - ACC_LSB;
  uint64_t mant = 0;
  for (int k = top; k >= low; k--) mant = (mant << 1) | (uint64_t)acc_bit(&a, k);
  int round = acc_bit(&a, low - 1);
  int sticky = 0;
  for (int k = low - 2; k >= 0 && !sticky; k--) sticky = acc_bit(&a, k);
  if (round && (sticky || (mant & 1u))) mant++;
  double r = ldexp((double)mant, low + ACC_LSB); /* +inf past the largest double */
  return neg ? -r : r;
}

/* magnitude comparison of two exact values: sign(|x| - |y|) */
static int acc_cmp_abs(const acc_t* x, const acc_t* y) {
  acc_t ax = *x, ay = *y;
  if (acc_sign(&ax) < 0) acc_negate(&ax);
  if (acc_sign(&ay) < 0) acc_negate(&ay);
  for (int j = ACC_W - 1; j >= 0; j--) {
    if (ax.w[j] != ay.w[j]) return ax.w[j] > ay.w[j] ? 1 : -1;
  }
  return 0;
}

double orc_exact_sum(const double* x, int64_t n) {
  acc_t a;
  acc_zero(&a);
  for (int64_t i = 0; i < n; i++) acc_add_double(&a, x[i], 0);
  return acc_to_double(&a);
}

double orc_exact_dot(const double* x, const double* y, int64_t n) {
  acc_t a;
  acc_zero(&a);
  for (int64_t i = 0; i < n; i++) acc_add_product(&a, x[i], y[i], 0);
  return acc_to_double(&a);
}

/* ------------------------------------------------------------------------ */
/* Decoding of the element types, straight from IEEE 754 binary16 and      */
/* binary32, the bfloat16 layout (top half of a binary32) and the two 8-bit */
/* formats of the OCP FP8 specification: E5M2 (IEEE-like: exponent bias 15, */
/* infinities and NaNs at the all-ones exponent) and E4M3 "fn" (bias 7, no  */
/* infinities, the only NaN is S.1111.111, so S.1111.110 = 448 is finite).  */
/* ------------------------------------------------------------------------ */
typedef struct {
  int nan, inf, sign;
  double v;     /* exact value when finite (signed; -0.0 for negative zero) */
  uint64_t mag; /* bit pattern without the sign bit */
} val_t;

static uint64_t raw_bits(const void* base, int64_t i, int dtype) {
  if (dtype == ORC_F64) {
    uint64_t b;
    memcpy(&b, (const char*)base + 8 * i, 8);
    return b;
  }
  if (dtype == ORC_F32) {
    uint32_t b;
    memcpy(&b, (const char*)base + 4 * i, 4);
    return b;
  }
  if (dtype == ORC_F8E4M3 || dtype == ORC_F8E5M2) return ((const uint8_t*)base)[i];
  uint16_t h;
  memcpy(&h, (const char*)base + 2 * i, 2);
  return h;
}

static val_t decode(uint64_t b, int dtype) {
  val_t r;
  memset(&r, 0, sizeof(r));
  int sbit, ebits, mbits, bias;
  if (dtype == ORC_F64) {
    sbit = 63, ebits = 11, mbits = 52, bias = 1023;
  } else if (dtype == ORC_F32) {
    sbit = 31, ebits = 8, mbits = 23, bias = 127;
  } else if (dtype == ORC_F16) {
    sbit = 15, ebits = 5, mbits = 10, bias = 15;
  } else if (dtype == ORC_BF16) {
    sbit = 15, ebits = 8, mbits = 7, bias = 127;
  } else if (dtype == ORC_F8E5M2) {
    sbit = 7, ebits = 5, mbits = 2, bias = 15;
  } else {
    sbit = 7, ebits = 4, mbits = 3, bias = 7;
  }
  r.sign = (int)((b >> sbit) & 1u);
  r.mag = b & ((1ull << sbit) - 1u);
  uint64_t e = r.mag >> mbits, m = r.mag & ((1ull << mbits) - 1u);
  uint64_t emax = (1ull << ebits) - 1u;
  if (dtype == ORC_F8E4M3) {
    if (r.mag == 0x7Fu) { /* the only NaN; the rest of the top binade is finite */
      r.nan = 1;
      return r;
    }
  } else if (e == emax) {
    r.nan = (m != 0);
    r.inf = (m == 0);
    return r;
  }
  double x;
  if (e == 0)
    x = ldexp((double)m, 1 - bias - mbits); /* subnormal */
  else
    x = ldexp((double)(m | (1ull << mbits)), (int)e - bias - mbits);
  r.v = r.sign ? -x : x;
  return r;
}

int64_t orc_ulp_key(uint64_t bits, int dtype) {
  val_t v = decode(bits, dtype);
  return v.sign ? -(int64_t)v.mag : (int64_t)v.mag;
}

/* ------------------------------------------------------------------------ */
/* Exact comparisons on the error of one pair.  The error d = c - g is held  */
/* as an unevaluated sum s + t of two doubles (Knuth's TwoSum, TAOCP vol. 2 */
/* 4.2.2), which is exact for any two finite doubles without overflow.       */
/* ------------------------------------------------------------------------ */
static void two_sum(double x, double y, double* s, double* t) {
  double sum = x + y;
  double yv = sum - x;
  double xv = sum - yv;
  *s = sum;
  *t = (x - xv) + (y - yv);
}

typedef struct {
  double s, t; /* |d| = (s + t) 2^sc exactly, s = RN64(|d| / 2^sc) */
  int sc;      /* 1 when c - g overflows binary64 (then both were halved), else 0 */
} mag2_t;

/* a += (neg ? -1 : +1) * x * 2^sc and the same for a product */
static void acc_add_double_sc(acc_t* a, double x, int sc, int neg) {
  if (x == 0.0) return;
  int e;
  uint64_t m = dbl_split(x, &e);
  acc_add_mag(a, (u128)m, e + sc, neg ^ (x < 0));
}
static void acc_add_product_sc(acc_t* a, double x, double y, int sc, int neg) {
  if (x == 0.0 || y == 0.0) return;
  int ex, ey;
  uint64_t mx = dbl_split(x, &ex), my = dbl_split(y, &ey);
  acc_add_mag(a, (u128)mx * (u128)my, ex + ey + sc, neg ^ (x < 0) ^ (y < 0));
}
static void acc_add_mag2(acc_t* x, mag2_t a, int neg) {
  acc_add_double_sc(x, a.s, a.sc, neg);
  acc_add_double_sc(x, a.t, a.sc, neg);
}

/* sign(a - y 2^k) for an exact two-term a and a double y >= 0 */
static int cmp_mag_dbl_pow2(mag2_t a, double y, int k) {
  acc_t x;
  acc_zero(&x);
  acc_add_mag2(&x, a, 0);
  acc_add_double_sc(&x, y, k, 1);
  return acc_sign(&x);
}

static int cmp_mag(mag2_t a, mag2_t b) {
  acc_t x;
  acc_zero(&x);
  acc_add_mag2(&x, a, 0);
  acc_add_mag2(&x, b, 1);
  return acc_sign(&x);
}

/* relative error a/|g|: 0 when a = 0, +inf when g = 0 < a */
typedef struct {
  mag2_t a;
  double absg;
} rel_t;

static int rel_kind(rel_t r) { /* 0: zero, 1: finite positive, 2: +inf */
  if (r.a.s == 0.0) return 0;
  if (r.absg == 0.0) return 2;
  return 1;
}

/* sign(r1 - r2), exactly: for finite positive values a1/g1 vs a2/g2 compare
 * a1*g2 with a2*g1 (both g > 0). */
static int cmp_rel(rel_t r1, rel_t r2) {
  int k1 = rel_kind(r1), k2 = rel_kind(r2);
  if (k1 != k2) return k1 > k2 ? 1 : -1;
  if (k1 != 1) return 0;
  acc_t x;
  acc_zero(&x);
  acc_add_product_sc(&x, r1.a.s, r2.absg, r1.a.sc, 0);
  acc_add_product_sc(&x, r1.a.t, r2.absg, r1.a.sc, 0);
  acc_add_product_sc(&x, r2.a.s, r1.absg, r2.a.sc, 1);
  acc_add_product_sc(&x, r2.a.t, r1.absg, r2.a.sc, 1);
  return acc_sign(&x);
}

/* the last bit of the stored significand (normal or subnormal) */
static int mant_is_even(double q) {
  uint64_t b;
  memcpy(&b, &q, 8);
  return (b & 1u) == 0;
}

/* RN64 of a finite positive quotient a/absg: the candidate double with the
 * smallest exact residual |a - q*absg|, ties to the even significand.  The
 * exact quotient lies within two units in the last place of RN64(a.s/absg),
 * so a window of four steps either side holds the answer. */
static double rel_value(rel_t r) {
  int k = rel_kind(r);
  if (k == 0) return 0.0;
  if (k == 2) return INFINITY;
  /* past the rounding threshold of the largest double, (2^54 - 1) 2^970, the quotient rounds to +inf */
  {
    acc_t x;
    acc_zero(&x);
    acc_add_mag2(&x, r.a, 0);
    int eg;
    uint64_t mg = dbl_split(r.absg, &eg);
    acc_add_mag(&x, (u128)mg * (((u128)1 << 54) - 1), eg + 970, 1);
    if (acc_sign(&x) >= 0) return INFINITY;
  }
  double q0 = ldexp(r.a.s / r.absg, r.a.sc);
  if (!(q0 <= DBL_MAX)) q0 = DBL_MAX;
  double best = 0.0;
  acc_t best_res;
  int have = 0;
  double q = q0;
  for (int i = 0; i < 4; i++) q = nextafter(q, 0.0);
  for (int step = 0; step < 9; step++, q = nextafter(q, INFINITY)) {
    if (isinf(q)) break;
    acc_t res;
    acc_zero(&res);
    acc_add_mag2(&res, r.a, 0);
    acc_add_product(&res, q, r.absg, 1);
    if (!have) {
      best = q, best_res = res, have = 1;
      continue;
    }
    int c = acc_cmp_abs(&res, &best_res);
    if (c < 0 || (c == 0 && mant_is_even(q) && !mant_is_even(best))) best = q, best_res = res;
  }
  return best;
}

/* floor(log2(a/absg)) for a > 0, absg > 0: the integer k with
 * absg*2^k <= a < absg*2^(k+1), found from an estimate by exact comparisons */
static int rel_log2_floor(mag2_t a, double absg) {
  int k = ilogb(a.s) + a.sc - ilogb(absg);
  while (cmp_mag_dbl_pow2(a, absg, k) < 0) k--;
  while (cmp_mag_dbl_pow2(a, absg, k + 1) >= 0) k++;
  return k;
}

/* ------------------------------------------------------------------------ */
/* The signature of one tensor.                                              */
/* ------------------------------------------------------------------------ */
static int tol_ok(double rtol, double atol, double* rtol_eff, double* atol_eff) {
  if (!(rtol >= 0.0) || !(atol >= 0.0)) return 0; /* also rejects NaN */
  float r32 = (float)rtol, a32 = (float)atol;     /* RN32 of the requested values */
  if (isinf(r32) || isinf(a32)) return 0;
  *rtol_eff = (double)r32;
  *atol_eff = (double)a32;
  return 1;
}

/* words, if not NULL, receives the exact sums of |c-g| and of (c-g)^2 over
 * the finite pairs: 2 * ORC_ACC_WORDS words (see orc_compare_segmented_sums) */
static void compare_range(const void* gb, const void* cb, int64_t n, int dtype, double rtol,
                          double atol, orc_stats* st, uint64_t* hist, uint64_t* words) {
  memset(st, 0, sizeof(*st));
  memset(hist, 0, sizeof(uint64_t) * 128);
  st->n = (uint64_t)n;
  st->rtol_eff = rtol;
  st->atol_eff = atol;
  st->argmax_abs = st->argmax_rel = st->argmax_ulp = -1;

  acc_t s_abs, s_sq, s_signed;
  acc_zero(&s_abs);
  acc_zero(&s_sq);
  acc_zero(&s_signed);

  int have_abs = 0, have_rel = 0, have_ulp = 0;
  mag2_t best_abs = {0.0, 0.0, 0};
  rel_t best_rel = {{0.0, 0.0, 0}, 0.0};
  uint64_t best_ulp = 0;

  for (int64_t i = 0; i < n; i++) {
    val_t g = decode(raw_bits(gb, i, dtype), dtype);
    val_t c = decode(raw_bits(cb, i, dtype), dtype);
    int gfin = !g.nan && !g.inf, cfin = !c.nan && !c.inf;
    int cls, relbin, ulpbin;
    int ulp_defined = !g.nan && !c.nan;
    int64_t kg = g.sign ? -(int64_t)g.mag : (int64_t)g.mag;
    int64_t kc = c.sign ? -(int64_t)c.mag : (int64_t)c.mag;
    /* |kc - kg| < 2^64: the unsigned difference is exact */
    uint64_t u = kc >= kg ? (uint64_t)kc - (uint64_t)kg : (uint64_t)kg - (uint64_t)kc;

    if (!gfin || !cfin) {
      int equal = (g.nan && c.nan) || (g.inf && c.inf && g.sign == c.sign);
      cls = equal ? ORC_EXACT : ORC_NAN_INF_ASYM;
      relbin = equal ? 0 : 63;
      if (!ulp_defined)
        ulpbin = equal ? 0 : 63;
      else
        ulpbin = u < 63 ? (int)u : 63;
    } else {
      st->n_finite++;
      double s, t;
      int sc = 0;
      two_sum(c.v, -g.v, &s, &t); /* d = c - g = s + t exactly */
      if (!isfinite(s)) {           /* binary64 operands whose difference overflows: */
        two_sum(0.5 * c.v, -0.5 * g.v, &s, &t); /* halving is exact at that size */
        sc = 1;
      }
      mag2_t a = (s < 0.0) ? (mag2_t){-s, -t, sc} : (mag2_t){s, t, sc};
      double absg = fabs(g.v);

      /* classification, in precedence order */
      if (a.s == 0.0) {
        cls = ORC_EXACT;
      } else {
        acc_t x; /* a - (atol + rtol*|g|) */
        acc_zero(&x);
        acc_add_mag2(&x, a, 0);
        acc_add_double(&x, atol, 1);
        acc_add_product(&x, rtol, absg, 1);
        if (acc_sign(&x) <= 0)
          cls = ORC_WITHIN_TOL;
        else if (g.v != 0.0 && c.v != 0.0 && g.sign != c.sign)
          cls = ORC_SIGN_FLIP;
        else
          cls = ORC_MISMATCH;
      }

      /* log2-relative-error bin */
      if (a.s == 0.0)
        relbin = 0;
      else if (absg == 0.0)
        relbin = 63;
      else {
        int k = rel_log2_floor(a, absg) + 48;
        relbin = k < 1 ? 1 : (k > 62 ? 62 : k);
      }
      ulpbin = u < 63 ? (int)u : 63;

      /* maxima, lowest index on ties */
      if (!have_abs || cmp_mag(a, best_abs) > 0) {
        best_abs = a;
        st->argmax_abs = i;
        have_abs = 1;
      }
      rel_t r = {a, absg};
      if (!have_rel || cmp_rel(r, best_rel) > 0) {
        best_rel = r;
        st->argmax_rel = i;
        have_rel = 1;
      }

      /* exact sums: d, |d| and d^2 = (s^2 + 2st + t^2) 4^sc */
      acc_add_double_sc(&s_signed, s, sc, 0);
      acc_add_double_sc(&s_signed, t, sc, 0);
      acc_add_mag2(&s_abs, a, 0);
      acc_add_product_sc(&s_sq, s, s, 2 * sc, 0);
      acc_add_product_sc(&s_sq, s, t, 2 * sc, 0);
      acc_add_product_sc(&s_sq, s, t, 2 * sc, 0);
      acc_add_product_sc(&s_sq, t, t, 2 * sc, 0);
    }

    if (ulp_defined && (!have_ulp || u > best_ulp)) {
      best_ulp = u;
      st->argmax_ulp = i;
      have_ulp = 1;
    }
    st->count[cls]++;
    hist[relbin]++;
    hist[64 + ulpbin]++;
  }

  if (have_abs) {
    acc_t x;
    acc_zero(&x);
    acc_add_mag2(&x, best_abs, 0);
    st->max_abs = acc_to_double(&x);
  }
  if (have_rel) st->max_rel = rel_value(best_rel);
  st->max_ulp = best_ulp;
  st->sum_abs = acc_to_double(&s_abs);
  st->sum_sq = acc_to_double(&s_sq);
  st->sum_signed = acc_to_double(&s_signed);
  if (words) {
    memcpy(words, s_abs.w, sizeof(s_abs.w));
    memcpy(words + ACC_W, s_sq.w, sizeof(s_sq.w));
  }
}

static int dtype_ok(int dtype) { return dtype == ORC_F32 || dtype == ORC_F16 || dtype == ORC_BF16; }
/* the compare (and the isclose grid built on it) also takes the 8-bit formats */
static int dtype_ok_cmp(int dtype) {
  return dtype_ok(dtype) || dtype == ORC_F8E4M3 || dtype == ORC_F8E5M2 || dtype == ORC_F64;
}
static int dtype_size(int dtype) {
  return dtype == ORC_F64 ? 8 : dtype == ORC_F32 ? 4 : (dtype == ORC_F16 || dtype == ORC_BF16 ? 2 : 1);
}

int orc_compare(const void* g, const void* c, int64_t n, int dtype, double rtol, double atol,
                orc_stats* st, uint64_t* hist) {
  double r, a;
  if (!dtype_ok_cmp(dtype) || n < 0 || !st || !hist || (n > 0 && (!g || !c))) return ORC_BAD_ARG;
  if (!tol_ok(rtol, atol, &r, &a)) return ORC_BAD_ARG;
  compare_range(g, c, n, dtype, r, a, st, hist, NULL);
  return ORC_OK;
}

int orc_compare_segmented(const void* g, const void* c, const int64_t* offsets, int64_t nseg,
                          int dtype, double rtol, double atol, orc_stats* st, uint64_t* hist) {
  return orc_compare_segmented_sums(g, c, offsets, nseg, dtype, rtol, atol, st, hist, NULL);
}

int orc_compare_segmented_sums(const void* g, const void* c, const int64_t* offsets, int64_t nseg,
                               int dtype, double rtol, double atol, orc_stats* st, uint64_t* hist,
                               uint64_t* words) {
  double r, a;
  if (!dtype_ok_cmp(dtype) || nseg < 0 || !offsets || (nseg > 0 && (!st || !hist))) return ORC_BAD_ARG;
  if (!tol_ok(rtol, atol, &r, &a)) return ORC_BAD_ARG;
  if (offsets[0] != 0) return ORC_BAD_ARG;
  for (int64_t s = 0; s < nseg; s++)
    if (offsets[s + 1] < offsets[s]) return ORC_BAD_ARG;
  if (offsets[nseg] > 0 && (!g || !c)) return ORC_BAD_ARG;
  int sz = dtype_size(dtype);
  for (int64_t s = 0; s < nseg; s++) {
    int64_t b = offsets[s], e = offsets[s + 1];
    compare_range((const char*)g + sz * b, (const char*)c + sz * b, e - b, dtype, r, a, st + s,
                  hist + 128 * s, words ? words + (size_t)s * 2 * ACC_W : NULL);
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Mean of the top errors (Section IV-B-3, "Mean of Top 10% Errors").  Every  */
/* finite |d| is kept exactly as s + t (s = RN64(|d|)); sorting on (s, t)   */
/* orders the exact values (RN64 is monotone, and equal s leave t1 - t2 as  */
/* the exact difference); the k largest are added in the exact accumulator. */
/* ------------------------------------------------------------------------ */
static int cmp_mag2_desc(const void* x, const void* y) {
  const mag2_t* a = (const mag2_t*)x;
  const mag2_t* b = (const mag2_t*)y;
  if (a->s != b->s) return a->s > b->s ? -1 : 1;
  if (a->t != b->t) return a->t > b->t ? -1 : 1;
  return 0;
}

/* RN-even double of (value of a) / k for a >= 0 and k >= 1: the value is
 * shifted up 128 bits before an exact long division, so the quotient carries
 * at least 64 significant bits and the remainder only sets the sticky bit. */
static double acc_div_rn(const acc_t* in, uint64_t k) {
  acc_t a = *in, q;
  for (int j = ACC_W - 1; j >= 2; j--) a.w[j] = a.w[j - 2];
  a.w[1] = a.w[0] = 0;
  u128 rem = 0;
  for (int j = ACC_W - 1; j >= 0; j--) {
    u128 cur = (rem << 64) | a.w[j];
    q.w[j] = (uint64_t)(cur / k);
    rem = cur % k;
  }
  int top = -1;
  for (int j = ACC_W - 1; j >= 0 && top < 0; j--)
    if (q.w[j]) top = j * 64 + 63 - __builtin_clzll(q.w[j]);
  if (top < 0) return 0.0;
  uint64_t mant = 0;
  for (int b = top; b > top - 53; b--) mant = (mant << 1) | (uint64_t)acc_bit(&q, b);
  int round = acc_bit(&q, top - 53);
  int sticky = rem != 0;
  for (int b = top - 54; b >= 0 && !sticky; b--) sticky = acc_bit(&q, b);
  if (round && (sticky || (mant & 1u))) mant++;
  return ldexp((double)mant, top - 52 + ACC_LSB - 128);
}

int orc_topk_mean(const void* g, const void* c, int64_t n, int dtype, uint64_t num, uint64_t den, orc_topk* out) {
  if (!dtype_ok(dtype) || n < 0 || !out || (n > 0 && (!g || !c)) || den == 0 || num == 0 || num > den)
    return ORC_BAD_ARG;
  memset(out, 0, sizeof(*out));
  mag2_t* m = (mag2_t*)malloc(sizeof(mag2_t) * (size_t)(n > 0 ? n : 1));
  if (!m) abort();
  uint64_t nf = 0;
  for (int64_t i = 0; i < n; i++) {
    val_t vg = decode(raw_bits(g, i, dtype), dtype), vc = decode(raw_bits(c, i, dtype), dtype);
    if (vg.nan || vg.inf || vc.nan || vc.inf) continue;
    double s, t;
    two_sum(vc.v, -vg.v, &s, &t); /* d = s + t exactly */
    m[nf].s = fabs(s);
    m[nf].t = s < 0 ? -t : t;     /* |d| = |s| + (sign of s) t */
    m[nf].sc = 0;                 /* these element types never overflow binary64 */
    nf++;
  }
  out->n_finite = nf;
  /* k = ceil(nf * num / den), exact */
  u128 prod = (u128)nf * num;
  uint64_t k = (uint64_t)((prod + den - 1) / den);
  out->k = k;
  if (k > 0) {
    qsort(m, (size_t)nf, sizeof(mag2_t), cmp_mag2_desc);
    acc_t a;
    acc_zero(&a);
    for (uint64_t i = 0; i < k; i++) {
      acc_add_double(&a, m[i].s, 0);
      acc_add_double(&a, m[i].t, 0);
    }
    out->threshold = m[k - 1].s;
    out->sum = acc_to_double(&a);
    out->mean = acc_div_rn(&a, k);
  }
  free(m);
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Context statistics (Section IV-C-2): every finite element decoded exactly */
/* and added, and its square added, in the fixed-point accumulator.          */
/* ------------------------------------------------------------------------ */
int orc_tensor_stats(const void* x, int64_t n, int dtype, orc_tstats* out) {
  if (!dtype_ok(dtype) || n < 0 || !out || (n > 0 && !x)) return ORC_BAD_ARG;
  memset(out, 0, sizeof(*out));
  out->n = (uint64_t)n;
  acc_t s1, s2;
  acc_zero(&s1);
  acc_zero(&s2);
  for (int64_t i = 0; i < n; i++) {
    val_t v = decode(raw_bits(x, i, dtype), dtype);
    if (v.nan) {
      out->n_nan++;
      continue;
    }
    if (v.inf) {
      out->n_inf++;
      continue;
    }
    /* extremes by value, -0 below +0 */
    if (out->n_finite == 0 || v.v < out->min || (v.v == out->min && signbit(v.v) && !signbit(out->min)))
      out->min = v.v;
    if (out->n_finite == 0 || v.v > out->max || (v.v == out->max && !signbit(v.v) && signbit(out->max)))
      out->max = v.v;
    out->n_finite++;
    acc_add_double(&s1, fabs(v.v), v.v < 0);
    acc_add_product(&s2, v.v, v.v, 0);
  }
  memcpy(out->sum_words, s1.w, sizeof(s1.w));
  memcpy(out->sum_sq_words, s2.w, sizeof(s2.w));
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Pseudo-error injector.                                                    */
/* Randomness: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random  */
/* numbers: as easy as 1, 2, 3", SC'11), key = the 64-bit seed, counter =    */
/* (element or draw index low/high word, model index, stream tag).           */
/* ------------------------------------------------------------------------ */
#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u
#define TAG_ELEM 0x454C454Du /* per-element draws */
#define TAG_POS 0x504F5331u  /* position draws of the fixed-count models */
#define TAG_CLASS 0x434C5353u /* NaN/Inf class of a fired element */

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; round++) {
    if (round > 0) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)PHILOX_M0 * c0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

static void draw(uint64_t seed, uint64_t index, uint32_t model, uint32_t tag, uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)index, (uint32_t)(index >> 32), model, tag};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  orc_philox4x32_10(ctr, key, out);
}

/* ---- float32 elementary functions, written out from their series so the
 * device injector can follow the same sequence of float32 roundings. ----- */
static float f32_from_bits(uint32_t b) {
  float f;
  memcpy(&f, &b, 4);
  return f;
}
static uint32_t f32_bits(float f) {
  uint32_t b;
  memcpy(&b, &f, 4);
  return b;
}

/* natural log of a positive normal float32.  Reduction x = m * 2^e with
 * m in [sqrt(1/2), sqrt(2)], then log m = 2 atanh(f), f = (m-1)/(m+1), from
 * the series 2(f + f^3/3 + ... + f^11/11); ln 2 split into a 12-bit head
 * (so e*head is exact) and a float32 tail. */
float orc_logf(float x) {
  const float C3 = 0x1.555556p-2f, C5 = 0x1.99999ap-3f, C7 = 0x1.24924ap-3f;
  const float C9 = 0x1.c71c72p-4f, C11 = 0x1.745d18p-4f;
  const float LN2_HI = 0x1.62ep-1f, LN2_LO = 0x1.0bfbe8p-15f, SQRT2 = 0x1.6a09e6p+0f;
  uint32_t b = f32_bits(x);
  int e = (int)(b >> 23) - 127;
  float m = f32_from_bits((b & 0x7FFFFFu) | 0x3F800000u);
  if (m > SQRT2) {
    m = m * 0.5f;
    e += 1;
  }
  float f = (m - 1.0f) / (m + 1.0f);
  float f2 = f * f;
  float p = fmaf(f2, C11, C9);
  p = fmaf(f2, p, C7);
  p = fmaf(f2, p, C5);
  p = fmaf(f2, p, C3);
  float tf = f + f;
  float tf3 = tf * f2;
  float lm = fmaf(tf3, p, tf);
  float ef = (float)e;
  return fmaf(ef, LN2_HI, fmaf(ef, LN2_LO, lm));
}

/* cos(2*pi*u) and sin(2*pi*u) for u in [0, 1): quadrant reduction on u
 * (exact: u = q/4 + r), then the Taylor series of cos and sin of x = 2 pi r,
 * |x| <= pi/4, and the quadrant's signs and swap:
 * cos(x + q pi/2), sin(x + q pi/2) for q = 0..3. */
static void sincos2pi(float u, float* s_out, float* c_out) {
  const float TWO_PI = 0x1.921fb6p+2f;
  const float I2 = 0x1p-1f, I4 = 0x1.555556p-5f, I6 = 0x1.6c16c2p-10f, I8 = 0x1.a01a02p-16f,
              I10 = 0x1.27e4fcp-22f;
  const float I3 = 0x1.555556p-3f, I5 = 0x1.111112p-7f, I7 = 0x1.a01a02p-13f, I9 = 0x1.71de3ap-19f;
  float q = rintf(u * 4.0f);
  float r = u - q * 0.25f;
  float x = r * TWO_PI;
  float x2 = x * x;
  float cp = fmaf(x2, -I10, I8);
  cp = fmaf(x2, cp, -I6);
  cp = fmaf(x2, cp, I4);
  cp = fmaf(x2, cp, -I2);
  float cosx = fmaf(x2, cp, 1.0f);
  float sp = fmaf(x2, I9, -I7);
  sp = fmaf(x2, sp, I5);
  sp = fmaf(x2, sp, -I3);
  float x3 = x * x2;
  float sinx = fmaf(x3, sp, x);
  switch ((int)q & 3) {
    case 0: *c_out = cosx; *s_out = sinx; break;
    case 1: *c_out = -sinx; *s_out = cosx; break;
    case 2: *c_out = -cosx; *s_out = -sinx; break;
    default: *c_out = sinx; *s_out = -cosx; break;
  }
}

float orc_cos2pi(float u) {
  float s, c;
  sincos2pi(u, &s, &c);
  return c;
}

float orc_sin2pi(float u) {
  float s, c;
  sincos2pi(u, &s, &c);
  return s;
}

/* Box-Muller: from u1 in (0, 1] and u2 in [0, 1), each the top 24 bits of a
 * Philox word, the two independent normals r cos(2 pi u2) and
 * r sin(2 pi u2), r = sqrt(-2 ln u1). */
void orc_normal_pair_from_words(uint32_t w0, uint32_t w1, float z[2]) {
  float u1 = (float)((w0 >> 8) + 1u) * 0x1p-24f;
  float u2 = (float)(w1 >> 8) * 0x1p-24f;
  float l = orc_logf(u1);
  float r = sqrtf(-2.0f * l);
  float s, c;
  sincos2pi(u2, &s, &c);
  z[0] = r * c;
  z[1] = r * s;
}

/* float32 -> binary16 bit pattern, round to nearest even or toward zero */
static uint16_t f32_to_f16(float x, int rtz) {
  uint32_t b = f32_bits(x);
  uint32_t sign = (b >> 16) & 0x8000u;
  uint32_t mag = b & 0x7FFFFFFFu;
  if (mag > 0x7F800000u) return (uint16_t)(sign | 0x7E00u);
  if (mag == 0x7F800000u) return (uint16_t)(sign | 0x7C00u);
  if (mag < 0x00800000u) return (uint16_t)sign; /* float32 subnormals are below half the smallest binary16 step */
  int e32 = (int)(mag >> 23);
  uint32_t m = (mag & 0x7FFFFFu) | 0x800000u; /* value = m * 2^(e32-150) */
  int e16 = e32 - 112;                        /* binary16 biased exponent */
  int q_exp = (e16 < 1 ? 1 : e16) - 25;       /* exponent of one binary16 step */
  int shift = q_exp - (e32 - 150);            /* low bits of m below that step */
  uint32_t q, rem, half;
  if (shift >= 32) {
    q = 0, rem = 1, half = 0x80000000u; /* nonzero remainder far below half a step */
  } else {
    q = m >> shift;
    rem = m & ((1u << shift) - 1u);
    half = 1u << (shift - 1);
  }
  if (!rtz && (rem > half || (rem == half && (q & 1u)))) q++;
  uint32_t bits = (e16 >= 1) ? ((uint32_t)(e16 - 1) << 10) + q : q;
  if (bits >= 0x7C00u) bits = rtz ? 0x7BFFu : 0x7C00u;
  return (uint16_t)(sign | bits);
}

static float f16_to_f32(uint16_t h) {
  val_t v = decode(h, ORC_F16);
  if (v.nan) return f32_from_bits(((uint32_t)(h & 0x8000u) << 16) | 0x7FC00000u);
  if (v.inf) return v.sign ? -INFINITY : INFINITY;
  return (float)v.v;
}

/* float32 -> bfloat16 bit pattern */
static uint16_t f32_to_bf16(float x, int rtz) {
  uint32_t b = f32_bits(x);
  if ((b & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((b >> 16) | 0x0040u);
  if (rtz) return (uint16_t)(b >> 16);
  uint32_t lsb = (b >> 16) & 1u;
  return (uint16_t)((b + 0x7FFFu + lsb) >> 16);
}

static float load_f32(const void* p, int64_t i, int dtype) {
  uint32_t b = raw_bits(p, i, dtype);
  if (dtype == ORC_F32) return f32_from_bits(b);
  if (dtype == ORC_BF16) return f32_from_bits(b << 16);
  return f16_to_f32((uint16_t)b);
}

static void store_f32(void* p, int64_t i, int dtype, float y) {
  if (dtype == ORC_F32) {
    memcpy((char*)p + 4 * i, &y, 4);
    return;
  }
  uint16_t h = (dtype == ORC_F16) ? f32_to_f16(y, 0) : f32_to_bf16(y, 0);
  memcpy((char*)p + 2 * i, &h, 2);
}

static int is_finite_bits(uint32_t b, int dtype) {
  val_t v = decode(b, dtype);
  return !v.nan && !v.inf;
}

static uint64_t bernoulli_threshold(double rate) {
  double t = floor(rate * 4294967296.0);
  if (t < 0.0) t = 0.0;
  if (t > 4294967296.0) t = 4294967296.0;
  return (uint64_t)t;
}

/* uniform integer in [0, n) from a 64-bit word: high half of word * n */
static uint64_t uniform_below(uint64_t word, uint64_t n) { return (uint64_t)(((u128)word * n) >> 64); }

int orc_inject(void* dst, const void* src, int64_t n, int dtype, const orc_inject_model* models,
               int nmodels, uint64_t seed, uint64_t* counts) {
  if (!dtype_ok(dtype) || n < 0 || nmodels < 0 || (nmodels > 0 && !models) || !counts) return ORC_BAD_ARG;
  if (n > 0 && (!dst || !src)) return ORC_BAD_ARG;
  int width = dtype == ORC_F32 ? 32 : 16;
  for (int m = 0; m < nmodels; m++) {
    const orc_inject_model* md = &models[m];
    if (md->kind < 0 || md->kind >= ORC_INJ_NKIND) return ORC_BAD_ARG;
    if (md->kind <= ORC_INJ_BITFLIP && (md->k < 0 || md->k > n)) return ORC_BAD_ARG;
    if (md->kind == ORC_INJ_BITFLIP &&
        (md->bit_lo < 0 || md->bit_hi < md->bit_lo || md->bit_hi >= width))
      return ORC_BAD_ARG;
    if ((md->kind == ORC_INJ_NAN_INF || md->kind == ORC_INJ_SIGNFLIP) && !(md->x >= 0.0 && md->x <= 1.0))
      return ORC_BAD_ARG;
    if (md->kind >= ORC_INJ_REL_GAUSS && md->kind <= ORC_INJ_BIAS && !isfinite(md->x)) return ORC_BAD_ARG;
    if (md->kind >= ORC_INJ_CAST_F16_RNE && dtype != ORC_F32) return ORC_BAD_ARG;
  }
  int sz = dtype_size(dtype);
  memmove(dst, src, (size_t)n * (size_t)sz);
  for (int m = 0; m < nmodels; m++) {
    const orc_inject_model* md = &models[m];
    uint64_t fired = 0;
    if (md->kind <= ORC_INJ_BITFLIP) {
      /* k distinct positions, in the order they are drawn */
      char* taken = (char*)calloc((size_t)(n > 0 ? n : 1), 1);
      if (!taken) abort();
      for (uint64_t j = 0; fired < (uint64_t)md->k; j++) {
        uint32_t w[4];
        draw(seed, j, (uint32_t)m, TAG_POS, w);
        uint64_t pos = uniform_below(((uint64_t)w[1] << 32) | w[0], (uint64_t)n);
        if (taken[pos]) continue;
        taken[pos] = 1;
        fired++;
        if (md->kind == ORC_INJ_RZ) {
          store_f32(dst, (int64_t)pos, dtype, 0.0f);
        } else if (md->kind == ORC_INJ_RV) {
          uint64_t from = uniform_below(((uint64_t)w[3] << 32) | w[2], (uint64_t)n);
          memcpy((char*)dst + sz * pos, (const char*)src + sz * from, (size_t)sz);
        } else {
          uint32_t span = (uint32_t)(md->bit_hi - md->bit_lo + 1);
          uint32_t bit = (uint32_t)md->bit_lo + (uint32_t)(((uint64_t)w[2] * span) >> 32);
          uint32_t b = raw_bits(dst, (int64_t)pos, dtype) ^ (1u << bit);
          if (sz == 4)
            memcpy((char*)dst + 4 * pos, &b, 4);
          else {
            uint16_t h = (uint16_t)b;
            memcpy((char*)dst + 2 * pos, &h, 2);
          }
        }
      }
      free(taken);
    } else {
      uint64_t thr = bernoulli_threshold(md->x);
      float x32 = (float)md->x;
      for (int64_t i = 0; i < n; i++) {
        /* one draw serves the block of four elements 4d .. 4d+3: element i
         * takes word i mod 4, or the normal its word pair gives (r cos for
         * the first element of the pair, r sin for the second) */
        uint32_t w[4];
        draw(seed, (uint64_t)i >> 2, (uint32_t)m, TAG_ELEM, w);
        int j = (int)(i & 3);
        uint32_t b = raw_bits(dst, i, dtype);
        if (md->kind == ORC_INJ_NAN_INF || md->kind == ORC_INJ_SIGNFLIP) {
          if ((uint64_t)w[j] >= thr) continue;
          fired++;
          uint32_t nb;
          if (md->kind == ORC_INJ_SIGNFLIP) {
            nb = b ^ (dtype == ORC_F32 ? 0x80000000u : 0x8000u);
          } else {
            uint32_t cw[4];
            draw(seed, (uint64_t)i, (uint32_t)m, TAG_CLASS, cw);
            uint32_t sel = cw[0] >> 30; /* 0,1: NaN; 2: +Inf; 3: -Inf */
            if (dtype == ORC_F32)
              nb = sel < 2 ? 0x7FC00000u : (sel == 2 ? 0x7F800000u : 0xFF800000u);
            else if (dtype == ORC_F16)
              nb = sel < 2 ? 0x7E00u : (sel == 2 ? 0x7C00u : 0xFC00u);
            else
              nb = sel < 2 ? 0x7FC0u : (sel == 2 ? 0x7F80u : 0xFF80u);
          }
          if (sz == 4)
            memcpy((char*)dst + 4 * i, &nb, 4);
          else {
            uint16_t h = (uint16_t)nb;
            memcpy((char*)dst + 2 * i, &h, 2);
          }
          continue;
        }
        if (!is_finite_bits(b, dtype)) continue; /* non-finite values pass through */
        fired++;
        float x = load_f32(dst, i, dtype);
        float y;
        float zp[2] = {0.0f, 0.0f};
        if (md->kind == ORC_INJ_REL_GAUSS || md->kind == ORC_INJ_ADD_GAUSS)
          orc_normal_pair_from_words(w[j & 2], w[(j & 2) + 1], zp);
        float z = zp[j & 1];
        if (md->kind == ORC_INJ_REL_GAUSS) {
          float scale = fmaf(x32, z, 1.0f); /* RN32(1 + sigma*z) */
          y = x * scale;
        } else if (md->kind == ORC_INJ_ADD_GAUSS) {
          y = fmaf(x32, z, x); /* RN32(x + sigma*z) */
        } else if (md->kind == ORC_INJ_BIAS) {
          y = fmaf(x32, fabsf(x), x); /* RN32(x + alpha*|x|) */
        } else {
          int rtz = (md->kind == ORC_INJ_CAST_F16_RTZ || md->kind == ORC_INJ_CAST_BF16_RTZ);
          if (md->kind <= ORC_INJ_CAST_F16_RTZ)
            y = f16_to_f32(f32_to_f16(x, rtz));
          else
            y = f32_from_bits((uint32_t)f32_to_bf16(x, rtz) << 16);
        }
        store_f32(dst, i, dtype, y);
      }
    }
    counts[m] = fired;
  }
  return ORC_OK;
}
