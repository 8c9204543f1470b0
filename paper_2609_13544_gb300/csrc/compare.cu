// Golden-vs-candidate error signature on sm_103a.
//
// Computes, per tensor or per segment of a packed tensor list, the error
// statistics of Section IV-B-3 ("FI Assessment Scores": the error is the
// absolute difference of golden and faulty values; max, mean and variance
// of it) plus the relative error, the ULP distance, a five-way class and two
// 64-bin histograms.  Every output is exact: integer outputs bit for bit,
// sums as the exact real sum rounded once to nearest-even binary64.
//
// Stage 1 (compare_stage1): a persistent grid streams both tensors once.
// CTA b owns the contiguous element range [lo_b, lo_{b+1}) and writes one
// Partial per segment piece it touches (slot s + b).  Per element pair:
//   - bitwise-equal vectors are counted and skipped;
//   - a "window" lane (same sign and binade, golden exponent inside the CTA's
//     window of binades) is exact in float32 arithmetic and integer ops:
//     d = +-u * 2^E with u = |bits(c) - bits(g)| the ULP distance, so
//     sum |d|, sum d, sum d^2 accumulate as integers u << (e - Lb) and
//     (u << (e - Lb))^2; the log2-relative bin is the exponent difference
//     of |d| and |g|; the tolerance test is one float32 fma (exact except
//     at equality, which goes to the general path);
//   - every other lane (non-finite, sign change, other binades, outside the
//     window, tolerance ties) takes the general path, which evaluates the
//     definitions exactly in binary64 (TwoSum) and adds its sum terms to a
//     CTA-wide carry-save fixed-point accumulator in shared memory.
// Stage 2 (compare_stage2): one CTA per segment merges that segment's
// partials in a fixed order; all merged quantities are integers or exact
// values, so the result does not depend on the grid.
#include <cuda_fp16.h>

#include <cstdint>

#include "peat_internal.h"

namespace peat {
namespace {

// ---------------------------------------------------------------------------
// element types
// ---------------------------------------------------------------------------
template <int DT>
struct Tr;
template <>
struct Tr<PEAT_F32> {
  static constexpr int BYTES = 4, VEC = 4, MB = 23, BIAS = 127, EMAX = 255;
  static constexpr int UB = 12;      // window lanes need u < 2^UB
  static constexpr int LBMIN = 24;   // |d| >= 2^(e-150) stays a normal float32
  static constexpr uint32_t SIGN = 0x80000000u, MAG = 0x7FFFFFFFu, SE = 0xFF800000u, INF = 0x7F800000u;
};
template <>
struct Tr<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 10, BIAS = 15, EMAX = 31;
  static constexpr int UB = 10, LBMIN = 1;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, SE = 0xFC00u, INF = 0x7C00u;
};
template <>
struct Tr<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 7, BIAS = 127, EMAX = 255;
  static constexpr int UB = 7, LBMIN = 8;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, SE = 0xFF80u, INF = 0x7F80u;
};

// Window of binades [Lb, Lb + SHMAX]: u << (e - Lb) stays below 2^32.
template <int DT>
struct Win {
  static constexpr int SHMAX = 32 - Tr<DT>::UB;
  // keep |g| < 2^126 inside the window so the reciprocal in the rel filter stays normal
  static constexpr int LBMAX = (Tr<DT>::EMAX == 255 ? 252 : Tr<DT>::EMAX - 1) - SHMAX;
  static constexpr int NPB = 63 + Tr<DT>::UB + 1;  // private rows: ULP 1..63, rel k in [-(MB+1), UB-MB-1]
};

constexpr int HALF = BLOCK / 2;
constexpr int NPB_MAX = 63 + 12 + 1;

template <int DT>
__device__ __forceinline__ float to_f32(uint32_t b) {
  if constexpr (DT == PEAT_F32) return __uint_as_float(b);
  else if constexpr (DT == PEAT_BF16) return __uint_as_float(b << 16);
  else return __half2float(__ushort_as_half((unsigned short)b));
}

template <int DT>
__device__ __forceinline__ uint32_t lane_bits(const uint4& v, int j) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (Tr<DT>::BYTES == 4) return w[j];
  else return (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
}

template <int DT>
__device__ __forceinline__ uint32_t load_scalar(const void* base, int64_t i) {
  if constexpr (Tr<DT>::BYTES == 4) return __ldg(reinterpret_cast<const uint32_t*>(base) + i);
  else return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(base) + i);
}

__device__ __forceinline__ uint4 load_vec(const void* base, int64_t byte_off) {
  const uint4* p = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(base) + byte_off);
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// ---------------------------------------------------------------------------
// exact arithmetic helpers (binary64; used off the hot path)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void two_sum(double x, double y, double& s, double& t) {
  s = __dadd_rn(x, y);
  double yv = __dsub_rn(s, x);
  double xv = __dsub_rn(s, yv);
  t = __dadd_rn(__dsub_rn(x, xv), __dsub_rn(y, yv));
}

// x = m * 2^e, m a 53-bit integer (x finite, nonzero)
__device__ __forceinline__ uint64_t split_double(double x, int& e) {
  uint64_t b = (uint64_t)__double_as_longlong(x) & 0x7FFFFFFFFFFFFFFFull;
  int be = (int)(b >> 52);
  uint64_t m = b & 0xFFFFFFFFFFFFFull;
  if (be == 0) {
    e = -1074;
    return m;
  }
  e = be - 1075;
  return m | (1ull << 52);
}

// Signed 32-bit digits of +-m * 2^e, m < 2^106, delivered to a callback
// (digit index, signed value).  LIMB_LSB <= e and the top digit stays in range
// for every value that occurs (checked by construction of the callers).
template <class F>
__device__ __forceinline__ void for_digits(unsigned __int128 m, int e, bool neg, F&& f) {
  if (m == 0) return;
  int p = e - LIMB_LSB;
  int j = p >> 5, r = p & 31;
  uint32_t md[4] = {(uint32_t)m, (uint32_t)(m >> 32), (uint32_t)(m >> 64), (uint32_t)(m >> 96)};
  uint32_t out[5];
  out[0] = md[0] << r;
#pragma unroll
  for (int k = 1; k < 4; k++) out[k] = (md[k] << r) | (r ? (md[k - 1] >> (32 - r)) : 0u);
  out[4] = r ? (md[3] >> (32 - r)) : 0u;
#pragma unroll
  for (int k = 0; k < 5; k++)
    if (out[k] && j + k < NLIMB) f(j + k, neg ? -(int64_t)out[k] : (int64_t)out[k]);
}

// A local exact accumulator (off the hot path: rare comparisons, stage 2).
struct XAcc {
  int64_t d[NLIMB];
  __device__ void zero() {
#pragma unroll
    for (int j = 0; j < NLIMB; j++) d[j] = 0;
  }
  __device__ void add_m(unsigned __int128 m, int e, bool neg) {
    for_digits(m, e, neg, [&](int j, int64_t v) { d[j] += v; });
  }
  __device__ void add_double(double x, bool neg = false) {
    if (x == 0.0) return;
    int e;
    uint64_t m = split_double(x, e);
    add_m(m, e, neg ^ (x < 0));
  }
  __device__ void add_prod(double x, double y, bool neg = false) {
    if (x == 0.0 || y == 0.0) return;
    int ex, ey;
    uint64_t mx = split_double(x, ex), my = split_double(y, ey);
    add_m((unsigned __int128)mx * my, ex + ey, neg ^ (x < 0) ^ (y < 0));
  }
  // carry-propagate: digits 0..NLIMB-2 into [0, 2^32), top digit signed
  __device__ void normalize() {
    int64_t carry = 0;
    for (int j = 0; j < NLIMB - 1; j++) {
      int64_t v = d[j] + carry;
      carry = v >> 32;  // arithmetic shift: floor division
      d[j] = v & 0xFFFFFFFFll;
    }
    d[NLIMB - 1] += carry;
  }
  __device__ int sign() {  // after normalize
    if (d[NLIMB - 1] < 0) return -1;
    for (int j = 0; j < NLIMB; j++)
      if (d[j]) return 1;
    return 0;
  }
  __device__ void negate() {
    for (int j = 0; j < NLIMB; j++) d[j] = -d[j];
    normalize();
  }
  // round-to-nearest-even binary64 of the exact value
  __device__ double to_double() {
    normalize();
    bool neg = sign() < 0;
    if (neg) negate();
    int top = -1;
    for (int j = NLIMB - 1; j >= 0; j--)
      if (d[j]) {
        top = j;
        break;
      }
    if (top < 0) return 0.0;
    // gather the value's leading 96 bits into hi:mid:lo digits
    uint64_t dtop = (uint64_t)d[top];
    int lz = __clzll(dtop);  // >= 0; dtop < 2^63
    int msb = top * 32 + 63 - lz;  // bit index of the leading one
    // take bits [msb-63, msb] as a 64-bit window, plus a sticky flag below
    uint64_t win = 0;
    bool sticky = false;
    for (int bit = msb; bit > msb - 64; bit--) {
      win <<= 1;
      if (bit >= 0) win |= ((uint64_t)d[bit >> 5] >> (bit & 31)) & 1ull;
    }
    for (int j = 0; j < NLIMB && !sticky; j++) {
      int lo_bit = j * 32, hi_bit = j * 32 + 31;
      if (hi_bit <= msb - 64) sticky = d[j] != 0;
      else if (lo_bit <= msb - 64) {
        int nb = msb - 64 - lo_bit + 1;
        uint64_t mask = nb >= 32 ? 0xFFFFFFFFull : ((1ull << nb) - 1);
        sticky = ((uint64_t)d[j] & mask) != 0;
      }
    }
    uint64_t mant = win >> 11;              // 53 bits
    uint64_t rest = win & 0x7FFull;         // 11 bits below
    bool round = (rest >> 10) & 1;
    bool st = sticky || (rest & 0x3FF);
    if (round && (st || (mant & 1))) mant++;
    double r = ldexp((double)mant, msb - 52 + LIMB_LSB);
    return neg ? -r : r;
  }
};

// sign(a1/g1 - a2/g2) for exact pairs a = hi + lo >= 0 and g >= 0, where
// g = 0 with a > 0 means +inf and a = 0 means 0.
__device__ int cmp_rel(double h1, double l1, double g1, double h2, double l2, double g2) {
  int k1 = h1 == 0.0 ? 0 : (g1 == 0.0 ? 2 : 1);
  int k2 = h2 == 0.0 ? 0 : (g2 == 0.0 ? 2 : 1);
  if (k1 != k2) return k1 > k2 ? 1 : -1;
  if (k1 != 1) return 0;
  XAcc x;
  x.zero();
  x.add_prod(h1, g2);
  x.add_prod(l1, g2);
  x.add_prod(h2, g1, true);
  x.add_prod(l2, g1, true);
  x.normalize();
  return x.sign();
}

// sign(pair - y) for a normalised binary64 pair and a double
__device__ __forceinline__ int cmp_pair_dbl(double hi, double lo, double y) {
  if (hi != y) return hi > y ? 1 : -1;
  return lo > 0 ? 1 : (lo < 0 ? -1 : 0);
}
__device__ __forceinline__ int cmp_pair(double h1, double l1, double h2, double l2) {
  if (h1 != h2) return h1 > h2 ? 1 : -1;
  return l1 > l2 ? 1 : (l1 < l2 ? -1 : 0);
}

// float32 lower bound of a nonnegative pair value
__device__ __forceinline__ float pair_to_f32_rd(double hi, double lo) {
  float f = __double2float_rd(hi);
  if ((double)f == hi && lo < 0) f = nextafterf(f, 0.0f);
  return f;
}

// ---------------------------------------------------------------------------
// shared memory
// ---------------------------------------------------------------------------
struct Smem {
  unsigned long long hist[HBINS];
  unsigned long long sacc[NSUM][NLIMB];
  unsigned long long cnt[8];
  MaxAbs wabs[BLOCK / 32];
  MaxRel wrel[BLOCK / 32];
  MaxUlp wulp[BLOCK / 32];
  long long wff[BLOCK / 32], wfu[BLOCK / 32];
  int lb;
  uint32_t priv[NPB_MAX * HALF];  // per-thread 16-bit counters, two threads per word
};

__device__ __forceinline__ void sacc_add(Smem& sm, int which, unsigned __int128 m, int e, bool neg) {
  for_digits(m, e, neg, [&](int j, int64_t v) {
    atomicAdd(&sm.sacc[which][j], (unsigned long long)v);
  });
}
__device__ __forceinline__ void sacc_add_double(Smem& sm, int which, double x) {
  if (x == 0.0) return;
  int e;
  uint64_t m = split_double(x, e);
  sacc_add(sm, which, m, e, x < 0);
}
__device__ __forceinline__ void sacc_add_prod(Smem& sm, int which, double x, double y) {
  if (x == 0.0 || y == 0.0) return;
  int ex, ey;
  uint64_t mx = split_double(x, ex), my = split_double(y, ey);
  sacc_add(sm, which, (unsigned __int128)mx * my, ex + ey, (x < 0) ^ (y < 0));
}

// ---------------------------------------------------------------------------
// per-thread state
// ---------------------------------------------------------------------------
struct Ctx {
  float rtol, atol;
  uint32_t lb_shift;  // Lb << MB
  uint32_t win_span;  // (SHMAX + 1) << MB
  uint32_t col, inc;  // private histogram column and increment
};

struct LaneState {
  uint32_t n_eq, n_simple, n_within, n_nonfinite;
  uint32_t n_gw, n_gm, n_ga, n_gf;  // general path: within, mismatch, asym, flip
  uint64_t P, N, Q;
  uint32_t Qh;
  float abs_f, rel_f;
  uint32_t ulp_f;
  MaxAbs mabs;
  MaxRel mrel;
  int64_t ulp_idx;
  int64_t first_fin, first_ulp;
};

__device__ __forceinline__ void state_init(LaneState& st) {
  st.n_eq = st.n_simple = st.n_within = st.n_nonfinite = 0;
  st.n_gw = st.n_gm = st.n_ga = st.n_gf = 0;
  st.P = st.N = st.Q = 0;
  st.Qh = 0;
  st.abs_f = 0.0f;
  st.rel_f = 0.0f;
  st.ulp_f = 0;
  st.mabs = MaxAbs{0.0, 0.0, -1};
  st.mrel = MaxRel{0.0, 0.0, 1.0, -1};
  st.ulp_idx = -1;
  st.first_fin = st.first_ulp = -1;
}

template <int DT>
__device__ __forceinline__ void note_first(LaneState& st, uint32_t G, uint32_t C, int64_t idx) {
  using T = Tr<DT>;
  uint32_t ag = G & T::MAG, ac = C & T::MAG;
  if (st.first_fin < 0 && ag < T::INF && ac < T::INF) st.first_fin = idx;
  if (st.first_ulp < 0 && ag <= T::INF && ac <= T::INF) st.first_ulp = idx;
}

// rel filter value for a new best: RD(rel) * (1 - 2^-20)
__device__ __forceinline__ float rel_filter(double hi, double lo, double g) {
  if (g == 0.0) return __int_as_float(0x7F800000);
  double q = __ddiv_rd(hi, g);
  (void)lo;
  return __fmul_rd(__double2float_rd(q), 0.99999904632568359375f);
}

// Exact update of the maxima for a window lane (index order: idx is larger
// than every index seen so far by this thread).
template <int DT>
__device__ __noinline__ LaneState window_candidate(LaneState st, uint32_t G, uint32_t C, int64_t idx) {
  using T = Tr<DT>;
  float gf = to_f32<DT>(G), cf = to_f32<DT>(C);
  float a = fabsf(__fsub_rn(cf, gf)), ag = fabsf(gf);
  uint32_t u = (uint32_t)abs((int32_t)C - (int32_t)G);
  if (a > st.abs_f) {
    double ad = (double)a;
    bool gt = st.mabs.idx < 0 || cmp_pair_dbl(st.mabs.hi, st.mabs.lo, ad) < 0;
    if (gt) {
      st.mabs = MaxAbs{ad, 0.0, idx};
      st.abs_f = a;
    }
  }
  if (u > st.ulp_f) {
    st.ulp_f = u;
    st.ulp_idx = idx;
  }
  float r = __fmul_rn(a, rcp_approx(ag));
  if (r > st.rel_f) {
    bool gt = st.mrel.idx < 0 || cmp_rel((double)a, 0.0, (double)ag, st.mrel.hi, st.mrel.lo, st.mrel.g) > 0;
    if (gt) {
      st.mrel = MaxRel{(double)a, 0.0, (double)ag, idx};
      st.rel_f = rel_filter((double)a, 0.0, (double)ag);
    }
  }
  (void)T::MB;
  return st;
}

// The general path: the definitions evaluated exactly, any pair.
template <int DT>
__device__ __noinline__ LaneState general_lane(LaneState st, uint32_t G, uint32_t C, int64_t idx, float rtol,
                                               float atol, Smem& sm) {
  using T = Tr<DT>;
  uint32_t ag = G & T::MAG, ac = C & T::MAG;
  bool gnan = ag > T::INF, cnan = ac > T::INF, ginf = ag == T::INF, cinf = ac == T::INF;
  bool gs = (G & T::SIGN) != 0, cs = (C & T::SIGN) != 0;
  int64_t kg = gs ? -(int64_t)ag : (int64_t)ag, kc = cs ? -(int64_t)ac : (int64_t)ac;
  uint64_t u = (uint64_t)(kc > kg ? kc - kg : kg - kc);
  bool ulpdef = !gnan && !cnan;
  if (gnan || cnan || ginf || cinf) {
    st.n_nonfinite++;
    bool equal = (gnan && cnan) || (ginf && cinf && gs == cs);
    if (equal) {
      st.n_eq++;
      return st;
    }
    st.n_ga++;
    atomicAdd(&sm.hist[63], 1ull);
    atomicAdd(&sm.hist[64 + (ulpdef ? (u < 63 ? (int)u : 63) : 63)], 1ull);
    if (ulpdef && u > 0) {
      if (u > st.ulp_f || (u == st.ulp_f && idx < st.ulp_idx)) {
        st.ulp_f = (uint32_t)u;
        st.ulp_idx = idx;
      }
    }
    return st;
  }
  double gv = (double)to_f32<DT>(G), cv = (double)to_f32<DT>(C);
  double s, t;
  two_sum(cv, -gv, s, t);
  double ahi = fabs(s), alo = s < 0 ? -t : t;
  double absg = fabs(gv);
  if (ahi == 0.0) {  // numerically equal (e.g. +0 and -0)
    st.n_eq++;
    return st;
  }
  // tolerance: a <= atol + rtol*|g|, exactly (rtol*|g| is exact in binary64)
  double P = (double)rtol * absg, Tt, tt;
  two_sum((double)atol, P, Tt, tt);
  int cls;
  if (cmp_pair(ahi, alo, Tt, tt) <= 0) cls = PEAT_WITHIN_TOL;
  else if (gv != 0.0 && cv != 0.0 && gs != cs) cls = PEAT_SIGN_FLIP;
  else cls = PEAT_MISMATCH;
  if (cls == PEAT_WITHIN_TOL) st.n_gw++;
  else if (cls == PEAT_SIGN_FLIP) st.n_gf++;
  else st.n_gm++;
  // log2-relative bin
  int rb;
  if (absg == 0.0) {
    rb = 63;
  } else {
    int k = ilogb(ahi) - ilogb(absg);
    while (cmp_pair_dbl(ahi, alo, ldexp(absg, k)) < 0) k--;
    while (cmp_pair_dbl(ahi, alo, ldexp(absg, k + 1)) >= 0) k++;
    k += 48;
    rb = k < 1 ? 1 : (k > 62 ? 62 : k);
  }
  atomicAdd(&sm.hist[rb], 1ull);
  atomicAdd(&sm.hist[64 + (u < 63 ? (int)u : 63)], 1ull);
  // maxima, full (value, index) order
  {
    int c = st.mabs.idx < 0 ? 1 : cmp_pair(ahi, alo, st.mabs.hi, st.mabs.lo);
    if (c > 0 || (c == 0 && idx < st.mabs.idx)) {
      st.mabs = MaxAbs{ahi, alo, idx};
      st.abs_f = pair_to_f32_rd(ahi, alo);
    }
  }
  {
    int c = st.mrel.idx < 0 ? 1 : cmp_rel(ahi, alo, absg, st.mrel.hi, st.mrel.lo, st.mrel.g);
    if (c > 0 || (c == 0 && idx < st.mrel.idx)) {
      st.mrel = MaxRel{ahi, alo, absg, idx};
      st.rel_f = rel_filter(ahi, alo, absg);
    }
  }
  if (u > 0 && (u > st.ulp_f || (u == st.ulp_f && idx < st.ulp_idx))) {
    st.ulp_f = (uint32_t)u;
    st.ulp_idx = idx;
  }
  // exact sums: d = s + t, |d| = ahi + alo, d^2 = s^2 + 2st + t^2
  sacc_add_double(sm, 0, s);
  sacc_add_double(sm, 0, t);
  sacc_add_double(sm, 1, ahi);
  sacc_add_double(sm, 1, alo);
  sacc_add_prod(sm, 2, s, s);
  sacc_add_prod(sm, 2, s, t);
  sacc_add_prod(sm, 2, s, t);
  sacc_add_prod(sm, 2, t, t);
  return st;
}

// One lane of the fast path.  Returns via bit masks which lanes need the
// general path (gen) or an exact maxima check (cand).
template <int DT>
__device__ __forceinline__ void window_lane(LaneState& st, uint32_t G, uint32_t C, int j, const Ctx& cx,
                                            Smem& sm, uint32_t& gen, uint32_t& cand) {
  using T = Tr<DT>;
  uint32_t ag = G & T::MAG;
  bool eq = G == C;
  bool eqf = eq && ag < T::INF;
  uint32_t rel_e = ag - cx.lb_shift;
  bool inwin = rel_e < cx.win_span;
  bool sse = ((G ^ C) & T::SE) == 0;
  int32_t delta = (int32_t)C - (int32_t)G;
  uint32_t u = (uint32_t)abs(delta);
  bool simple = !eq && sse && inwin;
  if constexpr (T::UB < T::MB) simple = simple && u < (1u << T::UB);
  float gf = to_f32<DT>(G), cf = to_f32<DT>(C);
  float s = __fsub_rn(cf, gf);
  float a = fabsf(s), agf = fabsf(gf);
  float thr = __fmaf_rn(cx.rtol, agf, cx.atol);
  bool within = a < thr;
  bool tie = a == thr;
  st.n_eq += eqf ? 1u : 0u;
  bool go = simple && !tie;
  if (!go && !eqf) gen |= 1u << j;
  if (go) {
    st.n_simple++;
    st.n_within += within ? 1u : 0u;
    int k = (int)(__float_as_uint(a) - __float_as_uint(agf)) >> 23;  // floor(log2(a/|g|))
    uint32_t ub = u < 63u ? u : 63u;
    atomicAdd(&sm.priv[(ub - 1) * HALF + cx.col], cx.inc);
    atomicAdd(&sm.priv[(63 + k + T::MB + 1) * HALF + cx.col], cx.inc);
    uint32_t sh = rel_e >> T::MB;
    uint32_t V = u << sh;
    if (s > 0.0f) st.P += V;
    else st.N += V;
    uint64_t v2 = (uint64_t)V * V;
    uint64_t q = st.Q + v2;
    st.Qh += q < st.Q ? 1u : 0u;
    st.Q = q;
    float r = __fmul_rn(a, rcp_approx(agf));
    if ((a > st.abs_f) | (u > st.ulp_f) | (r > st.rel_f)) cand |= 1u << j;
  }
}

template <int DT>
__device__ __forceinline__ uint32_t nonfinite_count(const uint4& v) {
  using T = Tr<DT>;
  uint32_t n = 0;
#pragma unroll
  for (int j = 0; j < T::VEC; j++) n += (lane_bits<DT>(v, j) & T::MAG) >= T::INF ? 1u : 0u;
  return n;
}

template <int DT>
__device__ __forceinline__ void do_vector(LaneState& st, const uint4& gv, const uint4& cv, int64_t base,
                                          const Ctx& cx, Smem& sm) {
  using T = Tr<DT>;
  bool alleq = (gv.x == cv.x) & (gv.y == cv.y) & (gv.z == cv.z) & (gv.w == cv.w);
  if ((st.first_fin | st.first_ulp) < 0) {
#pragma unroll
    for (int j = 0; j < T::VEC; j++) note_first<DT>(st, lane_bits<DT>(gv, j), lane_bits<DT>(cv, j), base + j);
  }
  if (alleq) {
    st.n_eq += T::VEC;
    uint32_t nf = nonfinite_count<DT>(gv);
    st.n_eq -= nf;              // non-finite equal lanes are counted by the general path
    if (nf) {
#pragma unroll
      for (int j = 0; j < T::VEC; j++) {
        uint32_t G = lane_bits<DT>(gv, j);
        if ((G & T::MAG) >= T::INF) st = general_lane<DT>(st, G, G, base + j, cx.rtol, cx.atol, sm);
      }
    }
    return;
  }
  uint32_t gen = 0, cand = 0;
#pragma unroll
  for (int j = 0; j < T::VEC; j++)
    window_lane<DT>(st, lane_bits<DT>(gv, j), lane_bits<DT>(cv, j), j, cx, sm, gen, cand);
  while (cand) {
    int j = __ffs(cand) - 1;
    cand &= cand - 1;
    st = window_candidate<DT>(st, lane_bits<DT>(gv, j), lane_bits<DT>(cv, j), base + j);
  }
  while (gen) {
    int j = __ffs(gen) - 1;
    gen &= gen - 1;
    st = general_lane<DT>(st, lane_bits<DT>(gv, j), lane_bits<DT>(cv, j), base + j, cx.rtol, cx.atol, sm);
  }
}

template <int DT>
__device__ __forceinline__ void do_scalar(LaneState& st, uint32_t G, uint32_t C, int64_t idx, const Ctx& cx,
                                          Smem& sm) {
  if ((st.first_fin | st.first_ulp) < 0) note_first<DT>(st, G, C, idx);
  uint32_t gen = 0, cand = 0;
  window_lane<DT>(st, G, C, 0, cx, sm, gen, cand);
  if (cand) st = window_candidate<DT>(st, G, C, idx);
  if (gen) st = general_lane<DT>(st, G, C, idx, cx.rtol, cx.atol, sm);
}

// ---------------------------------------------------------------------------
// CTA ranges
// ---------------------------------------------------------------------------
template <int DT>
__host__ __device__ __forceinline__ int64_t cta_lo(int64_t b, const CompareParams& p) {
  if (b <= 0) return 0;
  if (b >= p.nctas) return p.n_total;
  constexpr int VEC = Tr<DT>::VEC;
  if (p.p0 < 0 || p.p0 >= p.n_total) return (p.n_total / p.nctas) * b + (p.n_total % p.nctas) * b / p.nctas;
  int64_t nv = (p.n_total - p.p0) / VEC;
  int64_t lo = p.p0 + ((nv / p.nctas) * b + (nv % p.nctas) * b / p.nctas) * VEC;
  return lo < p.n_total ? lo : p.n_total;
}

// the CTA whose range holds element i (0 <= i < n_total)
template <int DT>
__device__ int cta_of(int64_t i, const CompareParams& p) {
  int lo = 0, hi = p.nctas - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (cta_lo<DT>(mid, p) <= i) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// first segment s with offsets[s+1] > i
__device__ int64_t seg_of(int64_t i, const int64_t* off, int64_t nseg) {
  int64_t lo = 0, hi = nseg - 1;
  while (lo < hi) {
    int64_t mid = (lo + hi) >> 1;
    if (off[mid + 1] > i) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

// ---------------------------------------------------------------------------
// reductions
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t shfl64(uint64_t v, int src) {
  uint32_t lo = __shfl_sync(0xFFFFFFFFu, (uint32_t)v, src);
  uint32_t hi = __shfl_sync(0xFFFFFFFFu, (uint32_t)(v >> 32), src);
  return ((uint64_t)hi << 32) | lo;
}
__device__ __forceinline__ uint64_t warp_sum64(uint64_t v) {
  for (int o = 16; o > 0; o >>= 1) {
    uint32_t lo = __shfl_down_sync(0xFFFFFFFFu, (uint32_t)v, o);
    uint32_t hi = __shfl_down_sync(0xFFFFFFFFu, (uint32_t)(v >> 32), o);
    v += ((uint64_t)hi << 32) | lo;
  }
  return v;
}
__device__ __forceinline__ double shfl_d(double v, int o) {
  return __longlong_as_double((long long)
      ((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)__double_as_longlong(v), o) |
       ((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)((uint64_t)__double_as_longlong(v) >> 32), o) << 32)));
}
__device__ __forceinline__ int64_t shfl_i64(int64_t v, int o) {
  return (int64_t)((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)v, o) |
                   ((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)((uint64_t)v >> 32), o) << 32));
}

__device__ __forceinline__ bool abs_better(const MaxAbs& x, const MaxAbs& y) {  // x beats y
  if (x.idx < 0) return false;
  if (y.idx < 0) return true;
  int c = cmp_pair(x.hi, x.lo, y.hi, y.lo);
  return c > 0 || (c == 0 && x.idx < y.idx);
}
__device__ __forceinline__ bool rel_better(const MaxRel& x, const MaxRel& y) {
  if (x.idx < 0) return false;
  if (y.idx < 0) return true;
  int c = cmp_rel(x.hi, x.lo, x.g, y.hi, y.lo, y.g);
  return c > 0 || (c == 0 && x.idx < y.idx);
}
__device__ __forceinline__ bool ulp_better(const MaxUlp& x, const MaxUlp& y) {
  if (x.idx < 0) return false;
  if (y.idx < 0) return true;
  return x.u > y.u || (x.u == y.u && x.idx < y.idx);
}
__device__ __forceinline__ int64_t min_idx(int64_t a, int64_t b) {
  if (a < 0) return b;
  if (b < 0) return a;
  return a < b ? a : b;
}

// Fold the per-thread 16-bit histograms and the window sums into the CTA
// totals.  All threads call it; ends with the private counters zeroed.
template <int DT>
__device__ void fold_round(LaneState& st, Smem& sm, int lb) {
  using T = Tr<DT>;
  constexpr int NPB = Win<DT>::NPB;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // window sums: P, N (< 2^48 per round), Q as 96 bits
  uint64_t P = warp_sum64(st.P), N = warp_sum64(st.N);
  uint64_t q0 = warp_sum64(st.Q & 0xFFFFFFFFull), q1 = warp_sum64(st.Q >> 32), q2 = warp_sum64(st.Qh);
  if (lane == 0) {
    const int lexp = lb - T::BIAS - T::MB;  // weight of V's bit 0
    if (P >= N) sacc_add(sm, 0, (unsigned __int128)(P - N), lexp, false);
    else sacc_add(sm, 0, (unsigned __int128)(N - P), lexp, true);
    sacc_add(sm, 1, (unsigned __int128)P + N, lexp, false);
    unsigned __int128 Q = (unsigned __int128)q0 + ((unsigned __int128)q1 << 32) + ((unsigned __int128)q2 << 64);
    sacc_add(sm, 2, Q, 2 * lexp, false);
  }
  st.P = st.N = st.Q = 0;
  st.Qh = 0;
  __syncthreads();
  // private histograms: one warp per row
  for (int r = warp; r < NPB; r += BLOCK / 32) {
    uint32_t sum = 0;
    for (int w = lane; w < HALF; w += 32) {
      uint32_t v = sm.priv[r * HALF + w];
      sum += (v & 0xFFFFu) + (v >> 16);
      sm.priv[r * HALF + w] = 0;
    }
    sum = __reduce_add_sync(0xFFFFFFFFu, sum);
    if (lane == 0 && sum) {
      int bin = r < 63 ? 64 + r + 1 : (r - 63) - T::MB - 1 + 48;
      sm.hist[bin] += sum;
    }
  }
  __syncthreads();
}

template <int DT>
__device__ void finish_piece(LaneState& st, Smem& sm, int lb, Partial* out, int64_t n_piece) {
  fold_round<DT>(st, sm, lb);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // counts
  uint32_t c[8] = {st.n_eq, st.n_simple, st.n_within, st.n_nonfinite, st.n_gw, st.n_gm, st.n_ga, st.n_gf};
#pragma unroll
  for (int k = 0; k < 8; k++) {
    uint32_t v = __reduce_add_sync(0xFFFFFFFFu, c[k]);
    if (lane == 0 && v) atomicAdd(&sm.cnt[k], (unsigned long long)v);
  }
  // maxima: warp tournament, then across warps
  MaxAbs ma = st.mabs;
  MaxRel mr = st.mrel;
  MaxUlp mu = MaxUlp{st.ulp_f, st.ulp_idx};
  int64_t ff = st.first_fin, fu = st.first_ulp;
  for (int o = 16; o > 0; o >>= 1) {
    MaxAbs oa{shfl_d(ma.hi, o), shfl_d(ma.lo, o), shfl_i64(ma.idx, o)};
    MaxRel orl{shfl_d(mr.hi, o), shfl_d(mr.lo, o), shfl_d(mr.g, o), shfl_i64(mr.idx, o)};
    MaxUlp ou{(uint64_t)shfl_i64((int64_t)mu.u, o), shfl_i64(mu.idx, o)};
    int64_t off = shfl_i64(ff, o), ofu = shfl_i64(fu, o);
    if (lane + o < 32) {
      if (abs_better(oa, ma)) ma = oa;
      if (rel_better(orl, mr)) mr = orl;
      if (ulp_better(ou, mu)) mu = ou;
      ff = min_idx(ff, off);
      fu = min_idx(fu, ofu);
    }
  }
  if (lane == 0) {
    sm.wabs[warp] = ma;
    sm.wrel[warp] = mr;
    sm.wulp[warp] = mu;
    sm.wff[warp] = ff;
    sm.wfu[warp] = fu;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < BLOCK / 32; w++) {
      if (abs_better(sm.wabs[w], ma)) ma = sm.wabs[w];
      if (rel_better(sm.wrel[w], mr)) mr = sm.wrel[w];
      if (ulp_better(sm.wulp[w], mu)) mu = sm.wulp[w];
      ff = min_idx(ff, sm.wff[w]);
      fu = min_idx(fu, sm.wfu[w]);
    }
    out->mabs = ma;
    out->mrel = mr;
    out->mulp = mu;
    out->first_fin = ff;
    out->first_ulp = fu;
    unsigned long long* cn = sm.cnt;
    out->cnt[PEAT_EXACT] = cn[0];
    out->cnt[PEAT_WITHIN_TOL] = cn[2] + cn[4];
    out->cnt[PEAT_MISMATCH] = (cn[1] - cn[2]) + cn[5];
    out->cnt[PEAT_NAN_INF_ASYM] = cn[6];
    out->cnt[PEAT_SIGN_FLIP] = cn[7];
    out->nonfinite = cn[3];
    out->n = (uint64_t)n_piece;
  }
  if (threadIdx.x < NSUM) {  // normalise the carry-save digits of one sum
    int k = threadIdx.x;
    long long carry = 0;
    for (int j = 0; j < NLIMB; j++) {
      long long v = (long long)sm.sacc[k][j] + carry;
      if (j < NLIMB - 1) {
        carry = v >> 32;
        v &= 0xFFFFFFFFll;
      }
      out->limbs[k][j] = v;
    }
  }
  for (int b = threadIdx.x; b < HBINS; b += BLOCK) out->hist[b] = sm.hist[b];
  __syncthreads();
  // reset the CTA totals for the next piece
  for (int b = threadIdx.x; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  if (threadIdx.x < 8) sm.cnt[threadIdx.x] = 0;
  state_init(st);
  __syncthreads();
}

// ---------------------------------------------------------------------------
// stage 1
// ---------------------------------------------------------------------------
template <int DT>
__global__ void __launch_bounds__(BLOCK, 2) compare_stage1(CompareParams p) {
  using T = Tr<DT>;
  constexpr int VEC = T::VEC;
  constexpr int SHMAX = Win<DT>::SHMAX;
  // lanes per thread per round stay below 2^16 (16-bit private counters)
  constexpr int64_t ROUND_VECS = (int64_t)BLOCK * (65535 / VEC);
  __shared__ Smem sm;
  const int tid = threadIdx.x;
  for (int b = tid; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = tid; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  for (int j = tid; j < Win<DT>::NPB * HALF; j += BLOCK) sm.priv[j] = 0;
  if (tid < 8) sm.cnt[tid] = 0;
  const int64_t lo = cta_lo<DT>(blockIdx.x, p), hi = cta_lo<DT>((int64_t)blockIdx.x + 1, p);
  LaneState st;
  state_init(st);
  Ctx cx;
  cx.rtol = p.rtol;
  cx.atol = p.atol;
  cx.win_span = (uint32_t)(SHMAX + 1) << T::MB;
  cx.col = tid & (HALF - 1);
  cx.inc = tid < HALF ? 1u : 65536u;
  __syncthreads();
  if (lo >= hi) return;
  int64_t s = seg_of(lo, p.offsets, p.nseg);
  int64_t pb = lo;
  while (pb < hi) {
    while (p.offsets[s + 1] <= pb) s++;  // skip empty segments
    const int64_t pe = min(hi, p.offsets[s + 1]);
    // vector body [vb, ve) on the aligned grid, scalar head and tail
    int64_t vb = pe, ve = pe;
    if (p.p0 >= 0 && p.p0 < p.n_total) {
      int64_t a0 = pb <= p.p0 ? p.p0 : p.p0 + ((pb - p.p0 + VEC - 1) / VEC) * VEC;
      int64_t a1 = pe <= p.p0 ? p.p0 : p.p0 + ((pe - p.p0) / VEC) * VEC;
      if (a0 < a1) vb = a0, ve = a1;
    }
    const int64_t nvec = (ve - vb) / VEC;
    // window of binades from the largest golden exponent in the first vectors
    if (tid == 0) sm.lb = 0;
    __syncthreads();
    if (tid < nvec) {
      uint4 gv = load_vec(p.g, (vb + (int64_t)tid * VEC) * T::BYTES);
      uint32_t emax = 0;
#pragma unroll
      for (int j = 0; j < VEC; j++) {
        uint32_t e = (lane_bits<DT>(gv, j) & T::MAG) >> T::MB;
        if (e < (uint32_t)T::EMAX && e > emax) emax = e;
      }
      atomicMax(&sm.lb, (int)emax);
    }
    __syncthreads();
    int lb = sm.lb + 2 - SHMAX;
    lb = lb < T::LBMIN ? T::LBMIN : (lb > Win<DT>::LBMAX ? Win<DT>::LBMAX : lb);
    cx.lb_shift = (uint32_t)lb << T::MB;
    // scalar head: fewer than VEC elements, or the whole piece in scalar mode
    // (then in rounds of at most 65535 elements per thread)
    {
      const int64_t h_end = vb < pe ? vb : pe;
      constexpr int64_t ROUND_ELEMS = (int64_t)BLOCK * 65535;
      for (int64_t r0 = pb; r0 < h_end; r0 += ROUND_ELEMS) {
        const int64_t r1 = min(h_end, r0 + ROUND_ELEMS);
        for (int64_t i = r0 + tid; i < r1; i += BLOCK)
          do_scalar<DT>(st, load_scalar<DT>(p.g, i), load_scalar<DT>(p.c, i), i, cx, sm);
        if (r1 < h_end) fold_round<DT>(st, sm, lb);
      }
    }
    // vector body in rounds
    for (int64_t r0 = 0; r0 < nvec; r0 += ROUND_VECS) {
      const int64_t r1 = min(nvec, r0 + ROUND_VECS);
      int64_t v = r0 + tid;
      // two vectors in flight per thread
      for (; v + BLOCK < r1; v += 2 * BLOCK) {
        const int64_t e0 = vb + v * VEC, e1 = vb + (v + BLOCK) * VEC;
        uint4 g0 = load_vec(p.g, e0 * T::BYTES), c0 = load_vec(p.c, e0 * T::BYTES);
        uint4 g1 = load_vec(p.g, e1 * T::BYTES), c1 = load_vec(p.c, e1 * T::BYTES);
        do_vector<DT>(st, g0, c0, e0, cx, sm);
        do_vector<DT>(st, g1, c1, e1, cx, sm);
      }
      if (v < r1) {
        const int64_t e0 = vb + v * VEC;
        uint4 g0 = load_vec(p.g, e0 * T::BYTES), c0 = load_vec(p.c, e0 * T::BYTES);
        do_vector<DT>(st, g0, c0, e0, cx, sm);
      }
      if (r1 < nvec) fold_round<DT>(st, sm, lb);
    }
    // scalar tail (fewer than VEC elements), after the body: lanes stay in index order
    if (vb < ve && ve < pe)
      for (int64_t i = ve + tid; i < pe; i += BLOCK)
        do_scalar<DT>(st, load_scalar<DT>(p.g, i), load_scalar<DT>(p.c, i), i, cx, sm);
    finish_piece<DT>(st, sm, lb, p.partials + s + blockIdx.x, pe - pb);
    pb = pe;
  }
}

// ---------------------------------------------------------------------------
// stage 2: one CTA per segment, fixed-order merge, exact finalisation
// ---------------------------------------------------------------------------
__device__ double rel_value(const MaxRel& m) {
  if (m.hi == 0.0) return 0.0;
  if (m.g == 0.0) return __longlong_as_double(0x7FF0000000000000ll);
  // RN64((hi+lo)/g): the candidate with the smallest exact residual, ties to even
  double q0 = __ddiv_rn(m.hi, m.g);
  double q = q0;
  for (int i = 0; i < 3; i++) q = nextafter(q, 0.0);
  double best = q;
  XAcc bres;
  bool have = false;
  for (int step = 0; step < 7; step++, q = nextafter(q, __longlong_as_double(0x7FF0000000000000ll))) {
    XAcc r;
    r.zero();
    r.add_double(m.hi);
    r.add_double(m.lo);
    r.add_prod(q, m.g, true);
    r.normalize();
    if (r.sign() < 0) r.negate();
    if (!have) {
      best = q, bres = r, have = true;
      continue;
    }
    int c = 0;
    for (int j = NLIMB - 1; j >= 0 && c == 0; j--)
      if (r.d[j] != bres.d[j]) c = r.d[j] > bres.d[j] ? 1 : -1;
    bool qeven = (__double_as_longlong(q) & 1) == 0, beven = (__double_as_longlong(best) & 1) == 0;
    if (c < 0 || (c == 0 && qeven && !beven)) best = q, bres = r;
  }
  return best;
}

template <int DT>
__global__ void __launch_bounds__(BLOCK) compare_stage2(CompareParams p) {
  const int64_t s = blockIdx.x;
  const int tid = threadIdx.x;
  const int64_t s0 = p.offsets[s], s1 = p.offsets[s + 1];
  __shared__ MaxAbs wabs[BLOCK / 32];
  __shared__ MaxRel wrel[BLOCK / 32];
  __shared__ MaxUlp wulp[BLOCK / 32];
  __shared__ long long wff[BLOCK / 32], wfu[BLOCK / 32];
  __shared__ unsigned long long hist[HBINS];
  __shared__ unsigned long long cnt[8];
  __shared__ long long limbs[NSUM][NLIMB];
  peat_stats_t* out = p.stats + s;
  if (s1 <= s0) {  // empty segment
    if (tid == 0) {
      peat_stats_t z;
      memset(&z, 0, sizeof(z));
      z.argmax_abs = z.argmax_rel = z.argmax_ulp = -1;
      z.rtol_eff = p.rtol;
      z.atol_eff = p.atol;
      *out = z;
    }
    if (p.hist)
      for (int b = tid; b < HBINS; b += BLOCK) p.hist[s * HBINS + b] = 0;
    return;
  }
  const int b0 = cta_of<DT>(s0, p), b1 = cta_of<DT>(s1 - 1, p);
  auto slot = [&](int b) -> const Partial* { return p.partials + s + b; };
  auto nonempty = [&](int b) { return cta_lo<DT>(b, p) < cta_lo<DT>((int64_t)b + 1, p); };
  // integer parts: one thread per counter / bin / digit, partials in order
  if (tid < HBINS) {
    unsigned long long h = 0;
    for (int b = b0; b <= b1; b++)
      if (nonempty(b)) h += slot(b)->hist[tid];
    hist[tid] = h;
  }
  if (tid >= HBINS && tid < HBINS + 7) {
    int k = tid - HBINS;
    unsigned long long v = 0;
    for (int b = b0; b <= b1; b++)
      if (nonempty(b)) v += k < 5 ? slot(b)->cnt[k] : (k == 5 ? slot(b)->nonfinite : slot(b)->n);
    cnt[k] = v;
  }
  if (tid >= 160 && tid < 160 + NSUM * NLIMB) {
    int k = (tid - 160) / NLIMB, j = (tid - 160) % NLIMB;
    long long v = 0;
    for (int b = b0; b <= b1; b++)
      if (nonempty(b)) v += slot(b)->limbs[k][j];
    limbs[k][j] = v;
  }
  // maxima
  MaxAbs ma{0.0, 0.0, -1};
  MaxRel mr{0.0, 0.0, 1.0, -1};
  MaxUlp mu{0, -1};
  int64_t ff = -1, fu = -1;
  for (int b = b0 + tid; b <= b1; b += BLOCK) {
    if (!nonempty(b)) continue;
    const Partial* q = slot(b);
    if (abs_better(q->mabs, ma)) ma = q->mabs;
    if (rel_better(q->mrel, mr)) mr = q->mrel;
    if (ulp_better(q->mulp, mu)) mu = q->mulp;
    ff = min_idx(ff, q->first_fin);
    fu = min_idx(fu, q->first_ulp);
  }
  const int lane = tid & 31, warp = tid >> 5;
  for (int o = 16; o > 0; o >>= 1) {
    MaxAbs oa{shfl_d(ma.hi, o), shfl_d(ma.lo, o), shfl_i64(ma.idx, o)};
    MaxRel orl{shfl_d(mr.hi, o), shfl_d(mr.lo, o), shfl_d(mr.g, o), shfl_i64(mr.idx, o)};
    MaxUlp ou{(uint64_t)shfl_i64((int64_t)mu.u, o), shfl_i64(mu.idx, o)};
    int64_t off = shfl_i64(ff, o), ofu = shfl_i64(fu, o);
    if (lane + o < 32) {
      if (abs_better(oa, ma)) ma = oa;
      if (rel_better(orl, mr)) mr = orl;
      if (ulp_better(ou, mu)) mu = ou;
      ff = min_idx(ff, off);
      fu = min_idx(fu, ofu);
    }
  }
  if (lane == 0) {
    wabs[warp] = ma;
    wrel[warp] = mr;
    wulp[warp] = mu;
    wff[warp] = ff;
    wfu[warp] = fu;
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < BLOCK / 32; w++) {
      if (abs_better(wabs[w], ma)) ma = wabs[w];
      if (rel_better(wrel[w], mr)) mr = wrel[w];
      if (ulp_better(wulp[w], mu)) mu = wulp[w];
      ff = min_idx(ff, wff[w]);
      fu = min_idx(fu, wfu[w]);
    }
    peat_stats_t r;
    r.n = cnt[6];
    r.count[PEAT_EXACT] = cnt[0];
    for (int k = 1; k < PEAT_NCLASS; k++) r.count[k] = cnt[k];
    r.n_finite = cnt[6] - cnt[5];
    // maxima: only strictly positive errors are recorded; a zero maximum is
    // attained first at the first finite (or ULP-defined) pair
    if (ma.idx >= 0) {
      r.max_abs = ma.hi;  // hi = RN64(|d|)
      r.argmax_abs = ma.idx - s0;
    } else {
      r.max_abs = 0.0;
      r.argmax_abs = ff >= 0 ? ff - s0 : -1;
    }
    if (mr.idx >= 0) {
      r.max_rel = rel_value(mr);
      r.argmax_rel = mr.idx - s0;
    } else {
      r.max_rel = 0.0;
      r.argmax_rel = ff >= 0 ? ff - s0 : -1;
    }
    if (mu.idx >= 0) {
      r.max_ulp = mu.u;
      r.argmax_ulp = mu.idx - s0;
    } else {
      r.max_ulp = 0;
      r.argmax_ulp = fu >= 0 ? fu - s0 : -1;
    }
    double sums[NSUM];
    for (int k = 0; k < NSUM; k++) {
      XAcc x;
      for (int j = 0; j < NLIMB; j++) x.d[j] = limbs[k][j];
      sums[k] = x.to_double();
    }
    r.sum_signed = sums[0];
    r.sum_abs = sums[1];
    r.sum_sq = sums[2];
    r.rtol_eff = p.rtol;
    r.atol_eff = p.atol;
    *out = r;
  }
  if (p.hist) {
    for (int b = tid; b < HBINS; b += BLOCK) {
      unsigned long long h = hist[b];
      if (b == 0 || b == 64) h += cnt[0];  // EXACT pairs: rel bin 0 and ULP bin 0
      p.hist[s * HBINS + b] = h;
    }
  }
}

template <int DT>
cudaError_t launch_t(const CompareParams& p, cudaStream_t st) {
  compare_stage1<DT><<<p.nctas, BLOCK, 0, st>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (p.nseg > 0) compare_stage2<DT><<<(unsigned)p.nseg, BLOCK, 0, st>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_compare(int dtype, const CompareParams& p, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return launch_t<PEAT_F32>(p, s);
    case PEAT_F16: return launch_t<PEAT_F16>(p, s);
    case PEAT_BF16: return launch_t<PEAT_BF16>(p, s);
  }
  return cudaErrorInvalidValue;
}

int compare_ctas_per_sm() { return 2; }
size_t compare_partial_bytes() { return sizeof(Partial); }

}  // namespace peat
