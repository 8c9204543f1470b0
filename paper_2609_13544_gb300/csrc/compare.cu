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
// CTA b owns the contiguous element range [lo_b, lo_{b+1}); per segment piece
// it touches it adds its integer totals (counts, histograms, sum digits) to
// the segment's accumulator with atomics and writes its maxima to slot s + b.
// Per element pair:
//   - bitwise-equal vectors are counted and skipped;
//   - a "window" lane -- same sign, at most one binade apart (ULP distance
//     u < 2^UB), both operands' steps at least 2^Lexp, |d| < 2^(24+Lexp) --
//     is exact in float32 and integer arithmetic: d = c - g is exact in
//     float32, V = |d| / 2^Lexp is an integer below 2^24, so sum |d|, sum d
//     and sum d^2 accumulate as integers; the log2-relative bin is the
//     exponent difference of |d| and |g| read from their bit patterns; the
//     tolerance test is one float32 fma, exact except at equality;
//   - every other lane (non-finite, sign change, zeros, wide gaps, outside
//     the window, tolerance ties) takes the general path, which evaluates the
//     definitions exactly with float32 error-free transforms and integer
//     digits, adding its sum terms to a CTA-wide carry-save fixed-point
//     accumulator in shared memory.
// Binary64 arithmetic is avoided in stage 1 (GB300 runs it at a small
// fraction of float32 rate); binary64 values appear only as containers.
// Stage 2 (compare_stage2): one CTA per segment merges the maxima of that
// segment's pieces, rounds the exact sums once and clears the accumulator;
// all merged quantities are integers or exact values, so the result does not
// depend on the grid or on the order of the atomics.
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
  static constexpr int UB = 12;       // window lanes need u < 2^UB
  static constexpr int LBMIN = 24;    // keeps 2^Lexp >= 2^-126 (normal float32)
  static constexpr int LBMAX = 221;   // keeps |g| < 2^126 (normal reciprocal)
  static constexpr uint32_t SIGN = 0x80000000u, MAG = 0x7FFFFFFFu, INF = 0x7F800000u;
};
template <>
struct Tr<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 10, BIAS = 15, EMAX = 31;
  static constexpr int UB = 10, LBMIN = 1, LBMAX = 30;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, INF = 0x7C00u;
};
template <>
struct Tr<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 7, BIAS = 127, EMAX = 255;
  static constexpr int UB = 7, LBMIN = 8, LBMAX = 221;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, INF = 0x7F80u;
};

// Private per-thread histogram rows: ULP bins 1..NU, then the log2-relative
// bins window lanes reach, k in [KLO, KHI] (fp16 goldens may be subnormal,
// whose ratios reach 2^MB).  ULP bins above NU use shared counters.
constexpr int NU = 15;
template <int DT>
struct Rows {
  static constexpr int KLO = -(Tr<DT>::MB + 1);
  static constexpr int KHI = DT == PEAT_F16 ? Tr<DT>::MB - 1 : Tr<DT>::UB - Tr<DT>::MB;
  static constexpr int NPB = NU + KHI - KLO + 1;
};
constexpr int HALF = BLOCK / 2;
constexpr int NPB_MAX = NU + 9 + 11 + 1;

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

// ---- bulk-copy (TMA) staging: mbarrier + cp.async.bulk, waits bounded -----
__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(unsigned long long* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
// global -> shared bulk copy of `bytes` (16-byte aligned, multiple of 16), completing on bar
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, unsigned long long* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(dst)),
               "l"(src), "r"(bytes), "r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ bool mbar_test(unsigned long long* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// wait for phase `parity` of bar to complete, giving up after `limit` polls
// (limit 0: give up without polling)
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, uint32_t parity, uint32_t limit) {
  for (uint32_t it = 0; it < limit; it++)
    if (mbar_test(bar, parity)) return true;
  return false;
}
// order earlier generic-proxy accesses of the stage before the next bulk write into it
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
constexpr uint32_t DRAIN_LIMIT = 1u << 26;  // polls before a drain wait gives up (far beyond any copy)

// ---------------------------------------------------------------------------
// exact integer digits
// ---------------------------------------------------------------------------
// x = m * 2^e with m an integer (x finite, nonzero); float32 and binary64
__device__ __forceinline__ uint32_t split_float(float x, int& e) {
  uint32_t b = __float_as_uint(x) & 0x7FFFFFFFu;
  uint32_t be = b >> 23, m = b & 0x7FFFFFu;
  if (be == 0) {
    e = -149;
    return m;
  }
  e = (int)be - 150;
  return m | 0x800000u;
}
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

// Signed 32-bit digits of +-m * 2^e (m < 2^128), delivered to f(digit, value).
// Every value that occurs is a multiple of 2^LIMB_LSB and below 2^352.
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

// A local exact accumulator: integer digits only (off the hot path).
struct XAcc {
  int64_t d[NLIMB];
  __device__ void zero() {
#pragma unroll
    for (int j = 0; j < NLIMB; j++) d[j] = 0;
  }
  __device__ void add_m(unsigned __int128 m, int e, bool neg) {
    for_digits(m, e, neg, [&](int j, int64_t v) { d[j] += v; });
  }
  // +-x * 2^sc
  __device__ void add_f(float x, bool neg = false, int sc = 0) {
    if (x == 0.0f) return;
    int e;
    uint32_t m = split_float(x, e);
    add_m(m, e + sc, neg ^ (x < 0));
  }
  __device__ void add_prod_f(float x, float y, bool neg = false, int sc = 0) {
    if (x == 0.0f || y == 0.0f) return;
    int ex, ey;
    uint32_t mx = split_float(x, ex), my = split_float(y, ey);
    add_m((unsigned __int128)((uint64_t)mx * my), ex + ey + sc, neg ^ (x < 0) ^ (y < 0));
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
    uint64_t dtop = (uint64_t)d[top];
    int msb = top * 32 + 63 - __clzll(dtop);  // bit index of the leading one
    // the 64 bits [msb-63, msb], plus a sticky flag for everything below
    uint64_t win = 0;
    for (int bit = msb; bit > msb - 64; bit--) {
      win <<= 1;
      if (bit >= 0) win |= ((uint64_t)d[bit >> 5] >> (bit & 31)) & 1ull;
    }
    bool sticky = false;
    for (int j = 0; j < NLIMB && !sticky; j++) {
      int lo_bit = j * 32, hi_bit = j * 32 + 31;
      if (hi_bit <= msb - 64) sticky = d[j] != 0;
      else if (lo_bit <= msb - 64) {
        int nb = msb - 64 - lo_bit + 1;
        uint64_t mask = nb >= 32 ? 0xFFFFFFFFull : ((1ull << nb) - 1);
        sticky = ((uint64_t)d[j] & mask) != 0;
      }
    }
    uint64_t mant = win >> 11;
    uint64_t rest = win & 0x7FFull;
    bool round = (rest >> 10) & 1;
    bool st = sticky || (rest & 0x3FF);
    if (round && (st || (mant & 1))) mant++;
    double r = ldexp((double)mant, msb - 52 + LIMB_LSB);
    return neg ? -r : r;
  }
};

// ---------------------------------------------------------------------------
// exact magnitudes as float32 pairs
// ---------------------------------------------------------------------------
// |d| is carried as (hi + lo) * 2^sc with hi = RN32(|d| 2^-sc), |lo| <= half a
// step of hi, sc in {0, 1} (sc = 1 only when |d| exceeds the float32 range).

__device__ __forceinline__ void two_sum_f(float x, float y, float& s, float& t) {
  s = __fadd_rn(x, y);
  float yv = __fsub_rn(s, x);
  float xv = __fsub_rn(s, yv);
  t = __fadd_rn(__fsub_rn(x, xv), __fsub_rn(y, yv));
}

// sign(x - y) for two exact pair magnitudes
__device__ __forceinline__ int cmp_mag(float h1, float l1, int s1, float h2, float l2, int s2) {
  if (s1 != s2) return s1 > s2 ? 1 : -1;  // scaled values exceed every unscaled float32
  if (h1 != h2) return h1 > h2 ? 1 : -1;
  return l1 > l2 ? 1 : (l1 < l2 ? -1 : 0);
}

// sign(a1/g1 - a2/g2), a = (hi + lo) 2^sc >= 0, g >= 0; g = 0 < a means +inf
__device__ int cmp_rel_exact(float h1, float l1, int s1, float g1, float h2, float l2, int s2, float g2) {
  int k1 = h1 == 0.0f ? 0 : (g1 == 0.0f ? 2 : 1);
  int k2 = h2 == 0.0f ? 0 : (g2 == 0.0f ? 2 : 1);
  if (k1 != k2) return k1 > k2 ? 1 : -1;
  if (k1 != 1) return 0;
  XAcc x;
  x.zero();
  x.add_prod_f(h1, g2, false, s1);
  x.add_prod_f(l1, g2, false, s1);
  x.add_prod_f(h2, g1, true, s2);
  x.add_prod_f(l2, g1, true, s2);
  x.normalize();
  return x.sign();
}

// sign(a1/g1 - a2/g2) for positive normal float32 values (a2 may be 0):
// compares the 48-bit products of the significands.
__device__ __forceinline__ int cmp_ratio_f(float a1, float g1, float a2, float g2) {
  if (a2 == 0.0f) return 1;
  uint32_t b1 = __float_as_uint(a1), c1 = __float_as_uint(g1), b2 = __float_as_uint(a2), c2 = __float_as_uint(g2);
  uint64_t P1 = (uint64_t)((b1 & 0x7FFFFFu) | 0x800000u) * ((c2 & 0x7FFFFFu) | 0x800000u);
  uint64_t P2 = (uint64_t)((b2 & 0x7FFFFFu) | 0x800000u) * ((c1 & 0x7FFFFFu) | 0x800000u);
  int x1 = (int)(b1 >> 23) + (int)(c2 >> 23), x2 = (int)(b2 >> 23) + (int)(c1 >> 23);
  if (x1 > x2 + 1) return 1;
  if (x2 > x1 + 1) return -1;
  if (x1 > x2) P1 <<= 1;
  else if (x2 > x1) P2 <<= 1;
  return P1 > P2 ? 1 : (P1 < P2 ? -1 : 0);
}

// float32 filter for a rel best: a value <= rel with a margin for the
// approximate per-lane ratio a * rcp(|g|)
__device__ __forceinline__ float rel_filter(float hi, int sc, float g) {
  if (g == 0.0f) return __int_as_float(0x7F800000);
  float q = __fdiv_rd(hi, g);
  if (sc) q = __fmul_rd(q, 2.0f);
  return __fmul_rd(q, 0.99999809265136719f);  // 1 - 2^-19
}

// ---------------------------------------------------------------------------
// shared memory
// ---------------------------------------------------------------------------
// Per-thread state touched only on the rare paths: the general-path counters
// and the exact maxima records.
struct Cold {
  float abs_hi, abs_lo;
  float rel_hi, rel_lo, rel_g;
  float rel_f;  // filter of the rel best
  uint32_t ulp;
  uint32_t n_gw, n_gm, n_ga, n_gf, n_nf, n_geq;
  int abs_sc, rel_sc;
  uint32_t pad;
  long long abs_idx, rel_idx, ulp_idx;
};

// Per-warp staging ring for the bulk copies: NSTAGE stages, each one warp
// tile of CHV 16-byte vectors of each tensor (two vectors per lane).
constexpr int NW = BLOCK / 32;
constexpr int NSTAGE = 3;
constexpr int CHV = 64;

struct __align__(128) Smem {
  uint4 ring_g[NW][NSTAGE][CHV];
  uint4 ring_c[NW][NSTAGE][CHV];
  unsigned long long bar[NW][NSTAGE];
  unsigned long long hist[HBINS];
  unsigned long long sacc[NSUM][NLIMB];
  unsigned long long cnt[8];
  Partial wbest[NW];
  int lb;
  uint32_t ovf[64];               // ULP bins NU+1..63 of window lanes (CTA-wide)
  Cold cold[BLOCK];
  uint32_t priv[NPB_MAX * HALF];  // per-thread 16-bit counters, two threads per word
  unsigned short qp[NW][CHV * 8]; // per-warp queue: tile positions of the unequal lanes
};

__device__ __forceinline__ void sacc_add(Smem& sm, int which, unsigned __int128 m, int e, bool neg) {
  for_digits(m, e, neg, [&](int j, int64_t v) { atomicAdd(&sm.sacc[which][j], (unsigned long long)v); });
}
__device__ __forceinline__ void sacc_add_f(Smem& sm, int which, float x, bool neg, int sc) {
  if (x == 0.0f) return;
  int e;
  uint32_t m = split_float(x, e);
  sacc_add(sm, which, m, e + sc, neg ^ (x < 0));
}
__device__ __forceinline__ void sacc_add_prod_f(Smem& sm, int which, float x, float y, int sc) {
  if (x == 0.0f || y == 0.0f) return;
  int ex, ey;
  uint32_t mx = split_float(x, ex), my = split_float(y, ey);
  sacc_add(sm, which, (unsigned __int128)((uint64_t)mx * my), ex + ey + sc, (x < 0) ^ (y < 0));
}

// ---------------------------------------------------------------------------
// per-thread hot state (registers)
// ---------------------------------------------------------------------------
struct Ctx {
  Cold* cold;         // this thread's rare-path record
  float rtol, atol;
  uint32_t lb_shift;  // Lb << MB
  uint32_t c0;        // 158 + Lexp: V = ((bits(|d|) << 8) | 2^31) >> (c0 - exponent(|d|))
  uint32_t col, inc;  // private histogram column and increment
};

struct Hot {
  uint32_t n_eq, n_win, n_within;
  uint64_t P, N, Q;
  float abs_f;         // best |d|: exact when abs_x, else a lower bound
  float rel_f;         // filter: <= best rel
  float rel_a, rel_g;  // best rel = rel_a / rel_g exactly when rel_x
  uint32_t ulp_f;
  bool abs_x, rel_x;
  int64_t first_fin, first_ulp;
};

__device__ __forceinline__ void hot_init(Hot& h) {
  h.n_eq = h.n_win = h.n_within = 0;
  h.P = h.N = h.Q = 0;
  h.abs_f = 0.0f;
  h.rel_f = 0.0f;
  h.rel_a = 0.0f;
  h.rel_g = 1.0f;
  h.ulp_f = 0;
  h.abs_x = h.rel_x = true;
  h.first_fin = h.first_ulp = -1;
}

__device__ __forceinline__ void cold_init(Cold& c) {
  c.abs_hi = c.abs_lo = 0.0f;
  c.rel_hi = c.rel_lo = 0.0f;
  c.rel_g = 1.0f;
  c.rel_f = 0.0f;
  c.ulp = 0;
  c.n_gw = c.n_gm = c.n_ga = c.n_gf = c.n_nf = c.n_geq = 0;
  c.abs_sc = c.rel_sc = 0;
  c.abs_idx = c.rel_idx = c.ulp_idx = -1;
}

// after the general path ran, refresh the hot copies from the cold records
__device__ __forceinline__ void hot_reload(Hot& h, const Cold& c) {
  h.abs_x = c.abs_lo == 0.0f && c.abs_sc == 0;
  h.abs_f = (c.abs_lo < 0.0f && c.abs_sc == 0) ? nextafterf(c.abs_hi, 0.0f) : c.abs_hi;
  // the integer ratio compare needs normal float32 operands
  h.rel_x = c.rel_lo == 0.0f && c.rel_sc == 0 &&
            (c.rel_idx < 0 || (c.rel_g >= 1.17549435e-38f && c.rel_hi >= 1.17549435e-38f));
  h.rel_a = c.rel_hi;
  h.rel_g = c.rel_g;
  h.rel_f = c.rel_f;
  h.ulp_f = c.ulp;
}

template <int DT>
__device__ __forceinline__ void note_first(Hot& h, uint32_t G, uint32_t C, int64_t idx) {
  using T = Tr<DT>;
  uint32_t ag = G & T::MAG, ac = C & T::MAG;
  if (h.first_fin < 0 && ag < T::INF && ac < T::INF) h.first_fin = idx;
  if (h.first_ulp < 0 && ag <= T::INF && ac <= T::INF) h.first_ulp = idx;
}

// Exact maxima update for a window lane; idx exceeds every index this thread
// has seen, so ties keep the current best.
__device__ __forceinline__ void window_update(Hot& h, Cold& cd, float a, float ag, uint32_t u, int64_t idx) {
  if (a > h.abs_f) {
    bool gt = h.abs_x || cmp_mag(a, 0.0f, 0, cd.abs_hi, cd.abs_lo, cd.abs_sc) > 0;
    if (gt) {
      cd.abs_hi = a;
      cd.abs_lo = 0.0f;
      cd.abs_sc = 0;
      cd.abs_idx = idx;
      h.abs_f = a;
      h.abs_x = true;
    }
  }
  if (u > h.ulp_f) {
    h.ulp_f = u;
    cd.ulp = u;
    cd.ulp_idx = idx;
  }
  float r = __fmul_rn(a, rcp_approx(ag));
  if (r > h.rel_f) {
    int c = h.rel_x ? cmp_ratio_f(a, ag, h.rel_a, h.rel_g)
                    : cmp_rel_exact(a, 0.0f, 0, ag, cd.rel_hi, cd.rel_lo, cd.rel_sc, cd.rel_g);
    if (c > 0) {
      cd.rel_hi = a;
      cd.rel_lo = 0.0f;
      cd.rel_sc = 0;
      cd.rel_g = ag;
      cd.rel_idx = idx;
      h.rel_a = a;
      h.rel_g = ag;
      h.rel_x = true;
      h.rel_f = rel_filter(a, 0, ag);
      cd.rel_f = h.rel_f;
    }
  }
}

// floor(log2(a / g)) for a = (hi + lo) 2^sc > 0 and g > 0 (float32 pair, any range)
__device__ int log2_ratio(float hi, float lo, int sc, float g) {
  float hs = hi, gs = g;
  if (hs < 1.17549435e-38f || gs < 1.17549435e-38f) {  // scale subnormals by 2^64
    if (hs >= 1.8446744e19f) return 200;              // ratio far above the clamp
    if (gs >= 1.8446744e19f) return -200;
    hs = __fmul_rn(hs, 1.8446744e19f);
    gs = __fmul_rn(gs, 1.8446744e19f);
  }
  uint32_t bh = __float_as_uint(hs), bg = __float_as_uint(gs);
  int k = ((int)(bh - bg)) >> 23;
  if (lo < 0.0f && (bh & 0x7FFFFFu) == (bg & 0x7FFFFFu)) k--;  // a just below 2^k g
  return k + sc;
}

// The general path: the definitions evaluated exactly, for any pair.
template <int DT>
__device__ __noinline__ void general_lane(Smem& sm, Cold& cd, uint32_t G, uint32_t C, int64_t idx, float rtol,
                                          float atol) {
  using T = Tr<DT>;
  uint32_t ag_m = G & T::MAG, ac_m = C & T::MAG;
  bool gnan = ag_m > T::INF, cnan = ac_m > T::INF, ginf = ag_m == T::INF, cinf = ac_m == T::INF;
  bool gs = (G & T::SIGN) != 0, cs = (C & T::SIGN) != 0;
  int64_t kg = gs ? -(int64_t)ag_m : (int64_t)ag_m, kc = cs ? -(int64_t)ac_m : (int64_t)ac_m;
  uint64_t u = (uint64_t)(kc > kg ? kc - kg : kg - kc);
  bool ulpdef = !gnan && !cnan;
  if (ulpdef && u > 0 && (u > cd.ulp || (u == cd.ulp && idx < cd.ulp_idx))) {
    cd.ulp = (uint32_t)u;
    cd.ulp_idx = idx;
  }
  if (gnan || cnan || ginf || cinf) {
    cd.n_nf++;
    bool equal = (gnan && cnan) || (ginf && cinf && gs == cs);
    if (equal) {
      cd.n_geq++;
      return;
    }
    cd.n_ga++;
    atomicAdd(&sm.hist[63], 1ull);
    atomicAdd(&sm.hist[64 + (ulpdef ? (u < 63 ? (int)u : 63) : 63)], 1ull);
    return;
  }
  float gf = to_f32<DT>(G), cf = to_f32<DT>(C);
  if (gf == cf) {  // +0 and -0
    cd.n_geq++;
    return;
  }
  float s, t;
  int sc = 0;
  two_sum_f(cf, -gf, s, t);
  if (!(fabsf(s) < __int_as_float(0x7F800000))) {  // |d| above the float32 range: halve exactly
    two_sum_f(__fmul_rn(cf, 0.5f), __fmul_rn(-gf, 0.5f), s, t);
    sc = 1;
  }
  float hi = fabsf(s), lo = s < 0.0f ? -t : t;
  float ag = fabsf(gf);
  // WITHIN_TOL: a <= atol + rtol |g|, decided in float32 when clear, exactly otherwise
  bool within;
  float thr = __fmaf_rn(rtol, ag, atol);
  if (sc == 0 && hi >= 1e-30f && thr >= 1e-30f && __fmul_rn(hi, 1.0000005f) < __fmul_rn(thr, 0.9999995f)) {
    within = true;
  } else if (sc == 0 && hi >= 1e-30f && __fmul_rn(hi, 0.9999995f) > __fmul_rn(thr, 1.0000005f)) {
    within = false;
  } else {
    XAcc x;
    x.zero();
    x.add_f(hi, false, sc);
    x.add_f(lo, false, sc);
    x.add_f(atol, true);
    x.add_prod_f(rtol, ag, true);
    x.normalize();
    within = x.sign() <= 0;
  }
  if (within) cd.n_gw++;
  else if (gf != 0.0f && cf != 0.0f && gs != cs) cd.n_gf++;
  else cd.n_gm++;
  // log2-relative bin and ULP bin
  int rb;
  if (ag == 0.0f) {
    rb = 63;
  } else {
    int k = log2_ratio(hi, lo, sc, ag) + 48;
    rb = k < 1 ? 1 : (k > 62 ? 62 : k);
  }
  atomicAdd(&sm.hist[rb], 1ull);
  atomicAdd(&sm.hist[64 + (u < 63 ? (int)u : 63)], 1ull);
  // maxima, full (value, index) order
  {
    int c = cd.abs_idx < 0 ? 1 : cmp_mag(hi, lo, sc, cd.abs_hi, cd.abs_lo, cd.abs_sc);
    if (c > 0 || (c == 0 && idx < cd.abs_idx)) {
      cd.abs_hi = hi;
      cd.abs_lo = lo;
      cd.abs_sc = sc;
      cd.abs_idx = idx;
    }
  }
  {
    bool maybe = cd.rel_idx < 0 || ag == 0.0f || sc ||
                 __fmul_rn(__fmul_rn(hi, rcp_approx(ag)), 1.00001f) >= cd.rel_f;
    if (maybe) {
      int c = cd.rel_idx < 0 ? 1 : cmp_rel_exact(hi, lo, sc, ag, cd.rel_hi, cd.rel_lo, cd.rel_sc, cd.rel_g);
      if (c > 0 || (c == 0 && idx < cd.rel_idx)) {
        cd.rel_hi = hi;
        cd.rel_lo = lo;
        cd.rel_sc = sc;
        cd.rel_g = ag;
        cd.rel_idx = idx;
        cd.rel_f = rel_filter(hi, sc, ag);
      }
    }
  }
  // exact sums: d = (s + t) 2^sc, |d| = (hi + lo) 2^sc, d^2 = (s^2 + 2st + t^2) 4^sc
  sacc_add_f(sm, 0, s, false, sc);
  sacc_add_f(sm, 0, t, false, sc);
  sacc_add_f(sm, 1, hi, false, sc);
  sacc_add_f(sm, 1, lo, false, sc);
  sacc_add_prod_f(sm, 2, s, s, 2 * sc);
  sacc_add_prod_f(sm, 2, s, t, 2 * sc + 1);
  sacc_add_prod_f(sm, 2, t, t, 2 * sc);
}

template <int DT>
__device__ __forceinline__ void window_cand(Hot& h, Cold& cd, uint32_t G, uint32_t C, int64_t idx) {
  float gf = to_f32<DT>(G), cf = to_f32<DT>(C);
  float a = fabsf(__fsub_rn(cf, gf)), ag = fabsf(gf);
  uint32_t u = (uint32_t)abs((int32_t)C - (int32_t)G);
  window_update(h, cd, a, ag, u, idx);
}

// bitmask of the lanes of a vector whose value is NaN or Inf
template <int DT>
__device__ __forceinline__ uint32_t nonfinite_mask(const uint4& v) {
  using T = Tr<DT>;
  if constexpr (T::BYTES == 2) {
    constexpr uint32_t ADD = (0x8000u - T::INF) * 0x10001u;  // sets bit 15 of a half iff mag >= INF
    uint32_t any = (((v.x & 0x7FFF7FFFu) + ADD) | ((v.y & 0x7FFF7FFFu) + ADD) | ((v.z & 0x7FFF7FFFu) + ADD) |
                    ((v.w & 0x7FFF7FFFu) + ADD)) & 0x80008000u;
    if (!any) return 0;
  }
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < T::VEC; j++) m |= ((lane_bits<DT>(v, j) & T::MAG) >= T::INF ? 1u : 0u) << j;
  return m;
}

// One unequal lane: the window fast path, or the general path.
template <int DT>
__device__ __forceinline__ void lane_proc(Hot& h, uint32_t G, uint32_t C, int64_t idx, const Ctx& cx, Smem& sm) {
  using T = Tr<DT>;
  const uint32_t ag = G & T::MAG, ac = C & T::MAG;
  const uint32_t u = (uint32_t)abs((int32_t)C - (int32_t)G);  // ULP distance for same-sign pairs
  uint32_t mg = ag, mc = ac;
  if constexpr (DT == PEAT_F16) {  // subnormal steps equal binade 1's
    mg = max(mg, 1u << T::MB);
    mc = max(mc, 1u << T::MB);
  }
  bool ok = ((G ^ C) & T::SIGN) == 0 && u < (1u << T::UB) && ag != 0u && mg >= cx.lb_shift && mc >= cx.lb_shift;
  const float gf = to_f32<DT>(G), cf = to_f32<DT>(C);
  const float s = __fsub_rn(cf, gf);
  const float a = fabsf(s), agf = fabsf(gf);
  const uint32_t ab = __float_as_uint(a);
  const uint32_t sh = cx.c0 - (ab >> 23);
  const float thr = __fmaf_rn(cx.rtol, agf, cx.atol);
  ok = ok && (sh - 8u) <= 23u && a != thr;  // 1 <= V < 2^24; tolerance ties go to the general path
  if (ok) {
    h.n_win++;
    h.n_within += a < thr ? 1u : 0u;
    const int k = (int)(ab - __float_as_uint(agf)) >> 23;  // floor(log2(|d| / |g|))
    uint32_t* uctr = u <= (uint32_t)NU ? &sm.priv[(u - 1) * HALF + cx.col] : &sm.ovf[u < 63u ? u : 63u];
    atomicAdd(uctr, u <= (uint32_t)NU ? cx.inc : 1u);
    atomicAdd(&sm.priv[(NU + k - Rows<DT>::KLO) * HALF + cx.col], cx.inc);
    const uint32_t V = ((ab << 8) | 0x80000000u) >> sh;  // |d| / 2^Lexp, exact
    if (s > 0.0f) h.P += V;
    else h.N += V;
    h.Q += (uint64_t)V * V;
    if ((a > h.abs_f) | (u > h.ulp_f) | (__fmul_rn(a, rcp_approx(agf)) > h.rel_f))
      window_update(h, *cx.cold, a, agf, u, idx);
  } else {
    Cold& cd = *cx.cold;
    general_lane<DT>(sm, cd, G, C, idx, cx.rtol, cx.atol);
    hot_reload(h, cd);
  }
}

// lanes of one vector whose golden value is NaN or Inf, as a bitmask
template <int DT>
__device__ __forceinline__ uint32_t nonfinite_lanes(const uint4& v) {
  using T = Tr<DT>;
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < T::VEC; j++) m |= ((lane_bits<DT>(v, j) & T::MAG) >= T::INF ? 1u : 0u) << j;
  return m;
}
// any NaN/Inf among the lanes of one vector (cheap test)
template <int DT>
__device__ __forceinline__ bool any_nonfinite(const uint4& v) {
  using T = Tr<DT>;
  if constexpr (T::BYTES == 2) {
    constexpr uint32_t ADD = (0x8000u - T::INF) * 0x10001u;  // sets bit 15 of a half iff its magnitude >= INF
    return ((((v.x & 0x7FFF7FFFu) + ADD) | ((v.y & 0x7FFF7FFFu) + ADD) | ((v.z & 0x7FFF7FFFu) + ADD) |
             ((v.w & 0x7FFF7FFFu) + ADD)) & 0x80008000u) != 0u;
  } else {
    uint32_t m = max(max(v.x & T::MAG, v.y & T::MAG), max(v.z & T::MAG, v.w & T::MAG));
    return m >= T::INF;
  }
}
// bitmask of the lanes whose bit patterns differ
template <int DT>
__device__ __forceinline__ uint32_t unequal_mask(const uint4& g, const uint4& c) {
  const uint32_t x[4] = {g.x ^ c.x, g.y ^ c.y, g.z ^ c.z, g.w ^ c.w};
  uint32_t m = 0;
  if constexpr (Tr<DT>::BYTES == 4) {
#pragma unroll
    for (int j = 0; j < 4; j++) m |= (x[j] != 0u ? 1u : 0u) << j;
  } else {
#pragma unroll
    for (int j = 0; j < 4; j++) m |= ((x[j] & 0xFFFFu) != 0u ? 1u : 0u) << (2 * j) | (x[j] > 0xFFFFu ? 2u : 0u) << (2 * j);
  }
  return m;
}

// Equal lanes of one vector: every bitwise-equal pair is EXACT; the ones
// holding NaN/Inf also count as non-finite pairs.
template <int DT>
__device__ __forceinline__ void count_equal(Hot& h, const uint4& g, uint32_t eqm, int64_t base, Cold& cd) {
  h.n_eq += __popc(eqm);
  if (eqm && any_nonfinite<DT>(g)) {
    const uint32_t nf = nonfinite_lanes<DT>(g) & eqm;
    cd.n_nf += __popc(nf);
  }
  (void)base;
}

// One warp tile of CHV vectors staged in shared memory: lane L owns vectors L
// and L + 32.  Equal lanes are counted in place; unequal lanes are queued (in
// element order) and processed 32 at a time, so every thread does useful work.
template <int DT>
__device__ __forceinline__ void do_tile(Hot& h, const uint4* gt, const uint4* ct, int nvalid, int64_t tile_base,
                                        const Ctx& cx, Smem& sm) {
  using T = Tr<DT>;
  constexpr int VEC = T::VEC;
  constexpr uint32_t FULL = (1u << VEC) - 1u;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool okA = lane < nvalid, okB = lane + 32 < nvalid;
  const uint4 z = make_uint4(0, 0, 0, 0);
  const uint4 gA = okA ? gt[lane] : z, cA = okA ? ct[lane] : z;
  const uint4 gB = okB ? gt[lane + 32] : z, cB = okB ? ct[lane + 32] : z;
  const int64_t baseA = tile_base + (int64_t)lane * VEC, baseB = baseA + 32 * VEC;
  if ((h.first_fin | h.first_ulp) < 0) {
    if (okA)
      for (int j = 0; j < VEC; j++) note_first<DT>(h, lane_bits<DT>(gA, j), lane_bits<DT>(cA, j), baseA + j);
    if (okB)
      for (int j = 0; j < VEC; j++) note_first<DT>(h, lane_bits<DT>(gB, j), lane_bits<DT>(cB, j), baseB + j);
  }
  const bool diff = ((gA.x ^ cA.x) | (gA.y ^ cA.y) | (gA.z ^ cA.z) | (gA.w ^ cA.w) | (gB.x ^ cB.x) | (gB.y ^ cB.y) |
                     (gB.z ^ cB.z) | (gB.w ^ cB.w)) != 0u;
  Cold& cd = *cx.cold;
  if (!__any_sync(0xFFFFFFFFu, diff)) {  // the whole warp tile is bitwise equal
    if (okA) count_equal<DT>(h, gA, FULL, baseA, cd);
    if (okB) count_equal<DT>(h, gB, FULL, baseB, cd);
    return;
  }
  const uint32_t nA = okA ? unequal_mask<DT>(gA, cA) : 0u, nB = okB ? unequal_mask<DT>(gB, cB) : 0u;
  if (okA) count_equal<DT>(h, gA, FULL & ~nA, baseA, cd);
  if (okB) count_equal<DT>(h, gB, FULL & ~nB, baseB, cd);
  // one scan of the packed counts gives the A-queue and B-queue offsets
  const uint32_t packed = __popc(nA) | (__popc(nB) << 16);
  uint32_t incl = packed;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  const uint32_t tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
  const uint32_t totA = tot & 0xFFFFu, total = totA + (tot >> 16);
  uint32_t posA = (incl & 0xFFFFu) - (packed & 0xFFFFu);
  uint32_t posB = totA + (incl >> 16) - (packed >> 16);
  unsigned short* q = sm.qp[warp];
#pragma unroll
  for (int j = 0; j < VEC; j++) {
    if ((nA >> j) & 1u) q[posA++] = (unsigned short)(lane * VEC + j);
    if ((nB >> j) & 1u) q[posB++] = (unsigned short)((lane + 32) * VEC + j);
  }
  __syncwarp();
  for (uint32_t e = lane; e < total; e += 32) {
    const uint32_t pos = q[e];
    uint32_t G, C;
    if constexpr (T::BYTES == 2) {
      G = reinterpret_cast<const unsigned short*>(gt)[pos];
      C = reinterpret_cast<const unsigned short*>(ct)[pos];
    } else {
      G = reinterpret_cast<const uint32_t*>(gt)[pos];
      C = reinterpret_cast<const uint32_t*>(ct)[pos];
    }
    lane_proc<DT>(h, G, C, tile_base + pos, cx, sm);
  }
  __syncwarp();
}

// one element outside the vector grid
template <int DT>
__device__ __forceinline__ void do_scalar(Hot& h, uint32_t G, uint32_t C, int64_t idx, const Ctx& cx, Smem& sm) {
  using T = Tr<DT>;
  if ((h.first_fin | h.first_ulp) < 0) note_first<DT>(h, G, C, idx);
  if (G == C) {
    h.n_eq++;
    if ((G & T::MAG) >= T::INF) cx.cold->n_nf++;
    return;
  }
  lane_proc<DT>(h, G, C, idx, cx, sm);
}

// ---------------------------------------------------------------------------
// CTA ranges: boundaries precomputed on the host
// ---------------------------------------------------------------------------
__device__ __forceinline__ int cta_of(int64_t i, const CompareParams& p) {
  int lo = 0, hi = p.nctas - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (p.bounds[mid] <= i) lo = mid;
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
// merging maxima records
// ---------------------------------------------------------------------------
__device__ __forceinline__ void part_none(Partial& r) {
  r.abs_hi = r.abs_lo = 0.0f;
  r.abs_sc = r.pad0 = 0;
  r.abs_idx = -1;
  r.rel_hi = r.rel_lo = 0.0f;
  r.rel_g = 1.0f;
  r.rel_sc = 0;
  r.rel_idx = -1;
  r.ulp = 0;
  r.ulp_idx = -1;
  r.first_fin = r.first_ulp = -1;
}

__device__ __forceinline__ int64_t min_idx(int64_t a, int64_t b) {
  if (a < 0) return b;
  if (b < 0) return a;
  return a < b ? a : b;
}

__device__ int cmp_rel_rec(float h1, float l1, int s1, float g1, float h2, float l2, int s2, float g2) {
  const float tiny = 1.17549435e-38f;
  if (l1 == 0.0f && l2 == 0.0f && s1 == 0 && s2 == 0 && h1 >= tiny && h2 >= tiny && g1 >= tiny && g2 >= tiny)
    return cmp_ratio_f(h1, g1, h2, g2);
  return cmp_rel_exact(h1, l1, s1, g1, h2, l2, s2, g2);
}

// x <- the better of x and y, field by field; ties to the lower index
__device__ void part_merge(Partial& x, const Partial& y) {
  if (y.abs_idx >= 0) {
    int c = x.abs_idx < 0 ? 1 : cmp_mag(y.abs_hi, y.abs_lo, y.abs_sc, x.abs_hi, x.abs_lo, x.abs_sc);
    if (c > 0 || (c == 0 && y.abs_idx < x.abs_idx)) {
      x.abs_hi = y.abs_hi;
      x.abs_lo = y.abs_lo;
      x.abs_sc = y.abs_sc;
      x.abs_idx = y.abs_idx;
    }
  }
  if (y.rel_idx >= 0) {
    int c = x.rel_idx < 0 ? 1 : cmp_rel_rec(y.rel_hi, y.rel_lo, y.rel_sc, y.rel_g, x.rel_hi, x.rel_lo, x.rel_sc, x.rel_g);
    if (c > 0 || (c == 0 && y.rel_idx < x.rel_idx)) {
      x.rel_hi = y.rel_hi;
      x.rel_lo = y.rel_lo;
      x.rel_sc = y.rel_sc;
      x.rel_g = y.rel_g;
      x.rel_idx = y.rel_idx;
    }
  }
  if (y.ulp_idx >= 0 && (x.ulp_idx < 0 || y.ulp > x.ulp || (y.ulp == x.ulp && y.ulp_idx < x.ulp_idx))) {
    x.ulp = y.ulp;
    x.ulp_idx = y.ulp_idx;
  }
  x.first_fin = min_idx(x.first_fin, y.first_fin);
  x.first_ulp = min_idx(x.first_ulp, y.first_ulp);
}

__device__ __forceinline__ int64_t shfl_i64(int64_t v, int o) {
  return (int64_t)((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)v, o) |
                   ((uint64_t)__shfl_down_sync(0xFFFFFFFFu, (uint32_t)((uint64_t)v >> 32), o) << 32));
}
__device__ __forceinline__ float shfl_f(float v, int o) { return __shfl_down_sync(0xFFFFFFFFu, v, o); }
__device__ __forceinline__ int shfl_int(int v, int o) { return __shfl_down_sync(0xFFFFFFFFu, v, o); }

// warp tournament; lane 0 ends with the warp's best
__device__ void part_warp_reduce(Partial& x) {
  const int lane = threadIdx.x & 31;
  for (int o = 16; o > 0; o >>= 1) {
    Partial y;
    y.abs_hi = shfl_f(x.abs_hi, o);
    y.abs_lo = shfl_f(x.abs_lo, o);
    y.abs_sc = shfl_int(x.abs_sc, o);
    y.abs_idx = shfl_i64(x.abs_idx, o);
    y.rel_hi = shfl_f(x.rel_hi, o);
    y.rel_lo = shfl_f(x.rel_lo, o);
    y.rel_g = shfl_f(x.rel_g, o);
    y.rel_sc = shfl_int(x.rel_sc, o);
    y.rel_idx = shfl_i64(x.rel_idx, o);
    y.ulp = (uint64_t)shfl_i64((int64_t)x.ulp, o);
    y.ulp_idx = shfl_i64(x.ulp_idx, o);
    y.first_fin = shfl_i64(x.first_fin, o);
    y.first_ulp = shfl_i64(x.first_ulp, o);
    if (lane + o < 32) part_merge(x, y);
  }
}

__device__ __forceinline__ uint64_t warp_sum64(uint64_t v) {
  for (int o = 16; o > 0; o >>= 1) v += (uint64_t)shfl_i64((int64_t)v, o);
  return v;
}

// Fold the per-thread 16-bit histograms and the window sums into the CTA
// totals.  All threads call it; it ends with the private counters zeroed.
template <int DT>
__device__ void fold_round(Hot& h, Smem& sm, int lexp) {
  constexpr int NPB = Rows<DT>::NPB;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // window sums: P, N < 2^40 and Q < 2^64 per thread per round; warp sums in 128 bits
  uint64_t P = warp_sum64(h.P), N = warp_sum64(h.N);
  uint64_t qlo = warp_sum64(h.Q & 0xFFFFFFFFull), qhi = warp_sum64(h.Q >> 32);
  if (lane == 0) {
    if (P >= N) sacc_add(sm, 0, (unsigned __int128)(P - N), lexp, false);
    else sacc_add(sm, 0, (unsigned __int128)(N - P), lexp, true);
    sacc_add(sm, 1, (unsigned __int128)P + N, lexp, false);
    sacc_add(sm, 2, (unsigned __int128)qlo + ((unsigned __int128)qhi << 32), 2 * lexp, false);
  }
  h.P = h.N = h.Q = 0;
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
      int bin = r < NU ? 64 + r + 1 : 48 + (r - NU) + Rows<DT>::KLO;
      sm.hist[bin] += sum;
    }
  }
  for (int b = threadIdx.x; b < 64; b += BLOCK) {  // ULP bins above NU
    if (b > NU && sm.ovf[b]) sm.hist[64 + b] += sm.ovf[b];
    sm.ovf[b] = 0;
  }
  __syncthreads();
}

// End of one segment piece: the integer totals go to the segment's
// accumulator (global atomics), the maxima to the CTA's partial slot.
template <int DT>
__device__ void finish_piece(Hot& h, Cold& cd, Smem& sm, int lexp, Partial* out, SegAcc* acc) {
  fold_round<DT>(h, sm, lexp);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t c[8] = {h.n_eq + cd.n_geq, h.n_win, h.n_within, cd.n_nf, cd.n_gw, cd.n_gm, cd.n_ga, cd.n_gf};
#pragma unroll
  for (int k = 0; k < 8; k++) {
    uint32_t v = __reduce_add_sync(0xFFFFFFFFu, c[k]);
    if (lane == 0 && v) atomicAdd(&sm.cnt[k], (unsigned long long)v);
  }
  Partial x;
  x.abs_hi = cd.abs_hi;
  x.abs_lo = cd.abs_lo;
  x.abs_sc = cd.abs_sc;
  x.pad0 = 0;
  x.abs_idx = cd.abs_idx;
  x.rel_hi = cd.rel_hi;
  x.rel_lo = cd.rel_lo;
  x.rel_g = cd.rel_g;
  x.rel_sc = cd.rel_sc;
  x.rel_idx = cd.rel_idx;
  x.ulp = cd.ulp;
  x.ulp_idx = cd.ulp_idx;
  x.first_fin = h.first_fin;
  x.first_ulp = h.first_ulp;
  part_warp_reduce(x);
  if (lane == 0) sm.wbest[warp] = x;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < BLOCK / 32; w++) part_merge(x, sm.wbest[w]);
    *out = x;
  }
  for (int b = threadIdx.x; b < HBINS; b += BLOCK)
    if (sm.hist[b]) atomicAdd(&acc->hist[b], sm.hist[b]);
  if (threadIdx.x < 8 && sm.cnt[threadIdx.x]) atomicAdd(&acc->cnt[threadIdx.x], sm.cnt[threadIdx.x]);
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) {
    unsigned long long v = (&sm.sacc[0][0])[j];
    if (v) atomicAdd(reinterpret_cast<unsigned long long*>(&acc->limbs[0][0]) + j, v);
  }
  __syncthreads();
  // reset the CTA totals for the next piece
  for (int b = threadIdx.x; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  if (threadIdx.x < 8) sm.cnt[threadIdx.x] = 0;
  hot_init(h);
  cold_init(cd);
  __syncthreads();
}

// ---------------------------------------------------------------------------
// stage 1
// ---------------------------------------------------------------------------
template <int DT>
__global__ void __launch_bounds__(BLOCK, 2) compare_stage1(CompareParams p) {
  using T = Tr<DT>;
  constexpr int VEC = T::VEC;
  // lanes per thread per round stay below 2^16 (16-bit private counters): each
  // warp tile gives a thread at most 2 VEC lanes
  constexpr int64_t ROUND_CHUNKS = (int64_t)NW * (65535 / (2 * VEC));
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int b = tid; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = tid; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  for (int j = tid; j < Rows<DT>::NPB * HALF; j += BLOCK) sm.priv[j] = 0;
  if (tid < 8) sm.cnt[tid] = 0;
  if (tid < 64) sm.ovf[tid] = 0;
  if (lane == 0) {
    for (int st = 0; st < NSTAGE; st++) mbar_init(&sm.bar[warp][st], 1);
    mbar_init_fence();
  }
  Ctx cx;
  cx.cold = &sm.cold[tid];
  cold_init(*cx.cold);
  const int64_t lo = p.bounds[blockIdx.x], hi = p.bounds[blockIdx.x + 1];
  Hot h;
  hot_init(h);
  cx.rtol = p.rtol;
  cx.atol = p.atol;
  cx.col = tid & (HALF - 1);
  cx.inc = tid < HALF ? 1u : 65536u;
  __syncthreads();
  if (lo >= hi) return;
  uint32_t seq = 0;      // this warp's bulk-copy stage uses so far (stage = seq % NSTAGE)
  bool failed = false;   // a pipeline wait expired: skip the data, keep the barriers
  int64_t s = seg_of(lo, p.offsets, p.nseg);
  int64_t pb = lo;
  const char* gbase = reinterpret_cast<const char*>(p.g);
  const char* cbase = reinterpret_cast<const char*>(p.c);
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
    const int64_t nchunk = (nvec + CHV - 1) / CHV;
    // start this warp's copies (chunk k = warp + NW * i) before anything else
    auto issue = [&](uint32_t sq, int64_t k) {
      const int st = (int)(sq % NSTAGE);
      const int64_t v0 = k * CHV;
      const uint32_t bytes = (uint32_t)(min((int64_t)CHV, nvec - v0) * 16);
      const int64_t off = (vb + v0 * VEC) * T::BYTES;
      fence_proxy_async();
      mbar_expect_tx(&sm.bar[warp][st], 2 * bytes);
      bulk_load(&sm.ring_g[warp][st][0], gbase + off, bytes, &sm.bar[warp][st]);
      bulk_load(&sm.ring_c[warp][st][0], cbase + off, bytes, &sm.bar[warp][st]);
    };
    const int64_t my_chunks = nchunk > warp ? (nchunk - warp + NW - 1) / NW : 0;
    if (lane == 0 && !failed)
      for (int64_t i = 0; i < NSTAGE && i < my_chunks; i++) issue(seq + (uint32_t)i, warp + NW * i);
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
    // V = |d| / 2^Lexp < 2^24 for u < 2^UB and golden binades up to 2 above the largest seen
    int lb = sm.lb + T::UB - 22;
    lb = lb < T::LBMIN ? T::LBMIN : (lb > T::LBMAX ? T::LBMAX : lb);
    const int lexp = lb - T::BIAS - T::MB;  // weight of V's unit
    cx.lb_shift = (uint32_t)lb << T::MB;
    cx.c0 = (uint32_t)(158 + lexp);
    // scalar head: fewer than VEC elements, or the whole piece in scalar mode
    // (then in rounds of at most 65535 elements per thread)
    {
      const int64_t h_end = vb < pe ? vb : pe;
      constexpr int64_t ROUND_ELEMS = (int64_t)BLOCK * 65535;
      for (int64_t r0 = pb; r0 < h_end; r0 += ROUND_ELEMS) {
        const int64_t r1 = min(h_end, r0 + ROUND_ELEMS);
        for (int64_t i = r0 + tid; i < r1; i += BLOCK)
          do_scalar<DT>(h, load_scalar<DT>(p.g, i), load_scalar<DT>(p.c, i), i, cx, sm);
        if (r1 < h_end) fold_round<DT>(h, sm, lexp);
      }
    }
    // vector body: warp w takes chunks w, w + NW, ... of CHV vectors from its
    // staging ring; NSTAGE chunks are in flight ahead of the one processed
    int64_t i = 0;  // this warp's chunk counter within the piece
    int64_t fail_i = -1;
    uint32_t fail_seq = 0;
    for (int64_t r0 = 0; r0 < nchunk; r0 += ROUND_CHUNKS) {
      const int64_t r1 = min(nchunk, r0 + ROUND_CHUNKS);
      for (int64_t k = warp + NW * i; k < r1; k = warp + NW * (++i)) {
        const int st = (int)(seq % NSTAGE);
        const uint32_t parity = (seq / NSTAGE) & 1u;
        if (!failed && !mbar_wait(&sm.bar[warp][st], parity, p.wait_limit)) {
          failed = true;  // chunks fail_i .. fail_i + NSTAGE - 1 may still be in flight
          fail_i = i;
          fail_seq = seq;
          if (lane == 0) atomicOr(p.status, 1u);
        }
        if (!failed) {
          const int64_t v0 = k * CHV;
          const int nvalid = (int)min((int64_t)CHV, nvec - v0);
          do_tile<DT>(h, sm.ring_g[warp][st], sm.ring_c[warp][st], nvalid, vb + v0 * VEC, cx, sm);
          if (lane == 0 && i + NSTAGE < my_chunks) issue(seq + NSTAGE, warp + NW * (i + NSTAGE));
        }
        seq++;
      }
      if (r1 < nchunk) fold_round<DT>(h, sm, lexp);
    }
    if (fail_i >= 0) {
      // copies this warp issued but never consumed: wait for them before the
      // staging memory is reused or the CTA exits
      for (int64_t j = fail_i; j < my_chunks && j < fail_i + NSTAGE; j++) {
        const uint32_t sq = fail_seq + (uint32_t)(j - fail_i);
        mbar_wait(&sm.bar[warp][sq % NSTAGE], (sq / NSTAGE) & 1u, DRAIN_LIMIT);
      }
    }
    // scalar tail (fewer than VEC elements), after the body: lanes stay in index order
    if (vb < ve && ve < pe)
      for (int64_t e = ve + tid; e < pe; e += BLOCK)
        do_scalar<DT>(h, load_scalar<DT>(p.g, e), load_scalar<DT>(p.c, e), e, cx, sm);
    finish_piece<DT>(h, *cx.cold, sm, lexp, p.partials + s + blockIdx.x, p.acc + s);
    pb = pe;
  }
}

// ---------------------------------------------------------------------------
// stage 2: one CTA per segment: merge the maxima of the segment's pieces,
// round the exact sums once, write the outputs, clear the accumulator
// ---------------------------------------------------------------------------
// RN64 of the quotient (hi + lo) 2^sc / g > 0: the candidate with the smallest
// exact residual, ties to the even significand
__device__ double rel_value(float hi, float lo, int sc, float g) {
  if (hi == 0.0f) return 0.0;
  if (g == 0.0f) return __longlong_as_double(0x7FF0000000000000ll);
  double num = __dadd_rn((double)hi, (double)lo) * (sc ? 2.0 : 1.0);
  double q0 = __ddiv_rn(num, (double)g);  // within a few units of the exact quotient
  double q = q0;
  for (int i = 0; i < 3; i++) q = nextafter(q, 0.0);
  double best = q;
  XAcc bres;
  bool have = false;
  for (int step = 0; step < 7; step++, q = nextafter(q, __longlong_as_double(0x7FF0000000000000ll))) {
    XAcc r;
    r.zero();
    r.add_f(hi, false, sc);
    r.add_f(lo, false, sc);
    r.add_prod(q, (double)g, true);
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

__global__ void __launch_bounds__(BLOCK) compare_stage2(CompareParams p) {
  const int64_t s = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t s0 = p.offsets[s], s1 = p.offsets[s + 1];
  SegAcc* acc = p.acc + s;
  __shared__ unsigned long long cnt[8];
  __shared__ long long limbs[NSUM][NLIMB];
  __shared__ double sums[NSUM];
  __shared__ Partial wbest[BLOCK / 32];
  // integer totals, then clear them for the next call
  unsigned long long hv = 0;
  if (tid < HBINS) {
    hv = acc->hist[tid];
    acc->hist[tid] = 0;
  }
  if (tid >= HBINS && tid < HBINS + 8) {
    cnt[tid - HBINS] = acc->cnt[tid - HBINS];
    acc->cnt[tid - HBINS] = 0;
  }
  if (tid >= 160 && tid < 160 + NSUM * NLIMB) {
    int j = tid - 160;
    (&limbs[0][0])[j] = (&acc->limbs[0][0])[j];
    (&acc->limbs[0][0])[j] = 0;
  }
  // maxima over the segment's pieces, in CTA order
  Partial x;
  part_none(x);
  if (s1 > s0) {
    const int b0 = cta_of(s0, p), b1 = cta_of(s1 - 1, p);
    for (int b = b0 + tid; b <= b1; b += BLOCK)
      if (p.bounds[b] < p.bounds[b + 1]) part_merge(x, p.partials[s + b]);
  }
  part_warp_reduce(x);
  if (lane == 0) wbest[warp] = x;
  __syncthreads();
  if (tid < NSUM) {
    XAcc a;
    for (int j = 0; j < NLIMB; j++) a.d[j] = limbs[tid][j];
    sums[tid] = a.to_double();
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < BLOCK / 32; w++) part_merge(x, wbest[w]);
    peat_stats_t r;
    const uint64_t n = (uint64_t)(s1 - s0);
    r.n = n;
    r.count[PEAT_EXACT] = cnt[0];
    r.count[PEAT_WITHIN_TOL] = cnt[2] + cnt[4];
    r.count[PEAT_MISMATCH] = (cnt[1] - cnt[2]) + cnt[5];
    r.count[PEAT_NAN_INF_ASYM] = cnt[6];
    r.count[PEAT_SIGN_FLIP] = cnt[7];
    r.n_finite = n - cnt[3];
    if (x.abs_idx >= 0) {
      r.max_abs = __dadd_rn((double)x.abs_hi, (double)x.abs_lo) * (x.abs_sc ? 2.0 : 1.0);
      r.argmax_abs = x.abs_idx - s0;
    } else {
      r.max_abs = 0.0;
      r.argmax_abs = x.first_fin >= 0 ? x.first_fin - s0 : -1;
    }
    if (x.rel_idx >= 0) {
      r.max_rel = rel_value(x.rel_hi, x.rel_lo, x.rel_sc, x.rel_g);
      r.argmax_rel = x.rel_idx - s0;
    } else {
      r.max_rel = 0.0;
      r.argmax_rel = x.first_fin >= 0 ? x.first_fin - s0 : -1;
    }
    if (x.ulp_idx >= 0) {
      r.max_ulp = x.ulp;
      r.argmax_ulp = x.ulp_idx - s0;
    } else {
      r.max_ulp = 0;
      r.argmax_ulp = x.first_ulp >= 0 ? x.first_ulp - s0 : -1;
    }
    r.sum_signed = sums[0];
    r.sum_abs = sums[1];
    r.sum_sq = sums[2];
    r.rtol_eff = p.rtol;
    r.atol_eff = p.atol;
    p.stats[s] = r;
  }
  if (p.hist && tid < HBINS) p.hist[s * HBINS + tid] = hv + ((tid == 0 || tid == 64) ? cnt[0] : 0ull);
}

template <int DT>
cudaError_t launch_t(const CompareParams& p, cudaStream_t st) {
  compare_stage1<DT><<<p.nctas, BLOCK, sizeof(Smem), st>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (p.nseg > 0) compare_stage2<<<(unsigned)p.nseg, BLOCK, 0, st>>>(p);
  return cudaGetLastError();
}

template <int DT>
int64_t bound_t(int64_t b, int nctas, int64_t n, int64_t p0) {
  if (b <= 0) return 0;
  if (b >= nctas) return n;
  constexpr int VEC = Tr<DT>::VEC;
  if (p0 < 0 || p0 >= n) return (n / nctas) * b + (n % nctas) * b / nctas;
  int64_t nv = (n - p0) / VEC;
  int64_t lo = p0 + ((nv / nctas) * b + (nv % nctas) * b / nctas) * VEC;
  return lo < n ? lo : n;
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

int64_t compare_cta_bound(int dtype, int64_t b, int nctas, int64_t n, int64_t p0) {
  switch (dtype) {
    case PEAT_F32: return bound_t<PEAT_F32>(b, nctas, n, p0);
    case PEAT_F16: return bound_t<PEAT_F16>(b, nctas, n, p0);
    default: return bound_t<PEAT_BF16>(b, nctas, n, p0);
  }
}

// once per device, before the first launch
cudaError_t compare_prepare() {
  cudaError_t e = cudaFuncSetAttribute(compare_stage1<PEAT_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sizeof(Smem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(compare_stage1<PEAT_F16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(Smem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(compare_stage1<PEAT_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)sizeof(Smem));
  return e;
}

int compare_ctas_per_sm() { return 2; }
size_t compare_partial_bytes() { return sizeof(Partial); }
size_t compare_segacc_bytes() { return sizeof(SegAcc); }
size_t compare_cold_bytes() { return sizeof(Cold) * BLOCK; }

}  // namespace peat
