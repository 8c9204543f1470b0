// The error signature (Section IV-B-3, with the classes, ULP distances and
// histograms of the compare) for binary64 operands: the FP32-FP64 pairs of
// Fig. 5 once the float32 side is widened (exactly) to binary64.
//
// d = c - g is an exact double-double (hi, lo) from Fast2Sum on the operands
// ordered by magnitude, held halved with a scale of one when the difference
// overflows binary64 (both operands are then large, so halving is exact).  Decisions that rounding could
// flip (the tolerance, the relative maximum) take a binary64 or float32 test
// with a margin first and otherwise the sign of an exact sum of integer
// terms; the relative bin comes from exponents and significands exactly; the
// three sums are added as 32-bit digits to a shared-memory superaccumulator
// per work item, merged per segment and rounded once.
#include <cstdint>

#include "exact64.cuh"
#include "meanvar.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

constexpr int TB = 256;
using namespace x64;

// significand in [1, 2) as 52 fraction bits, and exponent, of a finite nonzero double
__device__ __forceinline__ void norm_d(double x, uint64_t& f, int& e) {
  uint64_t m;
  int ex;
  split_d(x, m, ex);
  const int lz = __clzll((long long)m) - 11;  // shift the leading one to bit 52
  f = (m << lz) & 0xFFFFFFFFFFFFFull;
  e = ex + 52 - lz;
}

// floor(log2(a / ag)) for a > 0, ag > 0, exactly
__device__ __forceinline__ int rel_log2_floor64(const Mag& a, double ag) {
  uint64_t fa, fg;
  int ea, eg;
  norm_d(a.hi, fa, ea);
  norm_d(ag, fg, eg);
  const int k0 = ea + a.sc - eg;
  if (fa != fg) return fa > fg ? k0 : k0 - 1;
  return neg64(a.lo) ? k0 - 1 : k0;  // hi = ag 2^k0 exactly: lo decides
}

// relative error records: a / g with kind 0 (a = 0), 1 (finite), 2 (g = 0 < a)
struct Rel {
  Mag a;
  double g;
  int kind;
  int le;    // log2 of the ratio, approximately (kind 1): le + lf, le exact,
  float lf;  // lf = log2 of the significands' ratio within 2^-20
};

__device__ __forceinline__ void approx_log2(const Mag& a, double g, int& le, float& lf) {
  uint64_t fa, fg;
  int ea, eg;
  norm_d(a.hi, fa, ea);
  norm_d(g, fg, eg);
  const float ra = __uint_as_float(0x3F800000u | (uint32_t)(fa >> 29));
  const float rg = __uint_as_float(0x3F800000u | (uint32_t)(fg >> 29));
  le = ea + a.sc - eg;
  lf = __log2f(__fdividef(ra, rg));
}

// log2(x) - log2(y) of two finite ratios, within 2^-18 (clamped far from zero)
__device__ __forceinline__ float lg_diff(int xe, float xf, int ye, float yf) {
  const int de = xe - ye;
  if (de > 4) return 8.0f;
  if (de < -4) return -8.0f;
  return (float)de + (xf - yf);
}

// x > y exactly
__device__ bool rel_gt(const Rel& x, const Rel& y) {
  if (x.kind != y.kind) return x.kind > y.kind;
  if (x.kind != 1) return false;
  XTerm t[4] = {prod_term(x.a.hi, y.g, x.a.sc, false), prod_term(fabs(x.a.lo), y.g, x.a.sc, x.a.lo < 0.0),
                prod_term(y.a.hi, x.g, y.a.sc, true), prod_term(fabs(y.a.lo), x.g, y.a.sc, y.a.lo >= 0.0)};
  return xsign(t, 4) > 0;
}

// ---------------------------------------------------------------------------
// the per-item superaccumulator: 32-bit digits in signed 64-bit limbs

constexpr int SLSB = XLSB, SL = XL;
static_assert(SL == P64_LIMBS, "record limbs");

__device__ __forceinline__ void sacc_add(long long* acc, u128 m, int e, bool neg) {
  if (m == 0) return;
  const int p = e - SLSB;
  const int limb = p >> 5, sh = p & 31;
  const u128 lo = m << sh;
  const unsigned long long hi = sh ? (unsigned long long)(m >> (128 - sh)) : 0ull;
#pragma unroll
  for (int q = 0; q < 5; q++) {
    const unsigned long long dig = q < 4 ? (unsigned long long)(lo >> (32 * q)) & 0xFFFFFFFFull : hi & 0xFFFFFFFFull;
    if (dig) atomicAdd(reinterpret_cast<unsigned long long*>(acc + limb + q),
                       neg ? (unsigned long long)(-(long long)dig) : dig);
  }
}

// Per-thread windows in front of the superaccumulator: a term whose exponent
// lies within a fixed distance of the thread's first one is added to a
// register integer (signed 128 bits for sum d and sum |d|, 53-bit terms
// shifted by at most 56; unsigned 192 bits for sum d^2, 106-bit terms shifted
// by at most 70; at most 2^14 terms per thread and item, so neither
// overflows), any other term goes to the shared digits.  Flushed at the end
// of each item.
using i128 = __int128;

__device__ __forceinline__ void win_add(i128& acc, int& base, uint64_t m, int e, bool neg, long long* S) {
  if (m == 0) return;
  if (base == INT32_MIN) base = e - 28;
  const int sh = e - base;
  if (sh >= 0 && sh <= 56) {
    const i128 v = (i128)((u128)m << sh);
    acc += neg ? -v : v;
  } else {
    sacc_add(S, (u128)m, e, neg);
  }
}
__device__ __forceinline__ void win_flush(i128 acc, int base, long long* S) {
  if (acc == 0) return;
  const bool neg = acc < 0;
  sacc_add(S, neg ? (u128)(-acc) : (u128)acc, base, neg);
}

struct W192 {
  unsigned long long w0, w1, w2;
  int base;
};
__device__ __forceinline__ void win3_add(W192& a, u128 m, int e, long long* S) {
  if (m == 0) return;
  if (a.base == INT32_MIN) a.base = e - 35;
  const int sh = e - a.base;
  if (sh < 0 || sh > 70) {
    sacc_add(S, m, e, false);
    return;
  }
  const unsigned long long m0 = (unsigned long long)m, m1 = (unsigned long long)(m >> 64);
  unsigned long long v0, v1, v2;
  if (sh == 0) {
    v0 = m0, v1 = m1, v2 = 0;
  } else if (sh < 64) {
    v0 = m0 << sh, v1 = (m1 << sh) | (m0 >> (64 - sh)), v2 = m1 >> (64 - sh);
  } else {
    const int t = sh - 64;
    v0 = 0, v1 = m0 << t, v2 = (m1 << t) | (t ? m0 >> (64 - t) : 0ull);
  }
  a.w0 += v0;
  const unsigned long long c0 = a.w0 < v0 ? 1ull : 0ull;
  const unsigned long long s1 = a.w1 + v1;
  const unsigned long long c1 = (s1 < v1 ? 1ull : 0ull);
  a.w1 = s1 + c0;
  a.w2 += v2 + c1 + (a.w1 < c0 ? 1ull : 0ull);
}
__device__ __forceinline__ void win3_flush(const W192& a, long long* S) {
  // as two parts of at most 96 + 96 bits
  const u128 lo = ((u128)(a.w1 & 0xFFFFFFFFull) << 64) | a.w0;
  const u128 hi = ((u128)a.w2 << 32) | (a.w1 >> 32);
  if (lo) sacc_add(S, lo, a.base, false);
  if (hi) sacc_add(S, hi, a.base + 96, false);
}

// ---------------------------------------------------------------------------
// per-thread totals within one work item (offsets: position in the item + 1, 0 = none)

struct Acc64 {
  uint32_t cnt[PEAT_NCLASS], nfin;
  i128 sd, sa;   // windows of sum d and sum |d|
  int bd, ba;
  W192 sq;       // window of sum d^2
  Mag ma;
  uint32_t ia;
  Rel mr;
  uint32_t ir;
  unsigned long long mu;
  uint32_t iu;
};

__device__ __forceinline__ void acc64_init(Acc64& t) {
#pragma unroll
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] = 0;
  t.nfin = 0;
  t.sd = t.sa = 0;
  t.bd = t.ba = INT32_MIN;
  t.sq = W192{0ull, 0ull, 0ull, INT32_MIN};
  t.ma = Mag{0.0, 0.0, 0};
  t.ia = 0;
  t.mr = Rel{Mag{0.0, 0.0, 0}, 1.0, 0, 0, 0.0f};
  t.ir = 0;
  t.mu = 0;
  t.iu = 0;
}

__device__ __forceinline__ void hist_add(unsigned* H, int bin) {
  const unsigned grp = __match_any_sync(0xFFFFFFFFu, bin);
  if (bin >= 0 && (int)(threadIdx.x & 31) == __ffs(grp) - 1) atomicAdd(H + bin, (unsigned)__popc(grp));
}

// one pair slot of the warp (every lane calls it; ok: this lane holds the pair at item offset off)
__device__ __forceinline__ void pair64(const Cmp64Params& p, Acc64& t, unsigned* H, long long* S, uint64_t G,
                                       uint64_t C, bool ok, uint32_t off) {
  int relbin = -1, ulpbin = -1, cls = -1;
  if (ok) {
    const uint64_t mg = G & 0x7FFFFFFFFFFFFFFFull, mc = C & 0x7FFFFFFFFFFFFFFFull;
    const bool sg = (G >> 63) != 0, sc = (C >> 63) != 0;
    const uint64_t INF = 0x7FF0000000000000ull;
    const bool gnan = mg > INF, cnan = mc > INF, gfin = mg < INF, cfin = mc < INF;
    const long long kg = sg ? -(long long)mg : (long long)mg, kc = sc ? -(long long)mc : (long long)mc;
    const unsigned long long u = kc >= kg ? (unsigned long long)kc - (unsigned long long)kg
                                          : (unsigned long long)kg - (unsigned long long)kc;
    if (!gfin || !cfin) {
      const bool eq = (gnan && cnan) || (mg == INF && mc == INF && sg == sc);
      cls = eq ? PEAT_EXACT : PEAT_NAN_INF_ASYM;
      relbin = eq ? 0 : 63;
    } else {
      const double gd = from_bits64(G), cd = from_bits64(C);
      bool dneg;
      const Mag a = diff64(gd, cd, dneg);
      const double ag = from_bits64(mg);  // |g|
      const bool azero = bits64(a.hi) == 0;
      t.nfin++;
      // sums: d = +-(hi + lo) 2^sc, |d|, d^2 = (hi^2 + 2 hi lo + lo^2) 4^sc
      {
        uint64_t mh, ml;
        int eh, el;
        split_d(a.hi, mh, eh);
        split_d(a.lo, ml, el);  // split_d takes the magnitude
        const bool lneg = (bits64(a.lo) >> 63) != 0;
        win_add(t.sd, t.bd, mh, eh + a.sc, dneg, S);
        win_add(t.sa, t.ba, mh, eh + a.sc, false, S + SL);
        win3_add(t.sq, (u128)mh * mh, 2 * (eh + a.sc), S + 2 * SL);
        if (ml) {
          win_add(t.sd, t.bd, ml, el + a.sc, dneg != lneg, S);
          win_add(t.sa, t.ba, ml, el + a.sc, lneg, S + SL);
          if (lneg) sacc_add(S + 2 * SL, (u128)mh * ml, eh + el + 2 * a.sc + 1, true);  // rare: straight to digits
          else win3_add(t.sq, (u128)mh * ml, eh + el + 2 * a.sc + 1, S + 2 * SL);
          win3_add(t.sq, (u128)ml * ml, 2 * (el + a.sc), S + 2 * SL);
        }
      }
      if (t.ia == 0 || mag_gt(a, t.ma)) t.ma = a, t.ia = off + 1;
      // relative maximum: an approximate log2 rules out all but the candidates
      Rel r;
      r.a = a;
      r.g = ag;
      r.kind = azero ? 0 : (mg == 0 ? 2 : 1);
      r.le = 0;
      r.lf = 0.0f;
      if (r.kind == 1) approx_log2(a, ag, r.le, r.lf);
      const bool maybe = t.ir == 0 || r.kind > t.mr.kind ||
                         (r.kind == 1 && t.mr.kind == 1 && lg_diff(r.le, r.lf, t.mr.le, t.mr.lf) >= -0x1p-16f);
      if (maybe && (t.ir == 0 || rel_gt(r, t.mr))) t.mr = r, t.ir = off + 1;
      if (azero) {
        cls = PEAT_EXACT;
        relbin = 0;
      } else {
        if (within64(a, ag, p.rtol, p.atol)) cls = PEAT_WITHIN_TOL;
        else if (mg != 0 && mc != 0 && sg != sc) cls = PEAT_SIGN_FLIP;
        else cls = PEAT_MISMATCH;
        if (mg == 0) {
          relbin = 63;
        } else {
          const int k = rel_log2_floor64(a, ag) + 48;
          relbin = k < 1 ? 1 : (k > 62 ? 62 : k);
        }
      }
    }
    if (gnan || cnan) {
      ulpbin = (gnan && cnan) ? 0 : 63;
    } else {
      ulpbin = (int)(u < 63 ? u : 63);
      if (t.iu == 0 || u > t.mu) t.mu = u, t.iu = off + 1;
    }
  }
#pragma unroll
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] += cls == k;
  hist_add(H, relbin);
  hist_add(H, ulpbin < 0 ? -1 : 64 + ulpbin);
}

// x better than y: larger, or equal at a lower index (-1: absent, worst)
__device__ __forceinline__ bool better_mag(const Mag& x, long long ix, const Mag& y, long long iy) {
  if (ix < 0) return false;
  if (iy < 0) return true;
  return mag_gt(x, y) || (!mag_gt(y, x) && ix < iy);
}
__device__ __forceinline__ bool better_rel(const Rel& x, long long ix, const Rel& y, long long iy) {
  if (ix < 0) return false;
  if (iy < 0) return true;
  if (x.kind == 1 && y.kind == 1) {  // far apart: the approximations decide
    const float dl = lg_diff(x.le, x.lf, y.le, y.lf);
    if (fabsf(dl) > 0x1p-16f) return dl > 0.0f;
  }
  return rel_gt(x, y) || (!rel_gt(y, x) && ix < iy);
}
__device__ __forceinline__ bool better_u(unsigned long long x, long long ix, unsigned long long y, long long iy) {
  if (ix < 0) return false;
  if (iy < 0) return true;
  return x > y || (x == y && ix < iy);
}

// merge record o into r (both within one segment)
__device__ void rec_merge(Part64Rec& r, const Part64Rec& o) {
  for (int k = 0; k < PEAT_NCLASS; k++) r.cnt[k] += o.cnt[k];
  r.nfin += o.nfin;
  const Mag ra{r.ahi, r.alo, r.asc}, oa{o.ahi, o.alo, o.asc};
  if (better_mag(oa, o.ia, ra, r.ia)) r.ahi = o.ahi, r.alo = o.alo, r.asc = o.asc, r.ia = o.ia;
  const Rel rr{Mag{r.rhi, r.rlo, r.rsc}, r.rg, r.rkind, r.rle, r.rlf};
  const Rel orr{Mag{o.rhi, o.rlo, o.rsc}, o.rg, o.rkind, o.rle, o.rlf};
  if (better_rel(orr, o.ir, rr, r.ir))
    r.rhi = o.rhi, r.rlo = o.rlo, r.rsc = o.rsc, r.rg = o.rg, r.rkind = o.rkind, r.rle = o.rle, r.rlf = o.rlf,
    r.ir = o.ir;
  if (better_u(o.mu, o.iu, r.mu, r.iu)) r.mu = o.mu, r.iu = o.iu;
}

__device__ __forceinline__ void rec_from_acc(Part64Rec& r, const Acc64& a, long long ib) {
  for (int k = 0; k < PEAT_NCLASS; k++) r.cnt[k] = a.cnt[k];
  r.nfin = a.nfin;
  r.ahi = a.ma.hi, r.alo = a.ma.lo, r.asc = a.ma.sc, r.ia = a.ia ? ib + a.ia - 1 : -1;
  r.rhi = a.mr.a.hi, r.rlo = a.mr.a.lo, r.rsc = a.mr.a.sc, r.rg = a.mr.g, r.rkind = a.mr.kind, r.rle = a.mr.le, r.rlf = a.mr.lf;
  r.ir = a.ir ? ib + a.ir - 1 : -1;
  r.mu = a.mu, r.iu = a.iu ? ib + a.iu - 1 : -1;
}

// the CTA's records merged into thread 0's (every thread calls it)
__device__ void block_merge(Part64Rec& r, Part64Rec* buf) {
  buf[threadIdx.x] = r;
  __syncthreads();
  for (int w = TB / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) rec_merge(buf[threadIdx.x], buf[threadIdx.x + w]);
    __syncthreads();
  }
  r = buf[0];
  __syncthreads();
}

// carry-normalise n limbs of 32-bit digits (thread 0): every limb in [0, 2^32), the top one signed
__device__ void normalise(long long* d, int n) {
  long long carry = 0;
  for (int j = 0; j < n - 1; j++) {
    const long long v = d[j] + carry;
    carry = v >> 32;
    d[j] = v & 0xFFFFFFFFll;
  }
  d[n - 1] += carry;
}

__global__ void __launch_bounds__(TB, 2) compare64_stage1(Cmp64Params p) {
  __shared__ unsigned H[PEAT_HIST_BINS];
  __shared__ long long S[3 * SL];
  __shared__ Part64Rec buf[TB];
  pdl_trigger();  // the finalize kernel may start launching (it waits for this grid)
  const int lane = threadIdx.x & 31;
  for (long long item = blockIdx.x; item < p.nitems; item += gridDim.x) {
    const long long b = p.item_b[item], e = p.item_e[item], seg = p.item_seg[item];
    const long long base = p.offsets[seg];
    for (int k = threadIdx.x; k < PEAT_HIST_BINS; k += TB) H[k] = 0u;
    for (int k = threadIdx.x; k < 3 * SL; k += TB) S[k] = 0;
    __syncthreads();
    Acc64 acc;
    acc64_init(acc);
    // pairs of elements (one 16-byte vector of each tensor) on the absolute index grid
    const long long q0 = b >> 1, q1 = (e + 1) >> 1;
    for (long long q = q0 + threadIdx.x; __any_sync(0xFFFFFFFFu, q < q1); q += TB) {
      const bool okq = q < q1;
      const long long i0 = q << 1;
      uint64_t gw[2] = {0, 0}, cw[2] = {0, 0};
      if (okq && p.vec && i0 >= b && i0 + 2 <= e) {
        const ulonglong2 gv = __ldg(reinterpret_cast<const ulonglong2*>(p.g) + q);
        const ulonglong2 cv = __ldg(reinterpret_cast<const ulonglong2*>(p.c) + q);
        gw[0] = gv.x, gw[1] = gv.y, cw[0] = cv.x, cw[1] = cv.y;
      } else if (okq) {
        for (int j = 0; j < 2; j++)
          if (i0 + j >= b && i0 + j < e) {
            gw[j] = __ldg(reinterpret_cast<const unsigned long long*>(p.g) + i0 + j);
            cw[j] = __ldg(reinterpret_cast<const unsigned long long*>(p.c) + i0 + j);
          }
      }
#pragma unroll 1
      for (int j = 0; j < 2; j++) {
        const long long i = i0 + j;
        pair64(p, acc, H, S, j ? gw[1] : gw[0], j ? cw[1] : cw[0], okq && i >= b && i < e, (uint32_t)(i - b));
      }
    }
    win_flush(acc.sd, acc.bd, S);
    win_flush(acc.sa, acc.ba, S + SL);
    win3_flush(acc.sq, S + 2 * SL);
    Part64Rec r;
    rec_from_acc(r, acc, b - base);
    block_merge(r, buf);
    Part64* out = p.parts + item;
    if (threadIdx.x == 0) {
      out->rec = r;
      for (int s = 0; s < 3; s++) normalise(S + s * SL, SL);
    }
    __syncthreads();
    for (int k = threadIdx.x; k < 3 * SL; k += TB) out->limbs[k] = S[k];
    if (p.hist)
      for (int k = threadIdx.x; k < PEAT_HIST_BINS; k += TB)
        if (H[k]) atomicAdd(p.hist + seg * PEAT_HIST_BINS + k, (unsigned long long)H[k]);
    __syncthreads();
  }
  (void)lane;
}

// RN64 of a normalised limb sum (limbs in [0, 2^32), the top one signed), with
// the subnormal grid below 2^-1022 and +-inf past the largest double
__device__ double limbs_rn64(const long long* d) {
  // magnitude limbs
  unsigned long long m[SL];
  const bool neg = d[SL - 1] < 0;
  // a top limb of 32 bits or more is past 2^2080, far beyond the largest double
  if (d[SL - 1] >= (1ll << 32) || d[SL - 1] < -(1ll << 32))
    return neg ? -__longlong_as_double(0x7FF0000000000000ll) : __longlong_as_double(0x7FF0000000000000ll);
  long long borrow = 0;
  for (int j = 0; j < SL; j++) {
    long long v = neg ? -d[j] - borrow : d[j];
    if (neg) {
      borrow = v < 0 ? 1 : 0;
      v += borrow ? (1ll << 32) : 0;
    }
    m[j] = (unsigned long long)v;
  }
  int top = -1;
  for (int j = SL - 1; j >= 0 && top < 0; j--)
    if (m[j]) top = j * 32 + 31 - __clz((int)(uint32_t)m[j]);
  if (top < 0) return 0.0;
  auto bit = [&](int k) -> unsigned long long { return k < 0 ? 0ull : (m[k >> 5] >> (k & 31)) & 1ull; };
  int low = top - 52;
  if (low + SLSB < -1074) low = -1074 - SLSB;
  unsigned long long mant = 0;
  for (int k = top; k >= low; k--) mant = (mant << 1) | bit(k);
  const unsigned long long round = bit(low - 1);
  bool sticky = false;
  for (int k = low - 2; k >= 0 && !sticky; k--) sticky = bit(k) != 0;
  if (round && (sticky || (mant & 1ull))) mant++;
  const double r = ldexp((double)mant, low + SLSB);
  return neg ? -r : r;
}

// RN64 of (hi + lo) 2^sc / g (finite positive): the candidate around the
// binary64 quotient whose neighbouring midpoints bracket the exact value
__device__ double rel_value64(const Mag& a, double g) {
  // at or past (2^54 - 1) 2^970 (the rounding threshold of the largest double): +inf
  {
    uint64_t mg;
    int eg;
    split_d(g, mg, eg);
    XTerm t[3] = {dbl_term(a.hi, a.sc, false), dbl_term(fabs(a.lo), a.sc, a.lo < 0.0),
                  XTerm{(u128)mg * ((1ull << 54) - 1), eg + 970, true}};
    if (xsign(t, 3) >= 0) return __longlong_as_double(0x7FF0000000000000ll);
  }
  double q = ldexp(__ddiv_rn(a.hi, g), a.sc);
  if (!(q <= 1.7976931348623157e308)) q = 1.7976931348623157e308;
  // sign of x - m g for x = (hi + lo) 2^sc and a midpoint m = (q1 + q2) / 2
  auto above_mid = [&](double q1, double q2) -> int {
    XTerm t[4] = {dbl_term(a.hi, a.sc + 1, false), dbl_term(fabs(a.lo), a.sc + 1, a.lo < 0.0),
                  prod_term(q1, g, 0, true), prod_term(q2, g, 0, true)};
    return xsign(t, 4);
  };
  for (int it = 0; it < 8; it++) {
    const double up = nextafter(q, 1.0 / 0.0), dn = nextafter(q, 0.0);
    if (q < 1.7976931348623157e308) {  // below the threshold checked above, the result is finite
      const int su = above_mid(q, up);
      if (su > 0 || (su == 0 && (__double_as_longlong(q) & 1))) {
        q = up;
        continue;
      }
    }
    if (q > 0.0) {
      const int sd = above_mid(dn, q);
      if (sd < 0 || (sd == 0 && (__double_as_longlong(q) & 1))) {
        q = dn;
        continue;
      }
    }
    break;
  }
  return q;
}

__global__ void __launch_bounds__(TB) compare64_finalize(Cmp64Params p) {
  __shared__ Part64Rec buf[TB];
  __shared__ long long S[3 * SL];
  pdl_wait();  // stage 1 complete
  const long long seg = blockIdx.x;
  const long long f0 = p.seg_first[seg], f1 = p.seg_first[seg + 1];
  Part64Rec r;
  for (int k = 0; k < PEAT_NCLASS; k++) r.cnt[k] = 0;
  r.nfin = 0;
  r.ahi = r.alo = 0.0, r.asc = 0, r.ia = -1;
  r.rhi = r.rlo = 0.0, r.rsc = 0, r.rg = 1.0, r.rkind = 0, r.rle = 0, r.rlf = 0.0f, r.ir = -1;
  r.mu = 0, r.iu = -1;
  for (long long it = f0 + threadIdx.x; it < f1; it += TB) rec_merge(r, p.parts[it].rec);
  block_merge(r, buf);
  for (int k = threadIdx.x; k < 3 * SL; k += TB) {
    long long v = 0;
    for (long long it = f0; it < f1; it++) v += p.parts[it].limbs[k];
    S[k] = v;
  }
  __syncthreads();
  // the mean and variance of |d| from S1 = sum |d| and S2 = sum d^2, both SL
  // digits weighing 2^(32 j + SLSB) (two more after carrying)
  __shared__ MeanVarScratch<SL + 2, SL + 2, -SLSB / 32> mv;
  static_assert(SLSB % 32 == 0, "the S2 shift is a whole number of digits");
  if (threadIdx.x == 0) carry_to_digits(S + SL, SL, mv.A);
  if (threadIdx.x == 32) carry_to_digits(S + 2 * SL, SL, mv.B);
  mean_var_block(mv, r.nfin, SLSB);
  if (threadIdx.x != 0) return;
  peat_stats_t o;
  o.n = (uint64_t)(p.offsets[seg + 1] - p.offsets[seg]);
  for (int k = 0; k < PEAT_NCLASS; k++) o.count[k] = r.cnt[k];
  o.n_finite = r.nfin;
  o.max_abs = r.ia >= 0 ? (r.asc ? __dmul_rn(r.ahi, 2.0) : r.ahi) : 0.0;  // RN(2 x) = 2 RN(x), +inf on overflow
  o.argmax_abs = r.ia;
  if (r.ir < 0 || r.rkind == 0) o.max_rel = 0.0;
  else if (r.rkind == 2) o.max_rel = __longlong_as_double(0x7FF0000000000000ll);
  else o.max_rel = rel_value64(Mag{r.rhi, r.rlo, r.rsc}, r.rg);
  o.argmax_rel = r.ir;
  o.max_ulp = r.iu >= 0 ? r.mu : 0;
  o.argmax_ulp = r.iu;
  for (int s = 0; s < 3; s++) normalise(S + s * SL, SL);
  o.sum_signed = limbs_rn64(S);
  o.sum_abs = limbs_rn64(S + SL);
  o.sum_sq = limbs_rn64(S + 2 * SL);
  o.rtol_eff = p.rtol;
  o.atol_eff = p.atol;
  o.mean_abs = mv.mean;
  o.var_abs = mv.var;
  p.stats[seg] = o;
}

}  // namespace

cudaError_t launch_compare64(const Cmp64Params& p, int nctas, cudaStream_t s) {
  if (p.nitems == 0) {
    compare64_finalize<<<(unsigned)p.nseg, TB, 0, s>>>(p);
    return cudaGetLastError();
  }
  compare64_stage1<<<nctas, TB, 0, s>>>(p);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_dependent(compare64_finalize, (unsigned)p.nseg, TB, 0, s, p);  // overlaps stage 1's end
}

}  // namespace peat
