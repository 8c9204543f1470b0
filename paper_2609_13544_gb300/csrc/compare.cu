// Golden-vs-candidate error signature on sm_103a.
//
// Computes, per tensor or per segment of a packed tensor list, the error
// statistics of Section IV-B-3 ("FI Assessment Scores": the error is the
// absolute difference of golden and faulty values; max, mean and variance
// of it) plus the relative error, the ULP distance, a five-way class and two
// 64-bin histograms.  Every output is exact: integer outputs bit for bit,
// sums as the exact real sum rounded once to nearest-even binary64.
//
// One kernel (compare_stage1) per call: a persistent grid streams both
// tensors once through per-warp rings of bulk copies (cp.async.bulk +
// mbarrier).  CTA b owns the contiguous element range [lo_b, lo_{b+1}); per
// segment piece it touches it adds its integer totals (counts, histograms,
// sum digits) to the segment's accumulator with atomics and writes its maxima
// to slot s + b; the CTA that finishes a segment's last piece merges the
// slots in CTA order, rounds the exact sums once, writes the outputs and
// clears the accumulator.  All merged quantities are integers or exact
// values, so the result depends neither on the grid nor on the order of the
// atomics.  Per element pair:
//   - bitwise-equal pairs are counted (whole warp tiles at once when equal);
//   - unequal pairs of a tile are compacted into a per-warp queue (element
//     order) and processed 32 at a time;
//   - a "window" pair -- ULP distance u < 2^UB (so the signs agree and c is
//     within a factor 2 of g: c - g is exact in float32, Sterbenz), |g| at
//     least 2^(Lb+1-bias), |d| < 2^(Lexp+22) -- is finished in float32 and
//     integer arithmetic: V = |d| / 2^Lexp is an integer below 2^22, read
//     from the bits of |d| + 1.5 * 2^(Lexp+23), so sum |d|, sum d and sum d^2
//     accumulate as integers; the log2-relative bin is the exponent
//     difference of |d| and |g|; the tolerance test is one float32 fma, exact
//     except at equality; a pair updates the exact maxima only when it lies
//     strictly above the thread's current ones (its pairs arrive in index
//     order, so ties keep the earlier index);
//   - every other pair (non-finite, sign change, zeros, wide gaps, outside
//     the window, tolerance ties) is listed and evaluated exactly after the
//     piece, with float32 error-free transforms and integer digits added to a
//     CTA-wide carry-save fixed-point accumulator.
// Binary64 arithmetic is avoided per element (GB300 runs it at a small
// fraction of float32 rate); binary64 values appear only as containers and
// in the once-per-segment rounding.
#include <cuda_fp16.h>

#include <cstdint>

#include "exact.cuh"
#include "inject_models.cuh"
#include "meanvar.cuh"
#include <nvtx3/nvToolsExt.h>
#include "peat_internal.h"

namespace peat {
namespace {

// ---------------------------------------------------------------------------
// element types
// ---------------------------------------------------------------------------
// UBMAX: the largest ULP-distance bit length the window's position allows
// for (the window sits 20 - UB binades deep below the largest golden seen).
// LBMIN and LBMAX bound the window's floor binade Lb so that 2^Lexp is a
// normal float32 (Lexp = Lb - BIAS - MB) and 1.5 * 2^(Lexp+23) is finite.
template <int DT>
struct Tr;
template <>
struct Tr<PEAT_F32> {
  static constexpr int BYTES = 4, VEC = 4, MB = 23, BIAS = 127, EMAX = 255;
  static constexpr int UBMAX = 12, LBMIN = 24, LBMAX = 221;
  static constexpr uint32_t SIGN = 0x80000000u, MAG = 0x7FFFFFFFu, INF = 0x7F800000u;
};
template <>
struct Tr<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 10, BIAS = 15, EMAX = 31;
  static constexpr int UBMAX = 10, LBMIN = 1, LBMAX = 30;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, INF = 0x7C00u;
};
template <>
struct Tr<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8, MB = 7, BIAS = 127, EMAX = 255;
  static constexpr int UBMAX = 7, LBMIN = 8, LBMAX = 221;
  static constexpr uint32_t SIGN = 0x8000u, MAG = 0x7FFFu, INF = 0x7F80u;
};

// Private per-thread histogram rows (16-bit counters, two threads per word):
// ULP bins 1..63 in rows 0..62, then the log2-relative bins window pairs
// reach, k in [KLO, KHI] in rows 63 + k - KLO (fp16 goldens may be subnormal,
// whose ratios reach 2^(MB-1)).
constexpr int NUR = 63;  // ULP rows
template <int DT>
struct Rows {
  static constexpr int KLO = -(Tr<DT>::MB + 1);
  // a window pair has c within a factor 2 of g, so |d| < |g| (k <= -1) unless
  // g is an fp16 subnormal (|d| up to 2^MB - 1 steps of it)
  static constexpr int KHI = DT == PEAT_F16 ? Tr<DT>::MB - 1 : -1;
  static constexpr int NPB = NUR + KHI - KLO + 1;
};
constexpr int HALF = BLOCK / 2;
constexpr int ROWB = HALF * 4;  // bytes per private row
constexpr int NPB_MAX = NUR + 24;  // float32: k in [-24, -1]

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

// The candidate of a fused call: the golden after the call's element-wise
// models, in order (the same arithmetic as the injector's passes).
// (out of line: the scalar paths that call it are rare, and one copy keeps
// the generation code out of their inlined bodies)
template <int DT>
__device__ __noinline__ uint32_t inj_chain(const CompareParams& p, uint32_t b, int64_t i) {
  for (int m = 0; m < p.inj_n; m++) {
    bool fired;
    b = inj::apply_model<DT>(b, i, p.inj[m].kind, p.inj[m].model, p.inj[m].threshold, p.inj[m].x, p.inj_k0,
                             p.inj_k1, fired);
  }
  return b;
}
// candidate element i (golden bits G): generated (fused) or read
template <int DT, bool INJ>
__device__ __forceinline__ uint32_t cand_at(const CompareParams& p, int64_t i, uint32_t G) {
  if constexpr (INJ) return inj_chain<DT>(p, G, i);
  else return load_scalar<DT>(p.c, i);
}
template <int DT>
__device__ __forceinline__ void unpack_vec(const uint4& v, uint32_t (&e)[16 / Tr<DT>::BYTES]) {
#pragma unroll
  for (int j = 0; j < 16 / Tr<DT>::BYTES; j++) e[j] = lane_bits<DT>(v, j);
}
template <int DT>
__device__ __forceinline__ uint4 pack_vec(const uint32_t (&e)[16 / Tr<DT>::BYTES]) {
  if constexpr (Tr<DT>::BYTES == 4) return make_uint4(e[0], e[1], e[2], e[3]);
  else
    return make_uint4(e[0] | (e[1] << 16), e[2] | (e[3] << 16), e[4] | (e[5] << 16), e[6] | (e[7] << 16));
}

// the candidate vector of golden vector gv whose first element is i0: whole
// blocks of four (one draw each) when i0 is on the block grid, else element
// by element
template <int DT>
__device__ __forceinline__ uint4 inj_vec(const CompareParams& p, const uint4& gv, int64_t i0) {
  constexpr int VEC = 16 / Tr<DT>::BYTES, NB = VEC / 4;
  uint32_t e[VEC];
  unpack_vec<DT>(gv, e);
  if ((i0 & 3) == 0) {
    for (int m = 0; m < p.inj_n; m++) {
      const InjStep st = p.inj[m];
      inj::with_kind(st.kind, [&](auto k) {
        inj::apply_blocks<DT, decltype(k)::value, NB>(e, i0, st.model, st.threshold, st.x, p.inj_k0, p.inj_k1);
      });
    }
  } else {
#pragma unroll
    for (int j = 0; j < VEC; j++) e[j] = inj_chain<DT>(p, e[j], i0 + j);
  }
  return pack_vec<DT>(e);
}

// The candidate chunk of a fused call, ct[v] for golden gt[v], v = lane,
// lane + 32, ... < nvalid, vector v starting at element i0 + v VEC: model by
// model over the chunk (one branch on the kind per model, then code without
// branches), each lane rewriting its own vectors in place.  Out of line,
// called once per chunk.
template <int DT>
__device__ __noinline__ void inj_chunk(const CompareParams& p, const uint4* gt, uint4* ct, int nvalid, int64_t i0) {
  constexpr int VEC = 16 / Tr<DT>::BYTES, NB = VEC / 4;
  const int lane = threadIdx.x & 31;
  if ((i0 & 3) != 0) {  // off the block grid
    for (int v = lane; v < nvalid; v += 32) ct[v] = inj_vec<DT>(p, gt[v], i0 + (int64_t)v * VEC);
    return;
  }
  for (int m = 0; m < p.inj_n; m++) {
    const InjStep st = p.inj[m];
    const uint4* src = m == 0 ? gt : ct;
    inj::with_kind(st.kind, [&](auto k) {
      for (int v = lane; v < nvalid; v += 32) {
        uint32_t e[VEC];
        unpack_vec<DT>(src[v], e);
        inj::apply_blocks<DT, decltype(k)::value, NB>(e, i0 + (int64_t)v * VEC, st.model, st.threshold, st.x,
                                                       p.inj_k0, p.inj_k1);
        ct[v] = pack_vec<DT>(e);
      }
    });
  }
}

// one candidate vector, out of line (the window sample of a piece)
template <int DT>
__device__ __noinline__ uint4 inj_one(const CompareParams& p, uint4 gv, int64_t i0) {
  return inj_vec<DT>(p, gv, i0);
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
__device__ __noinline__ int cmp_rel_exact(float h1, float l1, int s1, float g1, float h2, float l2, int s2, float g2) {
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
// Exact maxima records and class counters of the general path (|d| as
// (hi + lo) 2^sc, see Partial); registers of run_general.
struct GenRec {
  float abs_hi, abs_lo;
  float rel_hi, rel_lo, rel_g;
  float rel_f;  // filter of the rel best
  uint32_t ulp;
  uint32_t n_gw, n_gm, n_ga, n_gf, n_nf, n_geq;
  int abs_sc, rel_sc;
  long long abs_idx, rel_idx, ulp_idx;
};

// Maxima of the window pairs one thread evaluated exactly (offsets from the
// CTA's first element; ties to the lower offset).  The rel record keeps |d|
// and |g| of its pair (rd = 0: none).
struct WinRec {
  float amax, rd, rg;
  uint32_t aidx, umax, uidx, ridx, pad;
};

// Per-warp staging ring for the bulk copies: NSTAGE stages, each one warp
// tile of CHV 16-byte vectors of each tensor (two vectors per lane).
constexpr int NW = BLOCK / 32;

// scratch of the mean and variance of |d|: S1 = sum |d| and S2 = sum d^2,
// both NLIMB digits weighing 2^(32 j + LIMB_LSB) (two more after carrying)
using MV = MeanVarScratch<NLIMB + 2, NLIMB + 2, -LIMB_LSB / 32>;
static_assert(LIMB_LSB % 32 == 0, "the S2 shift is a whole number of digits");

// scratch of a segment's finalization
struct FinScratch {
  unsigned long long cnt[8];
  long long limbs[NSUM * NLIMB];
  Partial wbest[NW];
  double sums[NSUM];
};
constexpr int NSTAGE = 2;  // a power of two: stage and phase are bit fields of the use count
constexpr int RWMAX = 6;   // window moves per warp and piece
constexpr int CHV = 64;
constexpr int GSM = 128;   // general pairs per piece kept in shared memory

struct __align__(128) Smem {
  union {  // the mean/variance scratch of a finalizing CTA reuses the (by then idle) staging ring
    uint4 ring_g[NW][NSTAGE][CHV];
    MV mv;
  };
  uint4 ring_c[NW][NSTAGE][CHV];
  unsigned long long bar[NW][NSTAGE];
  unsigned long long hist[HBINS];
  unsigned long long sacc[NSUM][NLIMB];
  unsigned long long cnt[8];
  Partial wbest[NW];
  long long lo;                    // the CTA's first element
  long long ff, fu;                // first finite pair, first pair without NaN (search result)
  uint32_t* glist;                 // this CTA's list of general pairs (offsets), GCAP entries
  uint32_t gn;                     // entries appended in this piece (may exceed GCAP)
  // the first GSM entries of the list stay here, with the pairs' bits
  uint32_t gs_off[GSM], gs_g[GSM], gs_c[GSM];
  uint32_t nfe;                    // bitwise-equal pairs holding NaN or Inf
  int last;                        // this CTA finished the last piece of a one-segment call
  unsigned pieces;                 // a one-segment call's pieces: the CTAs whose ranges are not empty
  FinScratch fin;
  int lb, ub;
  // each warp's windows in the current piece: window r applies from the warp's
  // chunk wstart[w][r] on (r = 0: the piece's initial window, also for the head)
  uint32_t nwin[NW];
  uint32_t wstart[NW][RWMAX + 1];
  int wlb[NW][RWMAX + 1];
  WinRec rec[BLOCK];
  uint32_t priv[NPB_MAX * HALF];   // per-thread 16-bit counters, two threads per word
  unsigned short qp[NW][CHV * 8];  // per-warp queue: tile positions of the unequal pairs
  // the general path's totals, one copy per warp (fewer threads contend for an
  // address), folded into hist and sacc at the end of each piece
  unsigned long long ghist[NW][HBINS];
  unsigned long long gsacc[NW][NSUM][NLIMB];
};

__device__ __forceinline__ void sacc_add(Smem& sm, int which, unsigned __int128 m, int e, bool neg) {
  for_digits(m, e, neg, [&](int j, int64_t v) { atomicAdd(&sm.sacc[which][j], (unsigned long long)v); });
}
// General-path terms, one per lane of a converged warp, into the warp's copy
// of the sum digits: lanes whose digit indices agree are summed in registers
// first (__match_any_sync groups them; the 32-bit reductions take each signed
// digit value as a signed 16-bit high part and an unsigned 16-bit low part,
// so that no group sum overflows), and one lane per group adds the total.
// Without this, the lanes of a warp would serialise on 64-bit shared atomics
// to the same few digits.
__device__ __forceinline__ void wsacc_add(Smem& sm, int which, uint64_t m, int e, bool neg, bool on) {
  on = on && m != 0;
  if (!__any_sync(0xFFFFFFFFu, on)) return;
  const int lane = threadIdx.x & 31;
  const int p = e - LIMB_LSB, j = p >> 5, r = p & 31;
  const uint32_t m0 = (uint32_t)m, m1 = (uint32_t)(m >> 32);
  const uint32_t out[3] = {m0 << r, (m1 << r) | (r ? m0 >> (32 - r) : 0u), r ? m1 >> (32 - r) : 0u};
  unsigned long long* d = sm.gsacc[threadIdx.x >> 5][which];
#pragma unroll
  for (int k = 0; k < 3; k++) {
    const bool ok = on && out[k] != 0u && (unsigned)(j + k) < (unsigned)NLIMB;
    const unsigned grp = __match_any_sync(0xFFFFFFFFu, ok ? j + k : -1);
    const int64_t v = ok ? (neg ? -(int64_t)out[k] : (int64_t)out[k]) : 0;
    const uint32_t slo = __reduce_add_sync(grp, (uint32_t)v & 0xFFFFu);
    const int32_t shi = (int32_t)__reduce_add_sync(grp, (uint32_t)(int32_t)(v >> 16));
    if (ok && lane == __ffs(grp) - 1) atomicAdd(d + j + k, (unsigned long long)((int64_t)shi * 65536 + slo));
  }
}
__device__ __forceinline__ void wsacc_add_f(Smem& sm, int which, float x, int sc, bool on) {
  int e = 0;
  const uint32_t m = x != 0.0f ? split_float(x, e) : 0u;
  wsacc_add(sm, which, m, e + sc, x < 0.0f, on);
}
__device__ __forceinline__ void wsacc_add_prod_f(Smem& sm, int which, float x, float y, int sc, bool on) {
  int ex = 0, ey = 0;
  const uint32_t mx = x != 0.0f ? split_float(x, ex) : 0u, my = y != 0.0f ? split_float(y, ey) : 0u;
  wsacc_add(sm, which, (uint64_t)mx * my, ex + ey + sc, (x < 0.0f) != (y < 0.0f), on);
}
// one histogram bin per lane (bin < 0: none), counted once per distinct bin
__device__ __forceinline__ void whist_add(Smem& sm, int bin) {
  const unsigned grp = __match_any_sync(0xFFFFFFFFu, bin);
  if (bin >= 0 && (threadIdx.x & 31) == __ffs(grp) - 1 && PEAT_CHECK(bin < HBINS))
    atomicAdd(&sm.ghist[threadIdx.x >> 5][bin], (unsigned long long)__popc(grp));
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

// The general path: the definitions evaluated exactly, for any pair.  The
// per-lane part: class counters and maxima into cd; the histogram bins and
// the sum terms it returns are added by the whole warp (general_lane).
struct GenOut {
  int hb0, hb1;      // log2-relative bin and 64 + ULP bin, or -1
  float s, t;        // d = (s + t) 2^sc, both zero when the pair adds no terms
  int sc;
};
template <int DT>
__device__ __forceinline__ void general_pair(GenRec& cd, GenOut& o, uint32_t G, uint32_t C, int64_t idx, float rtol,
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
    o.hb0 = 63;
    o.hb1 = 64 + (ulpdef ? (u < 63 ? (int)u : 63) : 63);
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
  o.hb0 = rb;
  o.hb1 = 64 + (u < 63 ? (int)u : 63);
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
  o.s = s;
  o.t = t;
  o.sc = sc;
}
// One general pair per lane of a converged warp (valid: the lane has one):
// the per-lane part, then the histogram bins and the exact sums, d = (s + t)
// 2^sc, |d| = (hi + lo) 2^sc with (hi, lo) = +-(s, t), d^2 = (s^2 + 2st +
// t^2) 4^sc, added by the whole warp.
template <int DT>
__device__ __forceinline__ void general_lane(Smem& sm, GenRec& cd, uint32_t G, uint32_t C, int64_t idx, float rtol,
                                             float atol, bool valid) {
  GenOut o{-1, -1, 0.0f, 0.0f, 0};
  if (valid) general_pair<DT>(cd, o, G, C, idx, rtol, atol);
  whist_add(sm, o.hb0);
  whist_add(sm, o.hb1);
  const bool on = o.s != 0.0f;
  const bool neg = o.s < 0.0f;
  const float hi = neg ? -o.s : o.s, lo = neg ? -o.t : o.t;
  wsacc_add_f(sm, 0, o.s, o.sc, on);
  wsacc_add_f(sm, 0, o.t, o.sc, on);
  wsacc_add_f(sm, 1, hi, o.sc, on);
  wsacc_add_f(sm, 1, lo, o.sc, on);
  wsacc_add_prod_f(sm, 2, o.s, o.s, 2 * o.sc, on);
  wsacc_add_prod_f(sm, 2, o.s, o.t, 2 * o.sc + 1, on);
  wsacc_add_prod_f(sm, 2, o.t, o.t, 2 * o.sc, on);
}

// ---------------------------------------------------------------------------
// per-thread window state and per-piece window constants (registers)
// ---------------------------------------------------------------------------
struct Lane {
  uint32_t sa, sn;   // this tile's sum of V, and of V over negative d
  uint32_t within;   // window pairs within tolerance
  uint32_t uneq;     // unequal pairs seen (the rest of the piece is bitwise equal)
  uint32_t ndef;     // pairs sent to the general path in the current tile
  uint64_t A, N, Q;  // this round's sums of V, of V over negative d, of V^2
};

// This thread's window maxima so far (its pairs come in increasing index
// order): a later pair at or below them cannot be a maximum of the piece, so
// only pairs strictly above one of them are evaluated exactly.
struct Thr {
  float ta;       // |d|
  uint32_t tu;    // ud
  float tra, trm; // ratio tra / trm
};

// The window (warp-uniform; a warp moves it when too many of a tile's pairs
// fall outside): Lb is the floor binade, Lexp = Lb - BIAS - MB the weight of
// V's unit.
struct Win {
  float rtol, atol;
  float gmin;       // smallest |g| of a window pair: 2^(Lb + 1 - BIAS)
  float lim;        // |d| < 2^(Lexp + 22)
  float M;          // 1.5 * 2^(Lexp + 23): bits(|d| + M) - bits(M) = |d| / 2^Lexp
  int lb;           // Lb
  uint32_t base;    // shared address of this thread's counter in private row 0
  uint32_t inc;     // 1 (low half of the word) or 65536 (high half)
};

// the window with floor binade lb
template <int DT>
__device__ __forceinline__ void set_window_lb(Win& W, int lb) {
  using Ty = Tr<DT>;
  const int lexp = lb - Ty::BIAS - Ty::MB;
  W.lb = lb;
  W.gmin = (DT == PEAT_F16 && lb == Ty::LBMIN) ? __uint_as_float((uint32_t)(127 - 24) << 23)
                                                 : __uint_as_float((uint32_t)(lb + 1 - Ty::BIAS + 127) << 23);
  W.lim = __uint_as_float((uint32_t)(lexp + 22 + 127) << 23);
  W.M = __uint_as_float(((uint32_t)(lexp + 23 + 127) << 23) | 0x400000u);
}
// The window placed for data whose largest finite golden exponent is emax and
// whose ULP distances have ubits bits: V = |d| / 2^Lexp < 2^22 for such pairs
// with goldens up to 2 binades above emax (one bit to spare on u).
template <int DT>
__device__ __forceinline__ int window_floor(int emax, int ubits) {
  using Ty = Tr<DT>;
  const int UB = min(ubits + 1, Ty::UBMAX);
  const int lb = emax + UB - 20;
  return lb < Ty::LBMIN ? Ty::LBMIN : (lb > Ty::LBMAX ? Ty::LBMAX : lb);
}
template <int DT>
__device__ __forceinline__ int win_lexp(const Win& W) {
  return W.lb - Tr<DT>::BIAS - Tr<DT>::MB;
}

__device__ __forceinline__ void lane_init(Lane& L) {
  L.sa = L.sn = 0;
  L.within = L.uneq = L.ndef = 0;
  L.A = L.N = L.Q = 0;
}
__device__ __forceinline__ void thr_init(Thr& T) {
  T.ta = 0.0f;
  T.tu = 0;
  T.tra = 0.0f;
  T.trm = 1.0f;
}
__device__ __forceinline__ void rec_init(WinRec& r) {
  r.amax = r.rd = 0.0f;
  r.rg = 1.0f;
  r.aidx = r.uidx = r.ridx = 0xFFFFFFFFu;
  r.umax = 0;
  r.pad = 0;
}
__device__ __forceinline__ void gen_init(GenRec& c) {
  c.abs_hi = c.abs_lo = 0.0f;
  c.rel_hi = c.rel_lo = 0.0f;
  c.rel_g = 1.0f;
  c.rel_f = 0.0f;
  c.ulp = 0;
  c.n_gw = c.n_gm = c.n_ga = c.n_gf = c.n_nf = c.n_geq = 0;
  c.abs_sc = c.rel_sc = 0;
  c.abs_idx = c.rel_idx = c.ulp_idx = -1;
}

__device__ __forceinline__ void red_shared(uint32_t addr, uint32_t v) {
  asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

// sign(an1 / m1 - an2 / m2) > 0 for the normalised ratios of window pairs
template <int DT>
__device__ __forceinline__ bool rel_greater(float an1, float m1, float an2, float m2) {
  const float p = __fmul_rn(an1, m2), q = __fmul_rn(an2, m1);
  if constexpr (DT == PEAT_F32) {
    // an has at most UB + 2 significant bits, m 24: the products need an
    // error term, which is exact (no underflow: both products exceed 2^-26)
    const float ep = __fmaf_rn(an1, m2, -p), eq = __fmaf_rn(an2, m1, -q);
    return p > q || (p == q && ep > eq);
  } else {
    // at most (UB + 2) + (MB + 1) <= 24 significant bits: both products exact
    return p > q;
  }
}

// ---------------------------------------------------------------------------
// one unequal pair
// ---------------------------------------------------------------------------

// The window test.  gr, cr: raw bits (bf16: the float32 bits, i.e. raw << 16);
// gf, cf: the values.  Also returns ud (the ULP distance, bf16: scaled by
// 2^16), s = c - g, a = |s| and thr.  u < 2^MB keeps c within a factor 2 of
// g (so c - g is exact in float32, Sterbenz); |g| >= gmin makes g and c
// multiples of 2^Lexp; |d| < lim bounds V below 2^22; a tolerance tie goes to
// the general path.  No sign test is needed: a pair of opposite signs has
// ud > 2^23 (float32, bf16 scaled) or > 2^10 (fp16), beyond the bound.
template <int DT>
__device__ __forceinline__ uint32_t ud_bound() {
  return DT == PEAT_BF16 ? (1u << Tr<DT>::MB) << 16 : 1u << Tr<DT>::MB;
}
template <int DT>
__device__ __forceinline__ bool in_window(uint32_t gr, uint32_t cr, float gf, float cf, const Win& W, uint32_t& ud,
                                          float& s, float& a, float& thr) {
  {
    const uint32_t dd = DT == PEAT_F16 ? cr - gr : __float_as_uint(cf) - __float_as_uint(gf);
    ud = (int32_t)dd < 0 ? 0u - dd : dd;
  }
  s = __fsub_rn(cf, gf);
  a = fabsf(s);
  const float ag = fabsf(gf);
  thr = __fmaf_rn(W.rtol, ag, W.atol);
  return ud < ud_bound<DT>() && ag >= W.gmin && a < W.lim && a != thr;
}

// normalised ratio |d| / |g| = an / mg, mg in [1, 2)
__device__ __forceinline__ void norm_ratio(float a, float gf, float& an, float& mg) {
  const uint32_t gb = __float_as_uint(gf);
  an = __uint_as_float(__float_as_uint(a) - (gb & 0x7F800000u) + 0x3F800000u);
  mg = __uint_as_float((gb & 0x007FFFFFu) | 0x3F800000u);
}

// a pair outside the window: append it to the CTA's general list (evaluated
// at the end of the piece; past GCAP entries the piece is rescanned).  G, C:
// the pair's raw bits, kept with the first GSM entries.
__device__ __forceinline__ void defer_pair(uint32_t li, uint32_t G, uint32_t C, Smem& sm) {
  const uint32_t slot = atomicAdd(&sm.gn, 1u);
  if (slot < (uint32_t)GCAP) sm.glist[slot] = li;
}


// Everything of one unequal pair except its maxima; returns whether the pair
// lies strictly above one of the warp's maxima (it is then evaluated exactly
// by rescan_pair).
template <int DT>
__device__ __forceinline__ bool pair_proc(Lane& L, const Thr& T, uint32_t gr, uint32_t cr, float gf, float cf,
                                          uint32_t li, const Win& W, Smem& sm) {
  uint32_t ud;
  float s, a, thr;
  if (!in_window<DT>(gr, cr, gf, cf, W, ud, s, a, thr)) {
    defer_pair(li, DT == PEAT_BF16 ? gr >> 16 : gr, DT == PEAT_BF16 ? cr >> 16 : cr, sm);
    L.ndef++;
    return false;
  }
  L.within += a < thr ? 1u : 0u;
  float an, mg;
  norm_ratio(a, gf, an, mg);
  const int k = (int)(__float_as_uint(an) - __float_as_uint(mg)) >> 23;  // floor(log2(|d| / |g|))
  red_shared(W.base + (uint32_t)((NUR - Rows<DT>::KLO + k) * ROWB), W.inc);
  const uint32_t u = min(DT == PEAT_BF16 ? ud >> 16 : ud, (uint32_t)NUR);  // ULP bin, 63 = 63 or more
  red_shared(W.base + (u - 1) * ROWB, W.inc);
  // exact sums in units of 2^Lexp
  const uint32_t V = __float_as_uint(__fadd_rn(a, W.M)) - __float_as_uint(W.M);
  L.sa += V;
  L.sn += s < 0.0f ? V : 0u;
  L.Q += (uint64_t)V * V;
  return (a > T.ta) | (ud > T.tu) | rel_greater<DT>(an, mg, T.tra, T.trm);
}

// a candidate pair (a window pair strictly above one of this thread's maxima,
// later in index than all of them): update the exact records and thresholds
template <int DT>
__device__ __forceinline__ void rescan_pair(uint32_t gr, uint32_t cr, float gf, float cf, uint32_t li, const Win& W,
                                            WinRec& r, Thr& T) {
  uint32_t ud;
  float s, a, thr;
  in_window<DT>(gr, cr, gf, cf, W, ud, s, a, thr);
  float an, mg;
  norm_ratio(a, gf, an, mg);
  if (a > T.ta) {
    T.ta = a;
    r.amax = a;
    r.aidx = li;
  }
  if (ud > T.tu) {
    T.tu = ud;
    r.umax = ud;
    r.uidx = li;
  }
  if (rel_greater<DT>(an, mg, T.tra, T.trm)) {
    T.tra = an;
    T.trm = mg;
    r.rd = a;
    r.rg = fabsf(gf);
    r.ridx = li;
  }
}

// element j of a 16-byte vector: raw bits in the form pair_proc takes, and value
template <int DT>
__device__ __forceinline__ void elem(const uint4& v, int j, uint32_t& r, float& f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (DT == PEAT_F32) {
    r = w[j];
    f = __uint_as_float(r);
  } else if constexpr (DT == PEAT_BF16) {
    const uint32_t x = w[j >> 1];
    r = (j & 1) ? (x & 0xFFFF0000u) : (x << 16);
    f = __uint_as_float(r);
  } else {
    const uint32_t x = w[j >> 1];
    const __half2 h = *reinterpret_cast<const __half2*>(&x);
    r = (j & 1) ? (x >> 16) : (x & 0xFFFFu);
    f = (j & 1) ? __high2float(h) : __low2float(h);
  }
}

// element at position pos of a staged tile
template <int DT>
__device__ __forceinline__ void elem_at(const uint4* t, uint32_t pos, uint32_t& r, float& f) {
  if constexpr (DT == PEAT_F32) {
    r = reinterpret_cast<const uint32_t*>(t)[pos];
    f = __uint_as_float(r);
  } else if constexpr (DT == PEAT_BF16) {
    r = (uint32_t)reinterpret_cast<const unsigned short*>(t)[pos] << 16;
    f = __uint_as_float(r);
  } else {
    const unsigned short x = reinterpret_cast<const unsigned short*>(t)[pos];
    r = x;
    f = __half2float(__ushort_as_half(x));
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
__device__ __forceinline__ void count_equal(const uint4& g, uint32_t eqm, Smem& sm) {
  if (eqm && any_nonfinite<DT>(g)) atomicAdd(&sm.nfe, (uint32_t)__popc(nonfinite_lanes<DT>(g) & eqm));
}

__device__ __forceinline__ uint64_t wsum64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

// This warp's window sums (in units of 2^lexp) into the CTA's exact
// accumulator: A, N < 2^38 and Q < 2^60 per thread between flushes; warp sums
// in 128 bits.
__device__ __forceinline__ void flush_sums(Lane& L, Smem& sm, int lexp) {
  const uint64_t A = wsum64(L.A), N = wsum64(L.N);
  const uint64_t qlo = wsum64(L.Q & 0xFFFFFFFFull), qhi = wsum64(L.Q >> 32);
  if ((threadIdx.x & 31) == 0) {
    const uint64_t P = A - N;  // sum of V over positive d
    if (P >= N) sacc_add(sm, 0, (unsigned __int128)(P - N), lexp, false);
    else sacc_add(sm, 0, (unsigned __int128)(N - P), lexp, true);
    sacc_add(sm, 1, (unsigned __int128)A, lexp, false);
    sacc_add(sm, 2, (unsigned __int128)qlo + ((unsigned __int128)qhi << 32), 2 * lexp, false);
  }
  L.A = L.N = L.Q = 0;
}

// When a tile sent many pairs (at least 32, and a quarter of its unequal
// ones) to the general path, the warp moves its window to the tile's own data
// -- largest finite golden exponent, largest same-sign ULP distance -- after
// flushing the sums kept in the old window's units, and logs the move so that
// a rescan of the piece applies to every pair the window it saw.  At most
// RWMAX moves per warp and piece.
// the window floor for the data of a staged tile (out of line: rarely run)
template <int DT>
__device__ __noinline__ int tile_window_floor(const uint4* gt, const uint4* ct, int nvalid) {
  using Ty = Tr<DT>;
  const int lane = threadIdx.x & 31;
  uint32_t emax = 0, umax = 0;
#pragma unroll
  for (int v = 0; v < 2; v++) {
    if (lane + 32 * v >= nvalid) continue;
    const uint4 gv = gt[lane + 32 * v], cv = ct[lane + 32 * v];
#pragma unroll
    for (int j = 0; j < Ty::VEC; j++) {
      const uint32_t G = lane_bits<DT>(gv, j), C = lane_bits<DT>(cv, j);
      const uint32_t e = (G & Ty::MAG) >> Ty::MB;
      if (e < (uint32_t)Ty::EMAX && e > emax) emax = e;
      if (((G ^ C) & Ty::SIGN) == 0u && (G & Ty::MAG) < Ty::INF && (C & Ty::MAG) < Ty::INF)
        umax = max(umax, G > C ? G - C : C - G);
    }
  }
  emax = __reduce_max_sync(0xFFFFFFFFu, emax);
  umax = __reduce_max_sync(0xFFFFFFFFu, umax);
  return window_floor<DT>((int)emax, 32 - __clz(umax));
}

// nd: the warp's general pairs of this tile, total: its unequal pairs
template <int DT>
__device__ __forceinline__ void maybe_rewindow(Lane& L, Win& W, const uint4* gt, const uint4* ct, int nvalid,
                                               uint32_t nd, uint32_t total, uint32_t ichunk, Smem& sm) {
  if (nd < 32u || nd * 4u < total) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t r = sm.nwin[warp];
  if (r >= (uint32_t)RWMAX) return;
  const int lb = tile_window_floor<DT>(gt, ct, nvalid);
  if (lb == W.lb) return;
  flush_sums(L, sm, win_lexp<DT>(W));
  set_window_lb<DT>(W, lb);
  __syncwarp();
  if (lane == 0) {
    sm.wstart[warp][r + 1] = ichunk + 1;
    sm.wlb[warp][r + 1] = lb;
    sm.nwin[warp] = r + 1;
  }
  __syncwarp();
}

// One warp tile of CHV vectors staged in shared memory: lane L owns vectors L
// and L + 32; tile element e sits at offset tli + e from the CTA's first
// element.  Equal pairs are counted in place.  When at most a quarter of the
// pairs differ, each lane works through its own unequal pairs (cheaper than
// compacting a few); otherwise they are queued (in element order) and
// processed 32 at a time, so every thread does useful work.  Pairs above the
// thread's maxima are then evaluated exactly.
template <int DT>
__device__ __forceinline__ void do_tile(Lane& L, Thr& T, const uint4* gt, int nvalid, uint32_t tli, Win& W,
                                        uint32_t ichunk, Smem& sm) {
  // the candidate ring sits a fixed distance after the golden ring
  const uint4* ct = gt + (offsetof(Smem, ring_c) - offsetof(Smem, ring_g)) / sizeof(uint4);
  using Ty = Tr<DT>;
  constexpr int VEC = Ty::VEC;
  constexpr uint32_t FULL = (1u << VEC) - 1u;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool okA = lane < nvalid, okB = lane + 32 < nvalid;
  uint4 gA, cA, gB, cB;
  if (nvalid == CHV) {  // a full tile (all but the last of a piece)
    gA = gt[lane];
    cA = ct[lane];
    gB = gt[lane + 32];
    cB = ct[lane + 32];
  } else {
    const uint4 z = make_uint4(0, 0, 0, 0);
    gA = okA ? gt[lane] : z;
    cA = okA ? ct[lane] : z;
    gB = okB ? gt[lane + 32] : z;
    cB = okB ? ct[lane + 32] : z;
  }
  const bool diff = ((gA.x ^ cA.x) | (gA.y ^ cA.y) | (gA.z ^ cA.z) | (gA.w ^ cA.w) | (gB.x ^ cB.x) | (gB.y ^ cB.y) |
                     (gB.z ^ cB.z) | (gB.w ^ cB.w)) != 0u;
  if (!__any_sync(0xFFFFFFFFu, diff)) {  // the whole warp tile is bitwise equal
    if (okA) count_equal<DT>(gA, FULL, sm);
    if (okB) count_equal<DT>(gB, FULL, sm);
    return;
  }
  const uint32_t nA = okA ? unequal_mask<DT>(gA, cA) : 0u, nB = okB ? unequal_mask<DT>(gB, cB) : 0u;
  if (okA) count_equal<DT>(gA, FULL & ~nA, sm);
  if (okB) count_equal<DT>(gB, FULL & ~nB, sm);
  // one scan of the packed counts gives the A-queue and B-queue offsets (10-bit
  // fields: a warp tile has at most 512 pairs)
  const uint32_t packed = __popc(nA) | (__popc(nB) << 10);
  uint32_t incl = packed;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  const uint32_t tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
  const uint32_t totA = tot & 0x3FFu, total = totA + ((tot >> 10) & 0x3FFu);
  L.uneq += __popc(nA) + __popc(nB);
  if (total * 4u <= 64u * VEC) {
    // sparse tile: each lane visits its own unequal pairs (slot s < VEC:
    // element s of vector A, else element s - VEC of vector B; increasing index)
    uint32_t m = nA | (nB << VEC), cm = 0;
    while (m) {
      const uint32_t sl = __ffs(m) - 1;
      m &= m - 1u;
      const uint32_t pos = sl < (uint32_t)VEC ? lane * VEC + sl : (lane + 32) * VEC + sl - VEC;
      uint32_t gr, cr;
      float gf, cf;
      elem_at<DT>(gt, pos, gr, gf);
      elem_at<DT>(ct, pos, cr, cf);
      if (pair_proc<DT>(L, T, gr, cr, gf, cf, tli + pos, W, sm)) cm |= 1u << sl;
    }
    L.A += L.sa;
    L.N += L.sn;
    L.sa = L.sn = 0;
    if (cm) {
      WinRec& r = sm.rec[threadIdx.x];
      do {
        const uint32_t sl = __ffs(cm) - 1;
        cm &= cm - 1u;
        const uint32_t pos = sl < (uint32_t)VEC ? lane * VEC + sl : (lane + 32) * VEC + sl - VEC;
        uint32_t gr, cr;
        float gf, cf;
        elem_at<DT>(gt, pos, gr, gf);
        elem_at<DT>(ct, pos, cr, cf);
        rescan_pair<DT>(gr, cr, gf, cf, tli + pos, W, r, T);
      } while (cm);
    }
    L.ndef = 0;  // sparse tiles never move the window (a quarter of their pairs at most differ)
    __syncwarp();
    return;
  }
  uint32_t posA = (incl & 0x3FFu) - (packed & 0x3FFu);
  uint32_t posB = totA + ((incl >> 10) & 0x3FFu) - ((packed >> 10) & 0x3FFu);
  unsigned short* q = sm.qp[warp];
#pragma unroll
  for (int j = 0; j < VEC; j++) {
    if ((nA >> j) & 1u) q[posA++] = (unsigned short)(lane * VEC + j);
    if ((nB >> j) & 1u) q[posB++] = (unsigned short)((lane + 32) * VEC + j);
  }
  __syncwarp();
  // two queue entries per iteration (e, e + 32: in index order per lane);
  // bit o of cm marks this lane's o-th entry as a maxima candidate
  uint32_t cm = 0;
  uint32_t ob = 1;
  for (uint32_t e = lane; e < total; e += 64, ob <<= 2) {
    const uint32_t pos0 = q[e];
    const bool two = e + 32 < total;
    const uint32_t pos1 = two ? q[e + 32] : pos0;
    uint32_t gr0, cr0, gr1, cr1;
    float gf0, cf0, gf1, cf1;
    elem_at<DT>(gt, pos0, gr0, gf0);
    elem_at<DT>(ct, pos0, cr0, cf0);
    elem_at<DT>(gt, pos1, gr1, gf1);
    elem_at<DT>(ct, pos1, cr1, cf1);
    if (pair_proc<DT>(L, T, gr0, cr0, gf0, cf0, tli + pos0, W, sm)) cm |= ob;
    if (two && pair_proc<DT>(L, T, gr1, cr1, gf1, cf1, tli + pos1, W, sm)) cm |= ob << 1;
  }
  L.A += L.sa;
  L.N += L.sn;
  L.sa = L.sn = 0;
  if (cm) {
    WinRec& r = sm.rec[threadIdx.x];
    do {
      const uint32_t o = __ffs(cm) - 1;
      cm &= cm - 1u;
      const uint32_t pos = q[lane + 32 * o];
      uint32_t gr, cr;
      float gf, cf;
      elem_at<DT>(gt, pos, gr, gf);
      elem_at<DT>(ct, pos, cr, cf);
      rescan_pair<DT>(gr, cr, gf, cf, tli + pos, W, r, T);
    } while (cm);
  }
  {
    const uint32_t nd = __reduce_add_sync(0xFFFFFFFFu, L.ndef);
    L.ndef = 0;
    maybe_rewindow<DT>(L, W, gt, ct, nvalid, nd, total, ichunk, sm);
  }
  __syncwarp();
}

// one element outside the vector grid (li: offset from the CTA's first
// element), with its maxima evaluated exactly
template <int DT>
__device__ __forceinline__ void do_scalar(Lane& L, Thr& T, uint32_t G, uint32_t C, uint32_t li, const Win& W,
                                          Smem& sm) {
  using Ty = Tr<DT>;
  if (G == C) {
    if ((G & Ty::MAG) >= Ty::INF) atomicAdd(&sm.nfe, 1u);
    return;
  }
  L.uneq++;
  uint32_t gr = G, cr = C;
  float gf, cf;
  if constexpr (DT == PEAT_F32) {
    gf = __uint_as_float(G);
    cf = __uint_as_float(C);
  } else if constexpr (DT == PEAT_BF16) {
    gr = G << 16;
    cr = C << 16;
    gf = __uint_as_float(gr);
    cf = __uint_as_float(cr);
  } else {
    gf = __half2float(__ushort_as_half((unsigned short)G));
    cf = __half2float(__ushort_as_half((unsigned short)C));
  }
  if (pair_proc<DT>(L, T, gr, cr, gf, cf, li, W, sm)) rescan_pair<DT>(gr, cr, gf, cf, li, W, sm.rec[threadIdx.x], T);
  L.A += L.sa;
  L.N += L.sn;
  L.sa = L.sn = 0;
}

// ---------------------------------------------------------------------------
// CTA ranges: boundaries precomputed on the host
// ---------------------------------------------------------------------------
// The last CTA b with bounds[b] <= i (0 <= i), searched by a whole warp:
// each round the lanes probe 32 evenly spaced bounds of the bracket and a
// ballot keeps the last one at or below i, so 32^r CTAs take r rounds of
// parallel loads instead of a chain of log2(nctas) dependent ones.
__device__ __forceinline__ int cta_of_warp(int64_t i, const CompareParams& p) {
  const int lane = threadIdx.x & 31;
  int lo = 0, hi = p.nctas - 1;  // bounds[lo] = 0 <= i: the answer lies in [lo, hi]
  while (lo < hi) {
    const int step = (hi - lo + 32) / 32;
    const int q = lo + lane * step;
    const bool ok = lane == 0 || (q <= hi && __ldg(p.bounds + q) <= i);  // a prefix of the lanes (bounds ascend)
    const int t = 31 - __clz(__ballot_sync(0xFFFFFFFFu, ok));
    lo += t * step;
    hi = min(hi, lo + step - 1);
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

__device__ __forceinline__ int cmp_rel_rec(float h1, float l1, int s1, float g1, float h2, float l2, int s2, float g2) {
  const float tiny = 1.17549435e-38f;
  if (l1 == 0.0f && l2 == 0.0f && s1 == 0 && s2 == 0 && h1 >= tiny && h2 >= tiny && g1 >= tiny && g2 >= tiny)
    return cmp_ratio_f(h1, g1, h2, g2);
  return cmp_rel_exact(h1, l1, s1, g1, h2, l2, s2, g2);
}

// x <- the better of x and y, field by field; ties to the lower index
__device__ __forceinline__ void part_merge(Partial& x, const Partial& y) {
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
__device__ __forceinline__ void part_warp_reduce(Partial& x) {
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


// warp sums of the general path's class counters into the CTA counters
__device__ __forceinline__ void gen_counts(const GenRec& g, Smem& sm) {
  const int lane = threadIdx.x & 31;
  const uint32_t gen = g.n_gw + g.n_gm + g.n_ga + g.n_gf + g.n_geq;
  const uint32_t c[7] = {g.n_geq, gen, g.n_nf, g.n_gw, g.n_gm, g.n_ga, g.n_gf};
  uint32_t v[7];
#pragma unroll
  for (int k = 0; k < 7; k++) v[k] = __reduce_add_sync(0xFFFFFFFFu, c[k]);
  if (lane == 0) {
    if (v[0]) atomicAdd(&sm.cnt[0], (unsigned long long)v[0]);
    if (v[1]) atomicAdd(&sm.cnt[1], 0ull - (unsigned long long)v[1]);  // general pairs are not window pairs
    if (v[2]) atomicAdd(&sm.cnt[3], (unsigned long long)v[2]);
    if (v[3]) atomicAdd(&sm.cnt[4], (unsigned long long)v[3]);
    if (v[4]) atomicAdd(&sm.cnt[5], (unsigned long long)v[4]);
    if (v[5]) atomicAdd(&sm.cnt[6], (unsigned long long)v[5]);
    if (v[6]) atomicAdd(&sm.cnt[7], (unsigned long long)v[6]);
  }
}

// The general pairs of a piece [pb, pe), evaluated exactly by every thread of
// the CTA: from the list when it held them all, else found again by a rescan
// of the piece with the same window test.  Out of line, so that the hot loop
// carries no call.  Leaves each warp's general maxima in sm.wbest[warp].
template <int DT, bool INJ>
__device__ __noinline__ void run_general(Win W, Smem& sm, const CompareParams& p, int64_t pb, int64_t pe,
                                         int64_t vb, int64_t ve) {
  // entered only after a barrier and with at least one general pair (finish_piece)
  const uint32_t n = sm.gn;
  const int64_t lo = sm.lo;
  GenRec cd;
  gen_init(cd);
  // whole warps in every round (general_lane adds with the whole warp)
  const uint32_t lane = threadIdx.x & 31u, w0 = threadIdx.x & ~31u;
  if (n <= (uint32_t)GCAP) {
    for (uint32_t b = w0; b < n; b += BLOCK) {
      const uint32_t e = b + lane;
      const bool valid = e < n;
      int64_t i = 0;
      uint32_t G = 0, C = 0;
      if (valid) {
        i = lo + sm.glist[e];
        if (!PEAT_CHECK(i >= 0 && i < p.n_total)) i = lo;  // a listed offset outside the tensor
        G = load_scalar<DT>(p.g, i);
        C = cand_at<DT, INJ>(p, i, G);
      }
      general_lane<DT>(sm, cd, G, C, i, W.rtol, W.atol, valid);
    }
  } else {
    for (int64_t b = pb + w0; b < pe; b += BLOCK) {
      const int64_t i = b + lane;
      bool want = false;
      uint32_t G = 0, C = 0;
      if (i < pe) {
        G = load_scalar<DT>(p.g, i);
        C = cand_at<DT, INJ>(p, i, G);
        want = G != C;
      }
      if (want) {
        uint32_t gr = G, cr = C;
        if constexpr (DT == PEAT_BF16) {
          gr = G << 16;
          cr = C << 16;
        }
        // the window this pair was tested with: the head ran with the initial
        // window, a body chunk with its warp's window of that time, the tail
        // with its thread's warp's last window
        int w = 0;
        uint32_t ik = 0;
        if (vb < ve && i >= vb) {
          if (i >= ve) {
            w = (int)(((i - ve) % BLOCK) >> 5);
            ik = 0xFFFFFFFFu;
          } else {
            const int64_t k = (i - vb) / (CHV * Tr<DT>::VEC);
            w = (int)(k % NW);
            ik = (uint32_t)(k / NW);
          }
        }
        int r = (int)sm.nwin[w];
        while (r > 0 && sm.wstart[w][r] > ik) r--;
        Win Wi = W;
        set_window_lb<DT>(Wi, sm.wlb[w][r]);
        uint32_t ud;
        float s, a, thr;
        want = !in_window<DT>(gr, cr, to_f32<DT>(G), to_f32<DT>(C), Wi, ud, s, a, thr);
      }
      general_lane<DT>(sm, cd, G, C, i, W.rtol, W.atol, want);
    }
  }
  gen_counts(cd, sm);
  Partial x;
  part_none(x);
  x.abs_hi = cd.abs_hi;
  x.abs_lo = cd.abs_lo;
  x.abs_sc = cd.abs_sc;
  x.abs_idx = cd.abs_idx;
  x.rel_hi = cd.rel_hi;
  x.rel_lo = cd.rel_lo;
  x.rel_g = cd.rel_g;
  x.rel_sc = cd.rel_sc;
  x.rel_idx = cd.rel_idx;
  x.ulp = cd.ulp;
  x.ulp_idx = cd.ulp_idx;
  part_warp_reduce(x);
  if ((threadIdx.x & 31) == 0) sm.wbest[threadIdx.x >> 5] = x;
  __syncthreads();
  if (threadIdx.x == 0) sm.gn = 0;
}

// [pb, pe): the lowest index of a finite pair and of a pair without NaN
// (the argmax when every error is zero), searched BLOCK elements at a time
// (the piece's first pair, which settles both unless it holds NaN or Inf, is
// tested when the piece starts; this search runs only when it did not)
template <int DT, bool INJ>
__device__ __noinline__ void first_pairs(Smem& sm, const CompareParams& p, int64_t pb, int64_t pe) {
  using Ty = Tr<DT>;
  constexpr long long NONE = 0x7FFFFFFFFFFFFFFFll;
  for (int64_t base = pb;; base += BLOCK) {
    __syncthreads();
    if (base >= pe || (sm.ff != NONE && sm.fu != NONE)) break;
    const int64_t i = base + threadIdx.x;
    if (i < pe) {
      const uint32_t Gi = load_scalar<DT>(p.g, i);
      const uint32_t ag = Gi & Ty::MAG, ac = cand_at<DT, INJ>(p, i, Gi) & Ty::MAG;
      if (ag < Ty::INF && ac < Ty::INF) atomicMin(&sm.ff, (long long)i);
      if (ag <= Ty::INF && ac <= Ty::INF) atomicMin(&sm.fu, (long long)i);
    }
  }
  __syncthreads();
}

// Fold the per-thread 16-bit histograms and the window sums into the CTA
// totals.  All threads call it; it ends with the private counters zeroed.
template <int DT>
__device__ void fold_round(Lane& L, Smem& sm, int lexp) {
  constexpr int NPB = Rows<DT>::NPB;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  flush_sums(L, sm, lexp);  // lexp: this warp's window
  __syncthreads();
  // private rows: one warp per row
  for (int r = warp; r < NPB; r += NW) {
    uint32_t sum = 0;
    for (int w = lane; w < HALF; w += 32) {
      const uint32_t v = sm.priv[r * HALF + w];
      sum += (v & 0xFFFFu) + (v >> 16);
      sm.priv[r * HALF + w] = 0;
    }
    sum = __reduce_add_sync(0xFFFFFFFFu, sum);
    if (lane == 0 && sum) {
      const int bin = r < NUR ? 64 + r + 1 : 48 + Rows<DT>::KLO + (r - NUR);
      if (PEAT_CHECK(bin >= 0 && bin < HBINS)) sm.hist[bin] += sum;
    }
  }
  __syncthreads();
}

__device__ void finalize_segment(const CompareParams& p, int64_t s, FinScratch& f, MV& mv);
__device__ void write_empty_segments(const CompareParams& p);

// End of one segment piece [pb, pe): the integer totals go to the segment's
// accumulator (global atomics), the maxima to the CTA's partial slot.  The
// CTA that finishes the segment's last piece then finalizes the segment.
template <int DT, bool INJ>
__device__ __forceinline__ void finish_piece(Lane& L, const Win& W, Smem& sm, const CompareParams& p,
                                             int64_t seg, int64_t pb, int64_t pe, int64_t vb, int64_t ve) {
  Partial* out = p.partials + seg + blockIdx.x;
  SegAcc* acc = p.acc + seg;
  // the piece's general pairs, if any: the out-of-line call (and its register
  // traffic) only when there is one
  __syncthreads();
  if (sm.gn != 0) {
    run_general<DT, INJ>(W, sm, p, pb, pe, vb, ve);
  } else if ((threadIdx.x & 31) == 0) {
    part_none(sm.wbest[threadIdx.x >> 5]);
  }
  fold_round<DT>(L, sm, win_lexp<DT>(W));  // ends with a barrier: the general path's per-warp totals are complete
  for (int b = threadIdx.x; b < HBINS; b += BLOCK) {
    unsigned long long v = 0;
#pragma unroll
    for (int w = 0; w < NW; w++) {
      v += sm.ghist[w][b];
      sm.ghist[w][b] = 0;
    }
    sm.hist[b] += v;
  }
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) {
    unsigned long long v = 0;
#pragma unroll
    for (int w = 0; w < NW; w++) {
      v += (&sm.gsacc[w][0][0])[j];
      (&sm.gsacc[w][0][0])[j] = 0;
    }
    (&sm.sacc[0][0])[j] += v;
  }
  if (sm.ff == 0x7FFFFFFFFFFFFFFFll || sm.fu == 0x7FFFFFFFFFFFFFFFll) first_pairs<DT, INJ>(sm, p, pb, pe);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t lo = sm.lo;
  // window pairs = unequal pairs - general pairs; EXACT = the piece length -
  // unequal pairs + general pairs found equal (64-bit wrapping adds; the
  // totals are non-negative)
  {
    const uint32_t vu = __reduce_add_sync(0xFFFFFFFFu, L.uneq), vw = __reduce_add_sync(0xFFFFFFFFu, L.within);
    if (lane == 0) {
      if (vu) {
        atomicAdd(&sm.cnt[1], (unsigned long long)vu);
        atomicAdd(&sm.cnt[0], 0ull - (unsigned long long)vu);
      }
      if (vw) atomicAdd(&sm.cnt[2], (unsigned long long)vw);
    }
    if (threadIdx.x == 0) {
      atomicAdd(&sm.cnt[0], (unsigned long long)(pe - pb));
      atomicAdd(&sm.cnt[3], (unsigned long long)sm.nfe);
    }
  }
  // maxima: this thread's window record, then the warp's, merged with the
  // warp's general best
  {
    const WinRec r = sm.rec[threadIdx.x];
    Partial w;
    part_none(w);
    if (r.amax > 0.0f) {
      w.abs_hi = r.amax;
      w.abs_idx = lo + r.aidx;
    }
    if (r.rd > 0.0f) {
      w.rel_hi = r.rd;
      w.rel_g = r.rg;
      w.rel_idx = lo + r.ridx;
    }
    if (r.umax > 0u) {
      w.ulp = DT == PEAT_BF16 ? r.umax >> 16 : r.umax;
      w.ulp_idx = lo + r.uidx;
    }
    part_warp_reduce(w);
    if (lane == 0) {
      Partial x = sm.wbest[warp];
      part_merge(x, w);
      sm.wbest[warp] = x;
    }
  }
  __syncthreads();
  if (warp == 0) {
    Partial x;
    if (lane < NW) x = sm.wbest[lane];
    else part_none(x);
    part_warp_reduce(x);
    if (lane == 0) {
      constexpr long long NONE = 0x7FFFFFFFFFFFFFFFll;
      x.first_fin = sm.ff == NONE ? -1 : sm.ff;
      x.first_ulp = sm.fu == NONE ? -1 : sm.fu;
      if (PEAT_CHECK(seg >= 0 && seg < p.nseg && seg + (int64_t)blockIdx.x < p.nseg + p.nctas && pb <= pe &&
                     pe <= p.n_total))
        *out = x;
    }
  }
  for (int b = threadIdx.x; b < HBINS; b += BLOCK)
    if (sm.hist[b]) atomicAdd(&acc->hist[b], sm.hist[b]);
  if (threadIdx.x < 8 && sm.cnt[threadIdx.x]) atomicAdd(&acc->cnt[threadIdx.x], sm.cnt[threadIdx.x]);
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) {
    const unsigned long long v = (&sm.sacc[0][0])[j];
    if (v) atomicAdd(reinterpret_cast<unsigned long long*>(&acc->limbs[0][0]) + j, v);
  }
  // publish, then count this piece: the segment's pieces are the CTAs whose
  // ranges meet it (a multi-segment call finalizes in a second launch, after
  // this one)
  if (p.nseg == 1) __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    sm.last = 0;
    if (p.nseg == 1) {  // one segment: its last CTA finalizes it (else a second launch does, in parallel)
      sm.last = atomicAdd(&acc->done, 1u) == sm.pieces - 1u;
    }
  }
  // reset the CTA totals for the next piece
  for (int b = threadIdx.x; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = threadIdx.x; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  if (threadIdx.x < 8) sm.cnt[threadIdx.x] = 0;
  if (threadIdx.x == 0) sm.nfe = 0;
  rec_init(sm.rec[threadIdx.x]);
  lane_init(L);
  __syncthreads();
  if (sm.last) {
    __threadfence();
    finalize_segment(p, seg, sm.fin, sm.mv);
  }
}

// ---------------------------------------------------------------------------
// stage 1
// ---------------------------------------------------------------------------
constexpr int CTAS_PER_SM = 2;

template <int DT, bool INJ>
__global__ void __launch_bounds__(BLOCK, CTAS_PER_SM) compare_stage1(CompareParams p) {
  using Ty = Tr<DT>;
  using R = Rows<DT>;
  constexpr int VEC = Ty::VEC;
  // pairs per thread per round stay below 2^16 (16-bit private counters): each
  // warp tile gives a thread at most 2 VEC pairs
  constexpr int64_t ROUND_CHUNKS = (int64_t)NW * (65535 / (2 * VEC));
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  pdl_trigger();  // a multi-segment call's finalize kernel may start launching (it waits for this grid)
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int b = tid; b < HBINS; b += BLOCK) sm.hist[b] = 0;
  for (int j = tid; j < NSUM * NLIMB; j += BLOCK) (&sm.sacc[0][0])[j] = 0;
  for (int j = tid; j < R::NPB * HALF; j += BLOCK) sm.priv[j] = 0;
  for (int j = tid; j < NW * HBINS; j += BLOCK) (&sm.ghist[0][0])[j] = 0;
  for (int j = tid; j < NW * NSUM * NLIMB; j += BLOCK) (&sm.gsacc[0][0][0])[j] = 0;
  if (tid < 8) sm.cnt[tid] = 0;
  rec_init(sm.rec[tid]);
  const int64_t lo = p.bounds[blockIdx.x], hi = p.bounds[blockIdx.x + 1];
  if (tid == 0) {
    sm.lo = lo;
    sm.gn = 0;
    sm.nfe = 0;
    sm.glist = p.glist + (size_t)blockIdx.x * GCAP;
  }
  if (lane == 0) {
    for (int st = 0; st < NSTAGE; st++) mbar_init(&sm.bar[warp][st], 1);
    mbar_init_fence();
  }
  Win W;
  W.rtol = p.rtol;
  W.atol = p.atol;
  W.base = smem_addr(&sm.priv[tid & (HALF - 1)]);
  W.inc = tid < HALF ? 1u : 65536u;
  Lane L;
  lane_init(L);
  if (p.nseg == 1 && p.n_total > 0 && warp == 0) {  // (counted here, off the tail of the last piece)
    const int b1 = cta_of_warp(p.n_total - 1, p), b0 = cta_of_warp(0, p);
    if (lane == 0) sm.pieces = (unsigned)(b1 - b0 + 1);
  }
  __syncthreads();
  if (blockIdx.x == 0 && p.has_empty) write_empty_segments(p);
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
      const int64_t off = (vb + v0 * VEC) * Ty::BYTES;
      fence_proxy_async();
      mbar_expect_tx(&sm.bar[warp][st], INJ ? bytes : 2 * bytes);
      bulk_load(&sm.ring_g[warp][st][0], gbase + off, bytes, &sm.bar[warp][st]);
      if (!INJ) bulk_load(&sm.ring_c[warp][st][0], cbase + off, bytes, &sm.bar[warp][st]);
    };
    const int64_t my_chunks = nchunk > warp ? (nchunk - warp + NW - 1) / NW : 0;
    if (lane == 0 && !failed)
      for (int64_t i = 0; i < NSTAGE && i < my_chunks; i++) issue(seq + (uint32_t)i, warp + NW * i);
    // the window from a sample of the piece: the largest finite golden
    // exponent and the largest same-sign ULP distance of the first vectors
    if (tid == 0) sm.lb = sm.ub = 0;
    __syncthreads();
    // the piece's first pair (its loads overlap the sample's)
    uint32_t G0 = 0, C0 = 0;
    if (tid == 0) {
      G0 = load_scalar<DT>(p.g, pb);
      C0 = cand_at<DT, INJ>(p, pb, G0);
    }
    if (tid < nvec) {
      const uint4 gv = load_vec(p.g, (vb + (int64_t)tid * VEC) * Ty::BYTES);
      const uint4 cv = INJ ? inj_one<DT>(p, gv, vb + (int64_t)tid * VEC)
                           : load_vec(p.c, (vb + (int64_t)tid * VEC) * Ty::BYTES);
      uint32_t emax = 0, umax = 0;
#pragma unroll
      for (int j = 0; j < VEC; j++) {
        const uint32_t G = lane_bits<DT>(gv, j), C = lane_bits<DT>(cv, j);
        const uint32_t e = (G & Ty::MAG) >> Ty::MB;
        if (e < (uint32_t)Ty::EMAX && e > emax) emax = e;
        if (((G ^ C) & Ty::SIGN) == 0u && (G & Ty::MAG) < Ty::INF && (C & Ty::MAG) < Ty::INF) {
          const uint32_t u = G > C ? G - C : C - G;
          umax = u > umax ? u : umax;
        }
      }
      atomicMax(&sm.lb, (int)emax);
      atomicMax(&sm.ub, (int)(32 - __clz(umax)));
    }
    if (tid == 0) {
      constexpr long long NONE = 0x7FFFFFFFFFFFFFFFll;
      const bool fin = (G0 & Ty::MAG) < Ty::INF && (C0 & Ty::MAG) < Ty::INF;
      sm.ff = fin ? pb : NONE;
      sm.fu = fin ? pb : NONE;
    }
    __syncthreads();
    // the piece's initial window, the first entry of every warp's window log
    {
      const int lb0 = window_floor<DT>(sm.lb, sm.ub);
      set_window_lb<DT>(W, lb0);
      if (lane == 0) {
        sm.nwin[warp] = 0;
        sm.wstart[warp][0] = 0;
        sm.wlb[warp][0] = lb0;
      }
    }
    Thr T;
    thr_init(T);
    auto scalar_range = [&](int64_t b0, int64_t b1) {
      for (int64_t i = b0 + tid; i < b1; i += BLOCK) {
        const uint32_t G = load_scalar<DT>(p.g, i);
        do_scalar<DT>(L, T, G, cand_at<DT, INJ>(p, i, G), (uint32_t)(i - lo), W, sm);
      }
    };
    // scalar head: fewer than VEC elements, or the whole piece in scalar mode
    // (then in rounds of at most 65535 elements per thread)
    {
      const int64_t h_end = vb < pe ? vb : pe;
      constexpr int64_t ROUND_ELEMS = (int64_t)BLOCK * 65535;
      for (int64_t r0 = pb; r0 < h_end; r0 += ROUND_ELEMS) {
        const int64_t r1 = min(h_end, r0 + ROUND_ELEMS);
        scalar_range(r0, r1);
        if (r1 < h_end) fold_round<DT>(L, sm, win_lexp<DT>(W));
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
        if (!failed && PEAT_CHECK(k * CHV < nvec && vb + k * CHV * VEC - lo < ((int64_t)1 << 32))) {
          const int64_t v0 = k * CHV;
          const int nvalid = (int)min((int64_t)CHV, nvec - v0);
          if constexpr (INJ) {
            // the candidate tile, generated from the golden tile into the candidate ring
            inj_chunk<DT>(p, sm.ring_g[warp][st], sm.ring_c[warp][st], nvalid, vb + v0 * VEC);
            __syncwarp();
          }
          do_tile<DT>(L, T, sm.ring_g[warp][st], nvalid, (uint32_t)(vb + v0 * VEC - lo), W, (uint32_t)i, sm);
          if (lane == 0 && i + NSTAGE < my_chunks) issue(seq + NSTAGE, warp + NW * (i + NSTAGE));
        }
        seq++;
      }
      if (r1 < nchunk) fold_round<DT>(L, sm, win_lexp<DT>(W));
    }
    if (fail_i >= 0) {
      // copies this warp issued but never consumed: wait for them before the
      // staging memory is reused or the CTA exits
      for (int64_t j = fail_i; j < my_chunks && j < fail_i + NSTAGE; j++) {
        const uint32_t sq = fail_seq + (uint32_t)(j - fail_i);
        mbar_wait(&sm.bar[warp][sq % NSTAGE], (sq / NSTAGE) & 1u, DRAIN_LIMIT);
      }
    }
    // scalar tail (fewer than VEC elements), after the body
    if (vb < ve && ve < pe) scalar_range(ve, pe);
    finish_piece<DT, INJ>(L, W, sm, p, s, pb, pe, vb, ve);
    pb = pe;
  }
}

// ---------------------------------------------------------------------------
// stage 2: one CTA per segment: merge the maxima of the segment's pieces,
// round the exact sums once, write the outputs, clear the accumulator
// ---------------------------------------------------------------------------
// RN64 of the quotient (hi + lo) 2^sc / g > 0.  When hi + lo is a binary64
// number (always, unless lo is more than 29 binades below hi) the numerator
// is exact and one correctly rounded division gives the answer; otherwise the
// candidate with the smallest exact residual wins, ties to the even significand.
__device__ double rel_value(float hi, float lo, int sc, float g) {
  if (hi == 0.0f) return 0.0;
  if (g == 0.0f) return __longlong_as_double(0x7FF0000000000000ll);
  const double dh = hi, dl = lo;
  const double num = __dadd_rn(dh, dl);
  if (__dsub_rn(num, dh) == dl) return __ddiv_rn(sc ? num * 2.0 : num, (double)g);
  double q = __ddiv_rn(sc ? num * 2.0 : num, (double)g);  // within a few units of the exact quotient
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
    const bool qeven = (__double_as_longlong(q) & 1) == 0, beven = (__double_as_longlong(best) & 1) == 0;
    if (c < 0 || (c == 0 && qeven && !beven)) best = q, bres = r;
  }
  return best;
}


// Copy of a partial written by another CTA (read from L2, past this SM's L1).
__device__ __forceinline__ Partial load_partial(const Partial* src) {
  Partial x;
  const unsigned long long* w = reinterpret_cast<const unsigned long long*>(src);
  unsigned long long* d = reinterpret_cast<unsigned long long*>(&x);
#pragma unroll
  for (int k = 0; k < (int)(sizeof(Partial) / 8); k++) d[k] = __ldcg(w + k);
  return x;
}

// The whole CTA, once every piece of segment s is in: merge the pieces'
// maxima in CTA order, round the exact sums once, write the outputs and clear
// the accumulator for the next call.  Uses the CTA's totals in shared memory
// as scratch (they are zero on entry and on exit).
__device__ __noinline__ void finalize_segment(const CompareParams& p, int64_t s, FinScratch& f, MV& mv) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t s0 = p.offsets[s], s1 = p.offsets[s + 1];
  SegAcc* acc = p.acc + s;
  long long* limbs = f.limbs;
  unsigned long long hv = 0;
  if (tid < HBINS) {
    hv = __ldcg(&acc->hist[tid]);
    acc->hist[tid] = 0;
  }
  if (tid >= HBINS && tid < HBINS + 8) {
    f.cnt[tid - HBINS] = __ldcg(&acc->cnt[tid - HBINS]);
    acc->cnt[tid - HBINS] = 0;
  }
  if (tid >= 160 && tid < 160 + NSUM * NLIMB) {
    const int j = tid - 160;
    limbs[j] = __ldcg(&acc->limbs[0][0] + j);
    (&acc->limbs[0][0])[j] = 0;
  }
  if (tid == 0) acc->done = 0;
  // maxima over the segment's pieces
  Partial x;
  part_none(x);
  {
    const int b0 = cta_of_warp(s0, p), b1 = cta_of_warp(s1 - 1, p);
    for (int b = b0 + tid; b <= b1; b += BLOCK) part_merge(x, load_partial(p.partials + s + b));
  }
  part_warp_reduce(x);
  if (lane == 0) f.wbest[warp] = x;
  __syncthreads();
  if (warp == 1 && lane < NSUM) f.sums[lane] = limbs_to_double(limbs + lane * NLIMB);
  if (warp == 0) {
    if (lane < NW) x = f.wbest[lane];
    else part_none(x);
    part_warp_reduce(x);
  }
  if (tid == 64) carry_to_digits(limbs + 1 * NLIMB, NLIMB, mv.A);  // S1 = sum |d|
  if (tid == 96) carry_to_digits(limbs + 2 * NLIMB, NLIMB, mv.B);  // S2 = sum d^2
  // the mean and variance of |d| over the finite pairs (synchronises the block)
  mean_var_block(mv, (uint64_t)(s1 - s0) - f.cnt[3], LIMB_LSB);
  if (tid == 0) {
    const unsigned long long* cnt = f.cnt;
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
    r.sum_signed = f.sums[0];
    r.sum_abs = f.sums[1];
    r.sum_sq = f.sums[2];
    r.rtol_eff = p.rtol;
    r.atol_eff = p.atol;
    r.mean_abs = mv.mean;
    r.var_abs = mv.var;
    if (p.status && (*reinterpret_cast<volatile unsigned int*>(p.status) & 1u))
      r.argmax_abs = r.argmax_rel = r.argmax_ulp = -2;  // a bounded wait expired: the outputs are invalid
    p.stats[s] = r;
  }
  if (p.hist && tid < HBINS) p.hist[s * HBINS + tid] = hv + ((tid == 0 || tid == 64) ? f.cnt[0] : 0ull);
  __syncthreads();
}

// Segments of a multi-segment call, one CTA each, after stage 1.
__global__ void __launch_bounds__(BLOCK) compare_finalize(CompareParams p) {
  __shared__ FinScratch f;
  __shared__ MV mv;
  pdl_wait();  // stage 1 complete
  if (p.offsets[blockIdx.x] < p.offsets[blockIdx.x + 1]) finalize_segment(p, blockIdx.x, f, mv);
}

// The outputs of every empty segment (no pairs): zero counts and sums, argmax -1.
__device__ __noinline__ void write_empty_segments(const CompareParams& p) {
  for (int64_t s = threadIdx.x; s < p.nseg; s += BLOCK) {
    if (p.offsets[s] != p.offsets[s + 1]) continue;
    peat_stats_t r;
    memset(&r, 0, sizeof(r));
    r.argmax_abs = r.argmax_rel = r.argmax_ulp = -1;
    r.rtol_eff = p.rtol;
    r.atol_eff = p.atol;
    p.stats[s] = r;
    if (p.hist)
      for (int b = 0; b < HBINS; b++) p.hist[s * HBINS + b] = 0;
  }
}

template <int DT>
cudaError_t launch_t(const CompareParams& p, cudaStream_t st) {
  // NVTX ranges (host-side enqueue of each stage) for profilers; no cost without one attached
  nvtxRangePushA(p.inj_n > 0 ? "peat inject+compare stage 1" : "peat compare stage 1");
  if (p.inj_n > 0) compare_stage1<DT, true><<<p.nctas, BLOCK, sizeof(Smem), st>>>(p);
  else compare_stage1<DT, false><<<p.nctas, BLOCK, sizeof(Smem), st>>>(p);
  cudaError_t e = cudaGetLastError();
  nvtxRangePop();
  if (e == cudaSuccess && p.stage1_event) e = cudaEventRecord(static_cast<cudaEvent_t>(p.stage1_event), st);
  if (e != cudaSuccess || p.nseg <= 1) return e;
  nvtxRangePushA("peat compare stage 2 (per-segment finalize)");
  // a programmatic dependent of stage 1 (its launch overlaps the end of stage
  // 1), unless an event was recorded between the two
  if (p.stage1_event) {
    compare_finalize<<<(unsigned)p.nseg, BLOCK, 0, st>>>(p);
    e = cudaGetLastError();
  } else {
    e = launch_dependent(compare_finalize, (unsigned)p.nseg, BLOCK, 0, st, p);
  }
  nvtxRangePop();
  return e;
}

template <int DT>
__host__ __device__ int64_t bound_t(int64_t b, int nctas, int64_t n, int64_t p0) {
  if (b <= 0) return 0;
  if (b >= nctas) return n;
  constexpr int VEC = Tr<DT>::VEC;
  if (p0 < 0 || p0 >= n) return (n / nctas) * b + (n % nctas) * b / nctas;
  int64_t nv = (n - p0) / VEC;
  int64_t lo = p0 + ((nv / nctas) * b + (nv % nctas) * b / nctas) * VEC;
  return lo < n ? lo : n;
}

// offsets {0, n} and the CTA bounds of a one-tensor call, written on the
// device; a non-null status word is cleared for the compare that follows
template <int DT>
__global__ void compare_bounds(int64_t* offsets, int64_t* bounds, int nctas, int64_t n, int64_t p0,
                               unsigned int* status) {
  for (int b = threadIdx.x; b <= nctas; b += blockDim.x) bounds[b] = bound_t<DT>(b, nctas, n, p0);
  if (threadIdx.x == 0) {
    offsets[0] = 0;
    offsets[1] = n;
    if (status) *status = 0u;
  }
}

}  // namespace

cudaError_t launch_bounds_on_device(int dtype, int64_t* offsets, int64_t* bounds, int nctas, int64_t n, int64_t p0,
                                    unsigned int* status, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: compare_bounds<PEAT_F32><<<1, BLOCK, 0, s>>>(offsets, bounds, nctas, n, p0, status); break;
    case PEAT_F16: compare_bounds<PEAT_F16><<<1, BLOCK, 0, s>>>(offsets, bounds, nctas, n, p0, status); break;
    case PEAT_BF16: compare_bounds<PEAT_BF16><<<1, BLOCK, 0, s>>>(offsets, bounds, nctas, n, p0, status); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

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
template <int DT, bool INJ>
cudaError_t prepare_one() {
  cudaError_t e =
      cudaFuncSetAttribute(compare_stage1<DT, INJ>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(Smem));
  if (e == cudaSuccess)  // as much shared memory as the SM offers: CTAS_PER_SM CTAs of sizeof(Smem) each
    e = cudaFuncSetAttribute(compare_stage1<DT, INJ>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  return e;
}
template <int DT>
cudaError_t prepare_t() {
  cudaError_t e = prepare_one<DT, false>();
  return e == cudaSuccess ? prepare_one<DT, true>() : e;
}

cudaError_t compare_prepare() {
  cudaError_t e = prepare_t<PEAT_F32>();
  if (e == cudaSuccess) e = prepare_t<PEAT_F16>();
  if (e == cudaSuccess) e = prepare_t<PEAT_BF16>();
  return e;
}

int compare_ctas_per_sm() { return CTAS_PER_SM; }
size_t compare_partial_bytes() { return sizeof(Partial); }
size_t compare_segacc_bytes() { return sizeof(SegAcc); }

cudaError_t register_digit_status_compare(unsigned int* word) { return set_digit_status_here(word); }

// The index arithmetic of for_digits run on the host (a test of the digit
// split and of its range check; no GPU involved).
int test_for_digits(uint64_t m_lo, uint64_t m_hi, int e, int neg, int64_t* out) {
  for (int j = 0; j < NLIMB; j++) out[j] = 0;
  t_host_digit_dropped = false;
  for_digits(((unsigned __int128)m_hi << 64) | m_lo, e, neg != 0, [&](int j, int64_t v) { out[j] += v; });
  return t_host_digit_dropped ? 1 : 0;
}

// The binary64 rounding of the exact quotients behind the mean and the
// variance, run on the host (a test of quot_rn; no GPU involved).
double test_quot_rn(uint64_t w_hi, uint64_t w_lo, int sticky, int e, uint64_t d) {
  return quot_rn(((unsigned __int128)w_hi << 64) | w_lo, sticky != 0, e, d);
}

}  // namespace peat
