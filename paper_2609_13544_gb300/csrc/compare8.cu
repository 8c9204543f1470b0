// The error signature (Section IV-B-3: maximum, mean and variance of
// |c - g|, with the classes, ULP distances and histograms of the compare) for
// the two 8-bit formats of the OCP FP8 specification, E4M3 and E5M2 (the
// paper lists 8-bit precisions among those a kernel may run in).
//
// Every finite value of these formats is an integer multiple of 2^-S (S = 9
// for E4M3, 16 for E5M2) below 2^32 in units of 2^-S, so d = c - g is an exact
// 64-bit integer D in those units and |d|, d and d^2 accumulate exactly as
// integers (d^2 in 128 bits), and the tolerance test is one integer
// comparison against a bound per golden magnitude computed exactly on the host.  Work items are contiguous runs of one segment; each
// item's totals go to a record of its own, and one CTA per segment merges
// its items (integer sums, maxima by exact comparison with the lowest index
// on ties: the order of the merge does not matter).
#include <cstdint>
#include <type_traits>

#include "meanvar.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

constexpr int TB = 256, NW = TB / 32;

template <int DT>
struct F8;
template <>
struct F8<PEAT_F8E4M3> {
  static constexpr int S = 9, MB = 3;  // value = K 2^-9; 3 fraction bits, bias 7
};
template <>
struct F8<PEAT_F8E5M2> {
  static constexpr int S = 16, MB = 2;  // value = K 2^-16; 2 fraction bits, bias 15
};

// magnitude (7 bits): 0 finite, 1 infinite, 2 NaN
template <int DT>
__device__ __forceinline__ int f8_kind(uint32_t mag) {
  if constexpr (DT == PEAT_F8E4M3) return mag == 0x7Fu ? 2 : 0;
  else return mag < 0x7Cu ? 0 : (mag == 0x7Cu ? 1 : 2);
}
// |value| 2^S of a finite magnitude: subnormal m, normal (2^MB + m) 2^(e - 1)
template <int DT>
__device__ __forceinline__ uint32_t f8_units(uint32_t mag) {
  constexpr int MB = F8<DT>::MB;
  const uint32_t e = mag >> MB, m = mag & ((1u << MB) - 1u);
  return e == 0 ? m : ((m | (1u << MB)) << (e - 1));
}

using u128 = unsigned __int128;
using i128 = __int128;

// totals of a run of pairs
struct Tot {
  unsigned long long cnt[PEAT_NCLASS], nfin;
  u128 s1, s2;  // sum |D|, sum D^2
  i128 sd;      // sum D
  unsigned long long ma;  // max |D|, at index ia (-1: no finite pair)
  long long ia;
  unsigned long long ra, rb;  // max |D| / |G| as the fraction ra / rb (rb = 0: +inf), at ir
  long long ir;
  unsigned long long mu;  // max ULP distance, at iu (-1: none)
  long long iu;
};

__device__ __forceinline__ void tot_init(Tot& t) {
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] = 0;
  t.nfin = 0;
  t.s1 = 0;
  t.s2 = 0;
  t.sd = 0;
  t.ma = 0, t.ia = -1;
  t.ra = 0, t.rb = 1, t.ir = -1;
  t.mu = 0, t.iu = -1;
}

// x better than y: larger, or equal at a lower index; an absent record (index -1) is worst
__device__ __forceinline__ bool better_u(unsigned long long x, long long ix, unsigned long long y, long long iy) {
  if (ix < 0) return false;
  if (iy < 0) return true;
  return x > y || (x == y && ix < iy);
}
// compare xa/xb with ya/yb (b = 0: +inf; a = 0 always carries b = 1)
__device__ __forceinline__ int cmp_frac(unsigned long long xa, unsigned long long xb, unsigned long long ya,
                                        unsigned long long yb) {
  if (xb == 0 || yb == 0) return (xb == 0) - (yb == 0);
  const u128 l = (u128)xa * yb, r = (u128)ya * xb;
  return (l > r) - (l < r);
}
__device__ __forceinline__ bool better_rel(unsigned long long xa, unsigned long long xb, long long ix,
                                           unsigned long long ya, unsigned long long yb, long long iy) {
  if (ix < 0) return false;
  if (iy < 0) return true;
  const int c = cmp_frac(xa, xb, ya, yb);
  return c > 0 || (c == 0 && ix < iy);
}

__device__ __forceinline__ void tot_merge(Tot& t, const Tot& o) {
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] += o.cnt[k];
  t.nfin += o.nfin;
  t.s1 += o.s1;
  t.s2 += o.s2;
  t.sd += o.sd;
  if (better_u(o.ma, o.ia, t.ma, t.ia)) t.ma = o.ma, t.ia = o.ia;
  if (better_rel(o.ra, o.rb, o.ir, t.ra, t.rb, t.ir)) t.ra = o.ra, t.rb = o.rb, t.ir = o.ir;
  if (better_u(o.mu, o.iu, t.mu, t.iu)) t.mu = o.mu, t.iu = o.iu;
}

__device__ __forceinline__ u128 shfl_u128(u128 v, int off) {
  const unsigned long long lo = __shfl_down_sync(0xFFFFFFFFu, (unsigned long long)v, off);
  const unsigned long long hi = __shfl_down_sync(0xFFFFFFFFu, (unsigned long long)(v >> 64), off);
  return ((u128)hi << 64) | lo;
}
__device__ __forceinline__ void tot_shfl(Tot& o, const Tot& t, int off) {
  for (int k = 0; k < PEAT_NCLASS; k++) o.cnt[k] = __shfl_down_sync(0xFFFFFFFFu, t.cnt[k], off);
  o.nfin = __shfl_down_sync(0xFFFFFFFFu, t.nfin, off);
  o.s1 = shfl_u128(t.s1, off);
  o.s2 = shfl_u128(t.s2, off);
  o.sd = (i128)shfl_u128((u128)t.sd, off);
  o.ma = __shfl_down_sync(0xFFFFFFFFu, t.ma, off);
  o.ia = __shfl_down_sync(0xFFFFFFFFu, t.ia, off);
  o.ra = __shfl_down_sync(0xFFFFFFFFu, t.ra, off);
  o.rb = __shfl_down_sync(0xFFFFFFFFu, t.rb, off);
  o.ir = __shfl_down_sync(0xFFFFFFFFu, t.ir, off);
  o.mu = __shfl_down_sync(0xFFFFFFFFu, t.mu, off);
  o.iu = __shfl_down_sync(0xFFFFFFFFu, t.iu, off);
}

// the CTA's totals, complete in thread 0 (every thread calls it)
__device__ void block_total(Tot& t, Tot* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int off = 16; off > 0; off >>= 1) {
    Tot o;
    tot_shfl(o, t, off);
    tot_merge(t, o);
  }
  if (lane == 0) warp_tot[warp] = t;
  __syncthreads();
  if (threadIdx.x == 0)
    for (int w = 1; w < NW; w++) tot_merge(t, warp_tot[w]);
  __syncthreads();
}

// floor(log2(a / b)) for a, b >= 1
__device__ __forceinline__ int floor_log2_ratio(unsigned long long a, unsigned long long b) {
  const int ea = 63 - __clzll((long long)a), eb = 63 - __clzll((long long)b);
  return (ea - eb) - ((a << (63 - ea)) < (b << (63 - eb)) ? 1 : 0);
}

// add one to shared bin `bin` for every lane that has one (bin < 0: none), one atomic per distinct bin
__device__ __forceinline__ void hist_add(unsigned* H, int bin) {
  const unsigned grp = __match_any_sync(0xFFFFFFFFu, bin);
  if (bin >= 0 && (int)(threadIdx.x & 31) == __ffs(grp) - 1) atomicAdd(H + bin, (unsigned)__popc(grp));
}

// A thread's totals within one work item, in the narrowest exact types:
// |D| < 2^19 (E4M3) or 2^33 (E5M2), at most 2^14 pairs per thread and item.
// Offsets are positions in the item plus one (0: none); they only grow along a
// thread's pairs, so a strict comparison keeps the earliest on ties.
template <int DT>
struct Acc8 {
  using A = typename std::conditional<DT == PEAT_F8E4M3, uint32_t, unsigned long long>::type;
  uint32_t cnt[PEAT_NCLASS], nfin;
  unsigned long long s1, s2lo, s2hi;
  long long sd;
  A ma;
  uint32_t ia;
  A ra;
  uint32_t rb, ir;
  float rt;  // ra / rb in float32 lowered by 1e-5 (more than its error): a pair below it cannot win
  uint32_t mu, iu;
};

template <int DT>
__device__ __forceinline__ void acc_init(Acc8<DT>& t) {
#pragma unroll
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] = 0;
  t.nfin = 0;
  t.s1 = t.s2lo = t.s2hi = 0;
  t.sd = 0;
  t.ma = 0, t.ia = 0;
  t.ra = 0, t.rb = 1, t.ir = 0, t.rt = 0.0f;
  t.mu = 0, t.iu = 0;
}

template <int DT>
__device__ __forceinline__ float to_f(typename Acc8<DT>::A a) {
  if constexpr (DT == PEAT_F8E4M3) return __uint2float_rn(a);
  else return __fmaf_rn(__uint2float_rn((uint32_t)(a >> 32)), 4294967296.0f, __uint2float_rn((uint32_t)a));
}

// xa / xb > ya / yb exactly (xb, yb: |g| in units, 0 = the ratio is +inf; xa = 0 carries xb = 1)
template <int DT>
__device__ __forceinline__ bool frac_gt(typename Acc8<DT>::A xa, uint32_t xb, typename Acc8<DT>::A ya, uint32_t yb) {
  if (xb == 0 || yb == 0) return xb == 0 && yb != 0;
  if constexpr (DT == PEAT_F8E4M3) {
    return (unsigned long long)xa * yb > (unsigned long long)ya * xb;  // below 2^37
  } else {
    const u128 l = (u128)xa * yb, r = (u128)ya * xb;
    return l > r;
  }
}

// one pair slot of the warp (every lane calls it; ok: this lane holds the pair at item offset off;
// amax: the tolerance bound per golden magnitude)
template <int DT>
__device__ __forceinline__ void pair8(const unsigned long long* amax, Acc8<DT>& t, unsigned* H, uint32_t G,
                                      uint32_t C, bool ok, uint32_t off) {
  using A = typename Acc8<DT>::A;
  int relbin = -1, ulpbin = -1, cls = -1;
  if (ok) {
    const uint32_t mg = G & 0x7Fu, mc = C & 0x7Fu, sg = G >> 7, sc = C >> 7;
    const int kg = f8_kind<DT>(mg), kc = f8_kind<DT>(mc);
    const int keyg = sg ? -(int)mg : (int)mg, keyc = sc ? -(int)mc : (int)mc;
    const uint32_t u = (uint32_t)(keyc > keyg ? keyc - keyg : keyg - keyc);
    const bool nan = kg == 2 || kc == 2;
    if (kg | kc) {
      const bool eq = (kg == 2 && kc == 2) || (kg == 1 && kc == 1 && sg == sc);
      cls = eq ? PEAT_EXACT : PEAT_NAN_INF_ASYM;
      relbin = eq ? 0 : 63;
    } else {
      const uint32_t Kg = f8_units<DT>(mg), Kc = f8_units<DT>(mc);
      A a;
      long long D;
      if constexpr (DT == PEAT_F8E4M3) {
        const int d = (sc ? -(int)Kc : (int)Kc) - (sg ? -(int)Kg : (int)Kg);
        D = d;
        a = (uint32_t)(d < 0 ? -d : d);
        t.s2lo += (unsigned long long)a * a;
      } else {
        D = (sc ? -(long long)Kc : (long long)Kc) - (sg ? -(long long)Kg : (long long)Kg);
        a = (unsigned long long)(D < 0 ? -D : D);
        const unsigned long long lo = a * a, hi = __umul64hi(a, a);
        t.s2lo += lo;
        t.s2hi += hi + (t.s2lo < lo ? 1ull : 0ull);
      }
      t.nfin++;
      t.s1 += a;
      t.sd += D;
      if (a > t.ma || t.ia == 0) t.ma = a, t.ia = off + 1;
      // the relative maximum: one float32 multiply rules out all but the candidates
      const uint32_t rb = a == 0 ? 1u : Kg;
      if (t.ir == 0 || to_f<DT>(a) >= __fmul_rn(t.rt, __uint2float_rn(rb))) {
        if (t.ir == 0 || frac_gt<DT>(a, rb, t.ra, t.rb)) {
          t.ra = a, t.rb = rb, t.ir = off + 1;
          t.rt = rb == 0 ? __int_as_float(0x7F800000)
                         : __fmul_rn(__fdiv_rn(to_f<DT>(a), __uint2float_rn(rb)), 0.99999f);
        }
      }
      if (a == 0) {
        cls = PEAT_EXACT;
        relbin = 0;
      } else {
        if ((unsigned long long)a <= amax[mg]) cls = PEAT_WITHIN_TOL;
        else if (Kg != 0 && Kc != 0 && sg != sc) cls = PEAT_SIGN_FLIP;
        else cls = PEAT_MISMATCH;
        if (Kg == 0) {
          relbin = 63;
        } else {
          const int k = floor_log2_ratio((unsigned long long)a, Kg) + 48;
          relbin = k < 1 ? 1 : (k > 62 ? 62 : k);
        }
      }
    }
    if (nan) {
      ulpbin = (kg == 2 && kc == 2) ? 0 : 63;  // no ULP distance with a NaN
    } else {
      ulpbin = (int)(u < 63 ? u : 63);
      if (u > t.mu || t.iu == 0) t.mu = u, t.iu = off + 1;
    }
  }
#pragma unroll
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] += cls == k;
  hist_add(H, relbin);
  hist_add(H, ulpbin < 0 ? -1 : 64 + ulpbin);
}

// a thread's item totals as segment totals (item starts at segment position ib)
template <int DT>
__device__ __forceinline__ void acc_to_tot(Tot& t, const Acc8<DT>& a, long long ib) {
#pragma unroll
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] = a.cnt[k];
  t.nfin = a.nfin;
  t.s1 = a.s1;
  t.s2 = ((u128)a.s2hi << 64) | a.s2lo;
  t.sd = a.sd;
  t.ma = a.ma, t.ia = a.ia ? ib + a.ia - 1 : -1;
  t.ra = a.ra, t.rb = a.rb, t.ir = a.ir ? ib + a.ir - 1 : -1;
  t.mu = a.mu, t.iu = a.iu ? ib + a.iu - 1 : -1;
}

__device__ __forceinline__ void store_tot(Part8* d, const Tot& t) {
  for (int k = 0; k < PEAT_NCLASS; k++) d->cnt[k] = t.cnt[k];
  d->nfin = t.nfin;
  d->s1lo = (unsigned long long)t.s1, d->s1hi = (unsigned long long)(t.s1 >> 64);
  d->s2lo = (unsigned long long)t.s2, d->s2hi = (unsigned long long)(t.s2 >> 64);
  d->sdlo = (unsigned long long)(u128)t.sd, d->sdhi = (unsigned long long)((u128)t.sd >> 64);
  d->ma = t.ma, d->ia = t.ia;
  d->ra = t.ra, d->rb = t.rb, d->ir = t.ir;
  d->mu = t.mu, d->iu = t.iu;
}
__device__ __forceinline__ void load_tot(Tot& t, const Part8* d) {
  for (int k = 0; k < PEAT_NCLASS; k++) t.cnt[k] = d->cnt[k];
  t.nfin = d->nfin;
  t.s1 = ((u128)d->s1hi << 64) | d->s1lo;
  t.s2 = ((u128)d->s2hi << 64) | d->s2lo;
  t.sd = (i128)(((u128)d->sdhi << 64) | d->sdlo);
  t.ma = d->ma, t.ia = d->ia;
  t.ra = d->ra, t.rb = d->rb, t.ir = d->ir;
  t.mu = d->mu, t.iu = d->iu;
}

template <int DT>
__global__ void __launch_bounds__(TB) compare8_stage1(Cmp8Params p) {
  __shared__ unsigned H[PEAT_HIST_BINS];
  __shared__ Tot warp_tot[NW];
  __shared__ unsigned long long AM[128];
  pdl_trigger();  // the finalize kernel may start launching (it waits for this grid)
  const int lane = threadIdx.x & 31;
  for (int k = threadIdx.x; k < 128; k += TB) AM[k] = p.amax[k];
  for (long long item = blockIdx.x; item < p.nitems; item += gridDim.x) {
    const long long b = p.item_b[item], e = p.item_e[item], seg = p.item_seg[item];
    const long long base = p.offsets[seg];  // indices are reported within the segment
    for (int k = threadIdx.x; k < PEAT_HIST_BINS; k += TB) H[k] = 0u;
    __syncthreads();
    Acc8<DT> acc;
    acc_init(acc);
    uint32_t nsame = 0;  // pairs of the equal-group fast path (rel and ULP bin 0)
    // groups of 16 elements on the absolute index grid, whole warps in every round
    const long long q0 = b >> 4, q1 = (e + 15) >> 4;
    for (long long q = q0 + threadIdx.x; __any_sync(0xFFFFFFFFu, q < q1); q += TB) {
      const bool okq = q < q1;
      const long long i0 = q << 4;
      uint32_t w[4] = {0u, 0u, 0u, 0u}, x[4] = {0u, 0u, 0u, 0u};
      if (okq && p.vec && i0 >= b && i0 + 16 <= e) {
        const uint4 gv = __ldg(reinterpret_cast<const uint4*>(p.g) + q);
        const uint4 cv = __ldg(reinterpret_cast<const uint4*>(p.c) + q);
        w[0] = gv.x, w[1] = gv.y, w[2] = gv.z, w[3] = gv.w;
        x[0] = cv.x, x[1] = cv.y, x[2] = cv.z, x[3] = cv.w;
      } else if (okq) {
#pragma unroll
        for (int j = 0; j < 16; j++) {
          const long long i = i0 + j;
          if (i >= b && i < e) {
            w[j >> 2] |= (uint32_t)__ldg(reinterpret_cast<const unsigned char*>(p.g) + i) << (8 * (j & 3));
            x[j >> 2] |= (uint32_t)__ldg(reinterpret_cast<const unsigned char*>(p.c) + i) << (8 * (j & 3));
          }
        }
      }
      // a warp slot of bitwise-equal, finite whole groups (decided for the whole warp):
      // 16 EXACT pairs per lane with |d| = 0 and u = 0
      bool fast = !okq;
      if (okq && p.vec && i0 >= b && i0 + 16 <= e && w[0] == x[0] && w[1] == x[1] && w[2] == x[2] && w[3] == x[3]) {
        bool fin = true;
#pragma unroll
        for (int j = 0; j < 16; j++) fin &= f8_kind<DT>((w[j >> 2] >> (8 * (j & 3))) & 0x7Fu) == 0;
        fast = fin;
      }
      if (__all_sync(0xFFFFFFFFu, fast)) {
        if (okq) {
          const uint32_t off = (uint32_t)(i0 - b);
          acc.cnt[PEAT_EXACT] += 16;
          acc.nfin += 16;
          if (acc.ia == 0) acc.ma = 0, acc.ia = off + 1;
          if (acc.ir == 0) acc.ra = 0, acc.rb = 1, acc.ir = off + 1, acc.rt = 0.0f;
          if (acc.iu == 0) acc.mu = 0, acc.iu = off + 1;
          nsame += 16;
        }
        continue;
      }
      // one copy of the pair code: the loop stays rolled (the body is long)
#pragma unroll 1
      for (int j = 0; j < 16; j++) {
        const long long i = i0 + j;
        const bool ok = okq && i >= b && i < e;
        const uint32_t gw = j < 8 ? (j < 4 ? w[0] : w[1]) : (j < 12 ? w[2] : w[3]);
        const uint32_t cw = j < 8 ? (j < 4 ? x[0] : x[1]) : (j < 12 ? x[2] : x[3]);
        pair8<DT>(AM, acc, H, (gw >> (8 * (j & 3))) & 0xFFu, (cw >> (8 * (j & 3))) & 0xFFu, ok, (uint32_t)(i - b));
      }
    }
    {
      const uint32_t ns = __reduce_add_sync(0xFFFFFFFFu, nsame);
      if (lane == 0 && ns) {
        atomicAdd(&H[0], ns);
        atomicAdd(&H[64], ns);
      }
    }
    Tot t;
    acc_to_tot<DT>(t, acc, b - base);
    block_total(t, warp_tot);
    if (threadIdx.x == 0) store_tot(p.parts + item, t);
    if (p.hist)
      for (int k = threadIdx.x; k < PEAT_HIST_BINS; k += TB)
        if (H[k]) atomicAdd(p.hist + seg * PEAT_HIST_BINS + k, (unsigned long long)H[k]);
    __syncthreads();
  }
}

// RN64 of a 128-bit magnitude
__device__ double u128_to_double(u128 x) {
  const unsigned long long hi = (unsigned long long)(x >> 64);
  if (hi == 0) return __ull2double_rn((unsigned long long)x);
  const int sh = __clzll((long long)hi);
  const u128 y = x << sh;
  // the top 64 bits, with every lower bit folded into a sticky bit below the rounding position
  const unsigned long long top = (unsigned long long)(y >> 64) | ((unsigned long long)y != 0 ? 1ull : 0ull);
  return ldexp(__ull2double_rn(top), 64 - sh);
}

template <int DT>
__global__ void __launch_bounds__(TB) compare8_finalize(Cmp8Params p) {
  __shared__ Tot warp_tot[NW];
  // S1 = s1 2^-S and S2 = s2 2^-2S: four digits each, no shift between them
  __shared__ MeanVarScratch<4, 4, 0> mv;
  __shared__ unsigned long long nfin;
  pdl_wait();  // stage 1 complete
  constexpr int S = F8<DT>::S;
  const long long seg = blockIdx.x;
  Tot t;
  tot_init(t);
  for (long long it = p.seg_first[seg] + threadIdx.x; it < p.seg_first[seg + 1]; it += TB) {
    Tot o;
    load_tot(o, p.parts + it);
    tot_merge(t, o);
  }
  block_total(t, warp_tot);
  if (threadIdx.x == 0) {
    for (int j = 0; j < 4; j++) {
      mv.A[j] = (uint32_t)(t.s1 >> (32 * j));
      mv.B[j] = (uint32_t)(t.s2 >> (32 * j));
    }
    nfin = t.nfin;
  }
  __syncthreads();
  mean_var_block(mv, nfin, -S);
  if (threadIdx.x != 0) return;
  peat_stats_t r;
  r.n = (uint64_t)(p.offsets[seg + 1] - p.offsets[seg]);
  for (int k = 0; k < PEAT_NCLASS; k++) r.count[k] = t.cnt[k];
  r.n_finite = t.nfin;
  r.max_abs = t.ia >= 0 ? ldexp((double)t.ma, -S) : 0.0;
  r.argmax_abs = t.ia;
  if (t.ir < 0 || t.ra == 0) r.max_rel = 0.0;
  else if (t.rb == 0) r.max_rel = __longlong_as_double(0x7FF0000000000000ll);
  else r.max_rel = __ddiv_rn((double)t.ra, (double)t.rb);  // both exact in binary64: one rounding
  r.argmax_rel = t.ir;
  r.max_ulp = t.iu >= 0 ? t.mu : 0;
  r.argmax_ulp = t.iu;
  r.sum_abs = ldexp(u128_to_double(t.s1), -S);
  r.sum_sq = ldexp(u128_to_double(t.s2), -2 * S);
  const double sdm = ldexp(u128_to_double(t.sd < 0 ? (u128)(-t.sd) : (u128)t.sd), -S);
  r.sum_signed = t.sd < 0 ? -sdm : sdm;
  r.rtol_eff = (double)p.rtol;
  r.atol_eff = (double)p.atol;
  r.mean_abs = mv.mean;
  r.var_abs = mv.var;
  p.stats[seg] = r;
}

template <int DT>
cudaError_t launch_t(const Cmp8Params& p, int nctas, cudaStream_t s) {
  if (p.nitems == 0) {
    compare8_finalize<DT><<<(unsigned)p.nseg, TB, 0, s>>>(p);
    return cudaGetLastError();
  }
  compare8_stage1<DT><<<nctas, TB, 0, s>>>(p);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_dependent(compare8_finalize<DT>, (unsigned)p.nseg, TB, 0, s, p);  // overlaps stage 1's end
}

}  // namespace

cudaError_t launch_compare8(int dtype, const Cmp8Params& p, int nctas, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F8E4M3: return launch_t<PEAT_F8E4M3>(p, nctas, s);
    case PEAT_F8E5M2: return launch_t<PEAT_F8E5M2>(p, nctas, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace peat
