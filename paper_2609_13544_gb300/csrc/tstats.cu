// Context statistics of recorded tensors (Section IV-C-2, "Rank-based
// Error-Data Correlation": the means and variances of the weight and
// activation tensors the error scores are correlated with), per tensor or per
// segment of a packed tensor list: counts of finite, NaN and infinite
// elements, the exact sum and sum of squares of the finite elements, their
// mean and population variance (each the exact value rounded once to
// nearest-even binary64), and the finite minimum and maximum.
//
// Stage 1 (tstats_stage1): CTA b owns the contiguous element range
// [bounds[b], bounds[b+1]) and walks the segments it meets.  A finite element
// x = +-m 2^(e-150) (m < 2^24, e the biased float32 exponent, 1 for
// subnormals) inside its warp's window e - Lb in [0, WSPAN] adds m << (e - Lb)
// to one of two 128-bit integers (by sign) and m^2 << 2(e - Lb) to a third;
// the window follows the data (placed 6 binades above the largest exponent a
// warp tile holds, moved when a tile leaves it), elements outside it go to
// fixed-point digits in shared memory.  At the end of a piece the integers
// become digits too, and the CTA adds its digits, counts and min/max keys to
// the segment's accumulator with atomics.
// Stage 2 (tstats_finalize, one CTA per segment): mean = S1 / n_f and
// variance = (n_f S2 - S1^2) / n_f^2, both from the exact digits with one
// rounding each; the accumulator is cleared for the next call.
#include <cuda_fp16.h>

#include <cstdint>

#include "exact.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

constexpr int TB = 256;
constexpr int WHEAD = 6;  // binades of a window above the largest exponent of the tile that placed it
constexpr int LB_UNSET = -1000;

// Per element type, decoded from the raw bits: an element is +-m 2^(ee - BM)
// with m below 2^(MB + 1) (the implicit bit for a normal value) and ee the
// exponent field (1 for subnormals); EINF marks infinities and NaNs.  A
// warp's window covers ee - Lb in [0, WSPAN].  Terms: t = m << (ee - Lb) and
// t^2.  16-bit types: t < 2^28, t^2 < 2^56 (one 32 x 32 -> 64 multiply), the
// signed sum of t in 64 bits and of t^2 in 128; float32: t < 2^54, t^2 <
// 2^108, both sums in 128 bits (by sign for t).  FLUSH in-window elements per
// lane at most between two flushes of the sums into digits.
template <int DT>
struct TS;
template <>
struct TS<PEAT_F32> {
  static constexpr int BYTES = 4, VEC = 4, BITS = 32, MB = 23, BM = 150, WSPAN = 30;
  static constexpr uint32_t EMASK = 0xFFu, EINF = 0xFFu, FLUSH = 1u << 18;
};
template <>
struct TS<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8, BITS = 16, MB = 10, BM = 25, WSPAN = 16;
  static constexpr uint32_t EMASK = 0x1Fu, EINF = 0x1Fu, FLUSH = 1u << 20;
};
template <>
struct TS<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8, BITS = 16, MB = 7, BM = 134;
  static constexpr uint32_t EMASK = 0xFFu, EINF = 0xFFu;
};

template <int DT>
__device__ __forceinline__ uint32_t ts_lane(const uint4& v, int j) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (TS<DT>::BYTES == 4) return w[j];
  else return (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
}

template <int DT>
__device__ __forceinline__ uint32_t ts_load(const void* base, int64_t i) {
  if constexpr (TS<DT>::BYTES == 4) return __ldg(reinterpret_cast<const uint32_t*>(base) + i);
  else return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(base) + i);
}

__device__ __forceinline__ uint4 ts_vec(const void* base, int64_t byte_off) {
  const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(base) + byte_off);
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(q));
  return v;
}

// raw bits -> an unsigned key in the order of the values (-0 below +0)
template <int DT>
__device__ __forceinline__ uint32_t raw_key(uint32_t r) {
  constexpr uint32_t SIGN = 1u << (TS<DT>::BITS - 1), ALL = TS<DT>::BITS == 32 ? 0xFFFFFFFFu : 0xFFFFu;
  return (r & SIGN) ? (~r & ALL) : (r | SIGN);
}
// the float32 bits of a raw element
template <int DT>
__device__ __forceinline__ uint32_t raw_to_f32(uint32_t r) {
  if constexpr (DT == PEAT_F32) return r;
  else if constexpr (DT == PEAT_BF16) return r << 16;
  else return __float_as_uint(__half2float(__ushort_as_half((unsigned short)r)));
}
template <int DT>
__device__ __forceinline__ uint32_t key_to_raw(uint32_t k) {
  constexpr uint32_t SIGN = 1u << (TS<DT>::BITS - 1), ALL = TS<DT>::BITS == 32 ? 0xFFFFFFFFu : 0xFFFFu;
  return (k & SIGN) ? (k & ~SIGN) : (~k & ALL);
}
// float32 bits -> an unsigned key in the order of the values
__device__ __forceinline__ uint32_t order_key(uint32_t b) { return (b & 0x80000000u) ? ~b : (b | 0x80000000u); }

__device__ __forceinline__ void lim_add(long long* lim, int j, int64_t v) {
  atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v);
}

// one lane's running totals
template <int DT>
struct TsLane {
  unsigned __int128 s1p = 0, s1n = 0;  // float32: sum of t by sign
  int64_t s1 = 0;                      // 16-bit types: signed sum of t
  unsigned __int128 s2 = 0;            // sum of t^2
  // 16-bit types, within one round of at most 32 elements per lane (terms
  // below 2^28 and 2^56): the sums as 64-bit multiply-adds, folded into s1
  // and s2 after every round
  uint64_t r1p = 0, r1n = 0, r2 = 0;
  uint32_t nnan = 0, ninf = 0, since = 0, slow = 0;
  uint32_t kmin = 0xFFFFFFFFu, kmax = 0;  // raw-order keys
};

__device__ __forceinline__ uint64_t wsum_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
__device__ __forceinline__ int64_t wsum_i64(int64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

// a round's 64-bit partial sums into the lane's totals (16-bit types)
template <int DT>
__device__ __forceinline__ void ts_fold(TsLane<DT>& L) {
  if constexpr (TS<DT>::BYTES == 2) {
    L.s1 += (int64_t)L.r1p - (int64_t)L.r1n;
    L.s2 += L.r2;
    L.r1p = L.r1n = L.r2 = 0;
  }
}

// The warp's integers into the CTA's digits (lim: S1, lim + NLIMB: S2), by
// all lanes of the warp together (lb is the same in every lane): each
// 128-bit sum is cut into 32-bit words, the words are summed over the warp
// in 64 bits, and lane 0 adds the totals as digits.
template <int DT>
__device__ __forceinline__ void ts_flush(TsLane<DT>& L, int lb, long long* lim) {
  if (lb != LB_UNSET) {
    const int u = lb - TS<DT>::BM;  // weight of a unit of t
    // S1 as a signed 128-bit value (|S1| < 2^73 per lane), S2 unsigned
    unsigned __int128 s1;
    if constexpr (TS<DT>::BYTES == 4) s1 = L.s1p - L.s1n;
    else s1 = (unsigned __int128)(__int128)L.s1;
    int64_t w1[4];
    uint64_t w2[4];
#pragma unroll
    for (int k = 0; k < 4; k++) {
      const uint32_t a = (uint32_t)(s1 >> (32 * k)), b2 = (uint32_t)(L.s2 >> (32 * k));
      w1[k] = wsum_i64(k == 3 ? (int64_t)(int32_t)a : (int64_t)a);  // the top word carries the sign
      w2[k] = wsum_u64(b2);
    }
    if ((threadIdx.x & 31) == 0) {
#pragma unroll
      for (int k = 0; k < 4; k++) {
        if (w1[k]) {
          const bool neg = w1[k] < 0;
          for_digits((uint64_t)(neg ? -w1[k] : w1[k]), u + 32 * k, neg, [&](int j, int64_t v) { lim_add(lim, j, v); });
        }
        if (w2[k]) for_digits(w2[k], 2 * u + 32 * k, false, [&](int j, int64_t v) { lim_add(lim + NLIMB, j, v); });
      }
    }
  }
  L.s1p = L.s1n = L.s2 = 0;
  L.s1 = 0;
  L.since = 0;
}

// an element outside the warp's window: its digits straight into the CTA's
// accumulator (out of line: rare, and the unrolled loop stays small enough
// for the instruction cache)
template <int DT>
__device__ __noinline__ void ts_slow(uint32_t m, int ee, bool neg, long long* lim) {
  const int ex = ee - TS<DT>::BM;  // |x| = m 2^ex
  for_digits(m, ex, neg, [&](int j, int64_t v) { lim_add(lim, j, v); });
  for_digits((uint64_t)m * m, 2 * ex, false, [&](int j, int64_t v) { lim_add(lim + NLIMB, j, v); });
}

template <int DT>
__device__ __forceinline__ void ts_elem(TsLane<DT>& L, uint32_t r, int lb, long long* lim) {
  using T = TS<DT>;
  const uint32_t e = (r >> T::MB) & T::EMASK, mant = r & ((1u << T::MB) - 1u);
  const bool neg = (r >> (T::BITS - 1)) & 1u;
  if (e == T::EINF) {
    if (mant) L.nnan++;
    else L.ninf++;
    return;
  }
  const uint32_t k = raw_key<DT>(r);
  L.kmin = min(L.kmin, k);
  L.kmax = max(L.kmax, k);
  const uint32_t m = mant | (e ? (1u << T::MB) : 0u);
  const int ee = e ? (int)e : 1, s = ee - lb;
  if ((unsigned)s <= (unsigned)T::WSPAN) {
    if constexpr (T::BYTES == 4) {
      const uint64_t t = (uint64_t)m << s;  // below 2^54
      if (neg) L.s1n += t;
      else L.s1p += t;
      L.s2 += ((unsigned __int128)__umul64hi(t, t) << 64) | (t * t);
    } else {
      // multiply-adds (the FMA pipe) rather than shifts and carries (ALU)
      const uint32_t t = m << s, ng = r >> 15;  // t below 2^28
      L.r1n += (uint64_t)t * ng;
      L.r1p += (uint64_t)t * (1u - ng);
      L.r2 += (uint64_t)t * t;  // below 2^56
    }
  } else if (m != 0) {
    ts_slow<DT>(m, ee, neg, lim);
    L.slow++;
  }
}

// largest exponent field of a vector's finite elements (0 if none)
template <int DT>
__device__ __forceinline__ int vec_emax(const uint4& v) {
  int em = 0;
#pragma unroll
  for (int j = 0; j < TS<DT>::VEC; j++) {
    const int e = (int)((ts_lane<DT>(v, j) >> TS<DT>::MB) & TS<DT>::EMASK);
    em = max(em, e == (int)TS<DT>::EINF ? 0 : e);
  }
  return em;
}

// one piece [a, b) of segment seg, inside this CTA's range
template <int DT>
__device__ void ts_piece(const TsParams& p, int64_t a, int64_t b, long long* lim, int& lb, TsLane<DT>& L) {
  constexpr int VEC = TS<DT>::VEC, B = TS<DT>::BYTES;
  const int lane = threadIdx.x & 31;
  // the vector grid inside the piece
  int64_t a0 = b, nv = 0;
  if (p.p0 >= 0 && p.p0 < p.n_total) {
    a0 = a <= p.p0 ? p.p0 : p.p0 + ((a - p.p0 + VEC - 1) / VEC) * VEC;
    if (a0 < b) nv = (b - a0) / VEC;
    else a0 = b;
  }
  // whole-CTA rounds of U TB vectors (U loads per thread in flight before any
  // is used), so every lane of a warp takes every round
  constexpr int U = 4;
  for (int64_t k0 = 0; k0 < nv; k0 += (int64_t)U * TB) {
    uint4 v[U];
    bool ok[U];
#pragma unroll
    for (int uu = 0; uu < U; uu++) {
      const int64_t k = k0 + uu * TB + threadIdx.x;
      ok[uu] = k < nv;
      v[uu] = ok[uu] ? ts_vec(p.x, (a0 + k * VEC) * B) : make_uint4(0, 0, 0, 0);
    }
    // place the warp's window on its first tile, and move it when a round
    // sent more than an eighth of the warp's elements to the digit path
    const uint32_t slow = __reduce_add_sync(0xFFFFFFFFu, L.slow);
    if (lb == LB_UNSET || slow > 32u * U * VEC / 8u) {
      int e = 0;
#pragma unroll
      for (int uu = 0; uu < U; uu++) e = max(e, ok[uu] ? vec_emax<DT>(v[uu]) : 0);
      const int em = __reduce_max_sync(0xFFFFFFFFu, e);
      if (em > 0) {
        ts_flush<DT>(L, lb, lim);
        lb = em + WHEAD - TS<DT>::WSPAN;
      }
    }
    L.slow = 0;
    // a flush before the next U VEC elements could pass FLUSH
    if (__any_sync(0xFFFFFFFFu, L.since > TS<DT>::FLUSH - U * VEC)) ts_flush<DT>(L, lb, lim);
#pragma unroll
    for (int uu = 0; uu < U; uu++) {
      if (ok[uu]) {
#pragma unroll
        for (int j = 0; j < VEC; j++) ts_elem<DT>(L, ts_lane<DT>(v[uu], j), lb, lim);
        L.since += VEC;
      }
    }
    ts_fold<DT>(L);
  }
  // the elements outside the vector grid: [a, a0) and [a0 + nv VEC, b), in
  // whole-CTA rounds as well
  const int64_t h = a0 - a, t0 = a0 + nv * VEC, ns = h + (b - t0);
  for (int64_t i0 = 0; i0 < ns; i0 += TB) {
    const int64_t i = i0 + threadIdx.x;
    const bool ok = i < ns;
    const uint32_t r = ok ? ts_load<DT>(p.x, i < h ? a + i : t0 + (i - h)) : 0u;
    const uint32_t slow = __reduce_add_sync(0xFFFFFFFFu, L.slow);
    if (lb == LB_UNSET || slow > 4u) {
      const int ef = (int)((r >> TS<DT>::MB) & TS<DT>::EMASK);
      const int em = __reduce_max_sync(0xFFFFFFFFu, ef == (int)TS<DT>::EINF ? 0 : ef);
      if (em > 0) {
        ts_flush<DT>(L, lb, lim);
        lb = em + WHEAD - TS<DT>::WSPAN;
      }
    }
    L.slow = 0;
    if (__any_sync(0xFFFFFFFFu, L.since >= TS<DT>::FLUSH)) ts_flush<DT>(L, lb, lim);
    if (ok) {
      ts_elem<DT>(L, r, lb, lim);
      L.since++;
    }
    ts_fold<DT>(L);
  }
  (void)lane;
}

template <int DT>
__global__ void __launch_bounds__(TB) tstats_stage1(TsParams p) {
  __shared__ long long lim[2 * NLIMB];
  __shared__ unsigned long long cnt[3];
  __shared__ unsigned int kmin_s, kmax_s;
  pdl_trigger();  // the finalize kernel may start launching (it waits for this grid)
  const int64_t lo = p.bounds[blockIdx.x], hi = p.bounds[blockIdx.x + 1];
  if (lo >= hi) return;
  // the segment holding lo: the last s with offsets[s] <= lo (empty segments skipped)
  int64_t s0 = 0, s1 = p.nseg;
  while (s1 - s0 > 1) {
    const int64_t mid = (s0 + s1) / 2;
    if (p.offsets[mid] <= lo) s0 = mid;
    else s1 = mid;
  }
  int64_t seg = s0;
  while (p.offsets[seg + 1] <= lo) seg++;
  int lb = LB_UNSET;
  for (int64_t a = lo; a < hi;) {
    const int64_t b = min(hi, p.offsets[seg + 1]);
    for (int j = threadIdx.x; j < 2 * NLIMB; j += TB) lim[j] = 0;
    if (threadIdx.x < 3) cnt[threadIdx.x] = 0;
    if (threadIdx.x == 0) {
      kmin_s = 0xFFFFFFFFu;
      kmax_s = 0;
    }
    __syncthreads();
    TsLane<DT> L;
    ts_piece<DT>(p, a, b, lim, lb, L);
    ts_flush<DT>(L, lb, lim);
    // finite = the piece's elements less the NaN and infinite ones
    const uint32_t nn = __reduce_add_sync(0xFFFFFFFFu, L.nnan), ni = __reduce_add_sync(0xFFFFFFFFu, L.ninf);
    // the lanes' extremes as float32 order keys (a lane with no finite element keeps neutral keys)
    const bool any = L.kmin != 0xFFFFFFFFu;
    const uint32_t kmn = __reduce_min_sync(0xFFFFFFFFu, any ? order_key(raw_to_f32<DT>(key_to_raw<DT>(L.kmin))) : 0xFFFFFFFFu),
                   kmx = __reduce_max_sync(0xFFFFFFFFu, any ? order_key(raw_to_f32<DT>(key_to_raw<DT>(L.kmax))) : 0u);
    if (threadIdx.x == 0) cnt[0] = (unsigned long long)(b - a);
    if ((threadIdx.x & 31) == 0) {
      if (nn) atomicAdd(&cnt[1], (unsigned long long)nn);
      if (ni) atomicAdd(&cnt[2], (unsigned long long)ni);
      atomicMin(&kmin_s, kmn);
      atomicMax(&kmax_s, kmx);
    }
    __syncthreads();
    TsAcc& acc = p.acc[seg];
    for (int j = threadIdx.x; j < 2 * NLIMB; j += TB)
      if (lim[j]) atomicAdd(reinterpret_cast<unsigned long long*>(&acc.limbs[0][0] + j), (unsigned long long)lim[j]);
    if (threadIdx.x == 0) {
      cnt[0] -= cnt[1] + cnt[2];
      if (cnt[0]) atomicAdd(&acc.nfin, cnt[0]);
      if (cnt[1]) atomicAdd(&acc.nnan, cnt[1]);
      if (cnt[2]) atomicAdd(&acc.ninf, cnt[2]);
      if (cnt[0]) {
        atomicMax(&acc.kmin_inv, ~kmin_s);
        atomicMax(&acc.kmax, kmax_s);
      }
    }
    __syncthreads();
    a = b;
    while (seg < p.nseg && p.offsets[seg + 1] <= a) seg++;
  }
}

// ---- stage 1 for bf16 elements: a histogram of bit patterns ----
// A 16-bit element has few values.  Per piece, the CTA places one window of
// WS exponents (from the largest finite exponent among the first vector of
// every thread, plus one binade of headroom) and counts every finite nonzero
// element inside it in a shared histogram indexed by (sign, exponent - Lb,
// significand field): one shared atomic per element, no per-element sums,
// keys or branches beyond the window test.  Zeros have two bins of their
// own; NaN, infinities, subnormals and elements outside the window go to the
// thread's slot (h16_slow below) or, further out, to the digits.  At the end
// of the piece each bin adds count * value and count * value^2 exactly
// (integers in units of the window's floor), and the extreme nonzero bins
// give the finite minimum and maximum.
template <int DT>
struct H16;
template <>
struct H16<PEAT_BF16> {
  static constexpr int WSB = 5, WS = 1 << WSB;  // 32 exponents: 8,192 bins
};
template <int DT>
constexpr int h16_bins() {
  return 2 * H16<DT>::WS << TS<DT>::MB;
}

// One thread's share of the nonzero elements the histogram does not take,
// in the thread's own shared-memory slot (no atomics, so a tensor whose bulk
// lies outside the window does not serialise on a few addresses): NaN and
// infinity counts, the extreme order keys of the finite ones, and the exact
// sums over the LW binades below the window, t = m 2^(e - lw) < 2^(MB + LW)
// in units of 2^(lw - BM) (sum of t as int64, of t^2 in 128 bits: a piece
// holds fewer than 2^32 elements, so a thread fewer than 2^24).  Binades
// above the window or further below go to the CTA's digits.
constexpr int LW = 28;
struct SlowSlot {
  long long s1;
  unsigned long long s2lo, s2hi;
  uint32_t kmn, kmx, nnan, ninf;
};

template <int DT>
__device__ __noinline__ void h16_slow(uint32_t r, int lw, SlowSlot& q, long long* lim) {
  using T = TS<DT>;
  const uint32_t e = (r >> T::MB) & T::EMASK, mant = r & ((1u << T::MB) - 1u);
  if (e == T::EINF) {
    if (mant) q.nnan++;
    else q.ninf++;
    return;
  }
  const uint32_t k = order_key(raw_to_f32<DT>(r));
  q.kmn = min(q.kmn, k);
  q.kmx = max(q.kmx, k);
  const uint32_t m = mant | (e ? (1u << T::MB) : 0u);
  if (!m) return;
  const int ee = e ? (int)e : 1;
  const bool neg = (r >> (T::BITS - 1)) & 1u;
  if (ee >= lw && ee - lw < LW) {
    const uint64_t t = (uint64_t)m << (ee - lw);
    q.s1 += neg ? -(long long)t : (long long)t;
    const unsigned __int128 s2 = (((unsigned __int128)q.s2hi << 64) | q.s2lo) + (unsigned __int128)t * t;
    q.s2lo = (uint64_t)s2;
    q.s2hi = (uint64_t)(s2 >> 64);
  } else {
    ts_slow<DT>(m, ee, neg, lim);
  }
}

template <int DT>
// four CTAs per SM (at most 64 registers: the piece end's wider sums must not
// cost the element loop its occupancy)
__global__ void __launch_bounds__(TB, 4) tstats_hist(TsParams p) {
  using T = TS<DT>;
  constexpr int VEC = T::VEC, B = T::BYTES, MB = T::MB, WS = H16<DT>::WS, WSB = H16<DT>::WSB;
  constexpr int NB = h16_bins<DT>();
  constexpr uint32_t WSM = (uint32_t)WS << MB, MAGM = (1u << (T::BITS - 1)) - 1u;
  pdl_trigger();  // the finalize kernel may start launching (it waits for this grid)
  extern __shared__ uint32_t hist[];  // NB bins, then the bins of +0 and -0
  __shared__ long long lim[2 * NLIMB];
  __shared__ unsigned long long cnt[3];
  __shared__ unsigned int kmin_s, kmax_s, emax_s;
  __shared__ unsigned long long red[4][TB / 32][4];
  __shared__ SlowSlot slow[TB];
  __shared__ int took_s;  // some warp of the piece took elements outside the window
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t lo = p.bounds[blockIdx.x], hi = p.bounds[blockIdx.x + 1];
  if (lo >= hi) return;
  int64_t s0 = 0, s1 = p.nseg;
  while (s1 - s0 > 1) {
    const int64_t mid = (s0 + s1) / 2;
    if (p.offsets[mid] <= lo) s0 = mid;
    else s1 = mid;
  }
  int64_t seg = s0;
  while (p.offsets[seg + 1] <= lo) seg++;
  const uint32_t hb = (uint32_t)__cvta_generic_to_shared(hist);
  for (int j = tid; j < NB + 2; j += TB) hist[j] = 0;
  for (int64_t a = lo; a < hi;) {
    const int64_t b = min(hi, p.offsets[seg + 1]);
    for (int j = tid; j < 2 * NLIMB; j += TB) lim[j] = 0;
    if (tid < 3) cnt[tid] = 0;
    if (tid == 0) {
      kmin_s = 0xFFFFFFFFu;
      kmax_s = 0;
      emax_s = 0;
      took_s = 0;
    }
    slow[tid] = SlowSlot{0, 0, 0, 0xFFFFFFFFu, 0u, 0u, 0u};
    // the vector grid inside the piece
    int64_t a0 = b, nv = 0;
    if (p.p0 >= 0 && p.p0 < p.n_total) {
      a0 = a <= p.p0 ? p.p0 : p.p0 + ((a - p.p0 + VEC - 1) / VEC) * VEC;
      if (a0 < b) nv = (b - a0) / VEC;
      else a0 = b;
    }
    __syncthreads();
    // the window: one binade above the largest finite exponent among the
    // first vector of every thread (or the tail's first elements)
    {
      uint32_t em = 0;
      if (tid < nv) {
        const uint4 v = ts_vec(p.x, (a0 + (int64_t)tid * VEC) * B);  // this thread's first vector of the piece
#pragma unroll
        for (int j = 0; j < VEC; j++) {
          const uint32_t e = (ts_lane<DT>(v, j) >> MB) & T::EMASK;
          if (e != T::EINF) em = max(em, e);
        }
      } else if (nv == 0 && a + tid < b) {
        const uint32_t e = (ts_load<DT>(p.x, a + tid) >> MB) & T::EMASK;
        if (e != T::EINF) em = e;
      }
      em = __reduce_max_sync(0xFFFFFFFFu, em);
      if (lane == 0 && em) atomicMax(&emax_s, em);
    }
    __syncthreads();
    const int lb = max(1, min((int)emax_s + 2 - WS, (int)T::EINF - WS));  // window exponents [lb, lb + WS)
    const int lw = max(1, lb - LW);                                        // the slots' binades [lw, lw + LW)
    const uint32_t lbm = (uint32_t)lb << MB;
    auto elem = [&](uint32_t r) {
      const uint32_t mag = r & MAGM, t = mag - lbm;
      if (t < WSM) {
        asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(hb + 4u * (t | ((r >> (T::BITS - 1)) << (WSB + MB)))),
                     "r"(1u)
                     : "memory");
      } else if (mag == 0) {
        asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(hb + 4u * (NB + (r >> (T::BITS - 1)))), "r"(1u)
                     : "memory");
      } else {
        h16_slow<DT>(r, lw, slow[tid], lim);
      }
    };
    constexpr int U = 4;
    for (int64_t k0 = 0; k0 < nv; k0 += (int64_t)U * TB) {
      uint4 v[U];
#pragma unroll
      for (int uu = 0; uu < U; uu++) {
        const int64_t k = k0 + uu * TB + tid;
        v[uu] = k < nv ? ts_vec(p.x, (a0 + k * VEC) * B) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int uu = 0; uu < U; uu++) {
        if (k0 + uu * TB + tid < nv) {
#pragma unroll
          for (int j = 0; j < VEC; j++) elem(ts_lane<DT>(v[uu], j));
        }
      }
    }
    {  // the elements outside the vector grid: [a, a0) and [a0 + nv VEC, b)
      const int64_t h = a0 - a, t0 = a0 + nv * VEC, ns = h + (b - t0);
      for (int64_t i = tid; i < ns; i += TB) elem(ts_load<DT>(p.x, i < h ? a + i : t0 + (i - h)));
    }
    __syncthreads();
    // the bins: exact sums in units of 2^(lb - BM) (S1 by sign, S2), the
    // extreme keys, and the bins cleared for the next piece
    unsigned __int128 s1p = 0, s1n = 0, s2 = 0;
    uint32_t kmn = 0xFFFFFFFFu, kmx = 0;
    for (int bin = tid; bin < NB + 2; bin += TB) {
      const uint32_t c = hist[bin];
      if (!c) continue;
      hist[bin] = 0;
      uint32_t r;
      if (bin >= NB) {
        r = (uint32_t)(bin - NB) << (T::BITS - 1);  // +0 or -0
      } else {
        const uint32_t sg = (uint32_t)bin >> (WSB + MB), slot = ((uint32_t)bin >> MB) & (WS - 1u);
        const uint32_t mant = (uint32_t)bin & ((1u << MB) - 1u);
        r = (sg << (T::BITS - 1)) | ((uint32_t)(lb + (int)slot) << MB) | mant;
        const uint64_t tt = (uint64_t)(mant | (1u << MB)) << slot;  // below 2^(MB + WS)
        const unsigned __int128 ct = (unsigned __int128)tt * c;
        if (sg) s1n += ct;
        else s1p += ct;
        s2 += ct * tt;  // below 2^(2 (MB + WS) + 32)
      }
      const uint32_t k = order_key(raw_to_f32<DT>(r));
      kmn = min(kmn, k);
      kmx = max(kmx, k);
    }
    // block totals: 32-bit words of each 128-bit sum (the window's, and the
    // slots' below it) summed over the warp, then over the warps by thread 0,
    // added as digits; the slots' counts and extreme keys with them
    {
      const SlowSlot q0 = slow[tid];
      const unsigned __int128 d = s1p - s1n;  // |S1| < 2^120: two's complement in 128 bits
#pragma unroll
      for (int q = 0; q < 4; q++) {
        uint64_t w1 = (uint32_t)(d >> (32 * q)), w2 = (uint32_t)(s2 >> (32 * q));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          w1 += __shfl_xor_sync(0xFFFFFFFFu, w1, o);
          w2 += __shfl_xor_sync(0xFFFFFFFFu, w2, o);
        }
        if (lane == 0) {
          red[0][warp][q] = w1;
          red[1][warp][q] = w2;
        }
      }
      // the slots: only a warp that took elements outside the window has work here
      const bool took = q0.kmn != 0xFFFFFFFFu || (q0.nnan | q0.ninf) != 0u;
      if (__any_sync(0xFFFFFFFFu, took)) {
        const unsigned __int128 dl = (unsigned __int128)(__int128)q0.s1;
        const unsigned __int128 s2l = ((unsigned __int128)q0.s2hi << 64) | q0.s2lo;
#pragma unroll
        for (int q = 0; q < 4; q++) {
          uint64_t w1 = (uint32_t)(dl >> (32 * q)), w2 = (uint32_t)(s2l >> (32 * q));
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            w1 += __shfl_xor_sync(0xFFFFFFFFu, w1, o);
            w2 += __shfl_xor_sync(0xFFFFFFFFu, w2, o);
          }
          if (lane == 0) {
            red[2][warp][q] = w1;
            red[3][warp][q] = w2;
          }
        }
        kmn = min(kmn, q0.kmn);
        kmx = max(kmx, q0.kmx);
        const uint32_t nn = __reduce_add_sync(0xFFFFFFFFu, q0.nnan), ni = __reduce_add_sync(0xFFFFFFFFu, q0.ninf);
        if (lane == 0) {
          if (nn) atomicAdd(&cnt[1], (unsigned long long)nn);
          if (ni) atomicAdd(&cnt[2], (unsigned long long)ni);
          took_s = 1;
        }
      } else if (lane < 4) {
        red[2][warp][lane] = 0;
        red[3][warp][lane] = 0;
      }
      kmn = __reduce_min_sync(0xFFFFFFFFu, kmn);
      kmx = __reduce_max_sync(0xFFFFFFFFu, kmx);
      if (lane == 0) {
        if (kmn != 0xFFFFFFFFu) atomicMin(&kmin_s, kmn);
        if (kmx) atomicMax(&kmax_s, kmx);
      }
    }
    __syncthreads();
    if (tid == 0) {
      // word q of S1 (two's complement) and of S2, each summed over the block;
      // S1's words rebuild its 128-bit value, whose sign is its top bit
      unsigned __int128 S1 = 0, S2w[4];
      for (int q = 0; q < 4; q++) {
        unsigned __int128 t1 = 0, t2 = 0;
        for (int w = 0; w < TB / 32; w++) {
          t1 += red[0][w][q];
          t2 += red[1][w][q];
        }
        S1 += t1 << (32 * q);
        S2w[q] = t2;
      }
      const int u = lb - T::BM;  // weight of a unit
      const bool neg = (S1 >> 127) != 0;
      const unsigned __int128 mag1 = neg ? (unsigned __int128)0 - S1 : S1;
      for_digits(mag1, u, neg, [&](int j, int64_t v) { lim_add(lim, j, v); });
      for (int q = 0; q < 4; q++)
        if (S2w[q]) for_digits(S2w[q], 2 * u + 32 * q, false, [&](int j, int64_t v) { lim_add(lim + NLIMB, j, v); });
      // the slots' sums, in units of 2^(lw - BM)
      unsigned __int128 L1 = 0;
      for (int q = 0; q < 4 && took_s; q++) {
        unsigned __int128 t1 = 0, t2 = 0;
        for (int w = 0; w < TB / 32; w++) {
          t1 += red[2][w][q];
          t2 += red[3][w][q];
        }
        L1 += t1 << (32 * q);
        const int ul = lw - T::BM;
        if (t2) for_digits(t2, 2 * ul + 32 * q, false, [&](int j, int64_t v) { lim_add(lim + NLIMB, j, v); });
      }
      const bool negl = (L1 >> 127) != 0;
      const unsigned __int128 magl = negl ? (unsigned __int128)0 - L1 : L1;
      if (magl) for_digits(magl, lw - T::BM, negl, [&](int j, int64_t v) { lim_add(lim, j, v); });
    }
    __syncthreads();
    TsAcc& acc = p.acc[seg];
    for (int j = tid; j < 2 * NLIMB; j += TB)
      if (lim[j]) atomicAdd(reinterpret_cast<unsigned long long*>(&acc.limbs[0][0] + j), (unsigned long long)lim[j]);
    if (tid == 0) {
      const unsigned long long nfin = (unsigned long long)(b - a) - cnt[1] - cnt[2];
      if (nfin) atomicAdd(&acc.nfin, nfin);
      if (cnt[1]) atomicAdd(&acc.nnan, cnt[1]);
      if (cnt[2]) atomicAdd(&acc.ninf, cnt[2]);
      if (nfin) {
        atomicMax(&acc.kmin_inv, ~kmin_s);
        atomicMax(&acc.kmax, kmax_s);
      }
    }
    __syncthreads();
    a = b;
    while (seg < p.nseg && p.offsets[seg + 1] <= a) seg++;
  }
}

// ---- stage 2: exact mean and variance ----
// Every loop below has compile-time bounds and is unrolled, so the digit
// arrays stay in registers.

// NLIMB carry-save digits -> sign and magnitude in base-2^32 digits
__device__ __forceinline__ bool to_magnitude(const long long* src, uint32_t (&d)[NLIMB]) {
  int64_t t[NLIMB], carry = 0;
#pragma unroll
  for (int j = 0; j < NLIMB; j++) {
    const int64_t v = src[j] + carry;
    carry = v >> 32;
    t[j] = v & 0xFFFFFFFFll;
  }
  t[NLIMB - 1] += carry * ((int64_t)1 << 32);  // the top digit carries the sign
  const bool neg = t[NLIMB - 1] < 0;
  if (neg) {
    carry = 0;
#pragma unroll
    for (int j = 0; j < NLIMB; j++) {
      const int64_t v = -t[j] + carry;
      carry = v >> 32;
      t[j] = v & 0xFFFFFFFFll;
    }
  }
#pragma unroll
  for (int j = 0; j < NLIMB; j++) d[j] = (uint32_t)t[j];
  return neg;
}

constexpr int SH = -LIMB_LSB / 32;  // S2 shifted up by -LIMB_LSB bits: a whole number of digits
static_assert(-LIMB_LSB % 32 == 0, "digit-aligned shift");
constexpr int ND = 2 * NLIMB + SH + 3;

// RN-even binary64 of N 2^scale / n^2 for a magnitude N of ND base-2^32
// digits and 1 <= n < 2^36: the leading 128 bits of N divided by n twice
// (each quotient keeps at least 55 significant bits), the dropped bits and the
// remainders as the sticky bit.
__device__ __forceinline__ double div_n2_rn(const uint32_t (&N)[ND], int scale, uint64_t n) {
  int top = -1;
#pragma unroll
  for (int j = 0; j < ND; j++)
    if (N[j]) top = j;
  if (top < 0) return 0.0;
  uint32_t w4 = 0, w3 = 0, w2 = 0, w1 = 0, w0 = 0;
  bool sticky = false;
#pragma unroll
  for (int j = 0; j < ND; j++) {
    if (j == top) w4 = N[j];
    if (j == top - 1) w3 = N[j];
    if (j == top - 2) w2 = N[j];
    if (j == top - 3) w1 = N[j];
    if (j == top - 4) w0 = N[j];
    if (j < top - 4 && N[j] != 0) sticky = true;
  }
  const int lz = __clz(w4);
  const unsigned __int128 win = ((unsigned __int128)w4 << 96) | ((unsigned __int128)w3 << 64) |
                                ((unsigned __int128)w2 << 32) | w1;
  const unsigned __int128 W = lz ? ((win << lz) | (w0 >> (32 - lz))) : win;
  if ((lz ? (uint32_t)(w0 << lz) : w0) != 0) sticky = true;
  const int E = 32 * (top - 3) - lz + scale;  // weight of W's last bit
  unsigned __int128 q2;
  if (n < ((uint64_t)1 << 32)) {  // n^2 fits 64 bits: one division
    const uint64_t d = n * n;
    q2 = W / d;
    if (W - q2 * d != 0) sticky = true;
  } else {
    const unsigned __int128 q = W / n;
    if (W - q * n != 0) sticky = true;
    q2 = q / n;
    if (q - q2 * n != 0) sticky = true;
  }
  const uint64_t qh = (uint64_t)(q2 >> 64);
  const int qlz = qh ? __clzll(qh) : 64 + __clzll((uint64_t)q2);
  const int shift = 64 - qlz;  // q2 >= 2^55: keep its leading 64 bits
  uint64_t m;
  if (shift >= 0) {
    m = (uint64_t)(q2 >> shift);
    if (shift > 0 && (q2 & (((unsigned __int128)1 << shift) - 1)) != 0) sticky = true;
  } else {
    m = (uint64_t)q2 << (-shift);
  }
  uint64_t mant = m >> 11;
  const uint64_t rbits = m & 0x7FFull;
  if (rbits > 0x400ull || (rbits == 0x400ull && (sticky || (mant & 1ull)))) mant++;
  return ldexp((double)mant, 11 + shift + E);
}

__device__ __forceinline__ double key_to_double(uint32_t k) {
  return (double)__uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// The exact population variance of one segment's accumulator (n_f > 0), by
// one warp: lane 0 turns the sums into magnitude digits, every lane adds the
// products of one or two columns of S1^2, lane 0 forms n_f S2 - S1^2 and
// rounds its quotient by n_f^2 once.
struct VarScratch {
  uint32_t A[NLIMB], B[NLIMB];
  unsigned __int128 col[2 * NLIMB];
};
__device__ __noinline__ double seg_variance(const TsAcc& acc, uint64_t nf, VarScratch& vs) {
  const int lane = threadIdx.x & 31;
  if (lane == 0) {
    uint32_t A[NLIMB], Bm[NLIMB];
    to_magnitude(acc.limbs[0], A);
    to_magnitude(acc.limbs[1], Bm);
#pragma unroll
    for (int j = 0; j < NLIMB; j++) {
      vs.A[j] = A[j];
      vs.B[j] = Bm[j];
    }
  }
  __syncwarp();
  for (int k = lane; k < 2 * NLIMB; k += 32) {
    unsigned __int128 c = 0;
    const int i0 = k < NLIMB ? 0 : k - NLIMB + 1, i1 = k < NLIMB ? k : NLIMB - 1;
    for (int i = i0; i <= i1; i++) c += (uint64_t)vs.A[i] * vs.A[k - i];
    vs.col[k] = c;
  }
  __syncwarp();
  double var = 0.0;
  if (lane == 0) {
    // N = n_f (S2 << SH digits) - S1^2, in units of 2^(2 LIMB_LSB)
    uint32_t N[ND];
    unsigned __int128 c = 0, carry = 0;
    uint32_t borrow = 0;
#pragma unroll
    for (int j = 0; j < ND; j++) {
      if (j >= SH && j < SH + NLIMB) c += (unsigned __int128)vs.B[j - SH] * nf;
      const uint32_t nb = (uint32_t)c;
      c >>= 32;
      unsigned __int128 col = carry;
      if (j < 2 * NLIMB) col += vs.col[j];
      const uint32_t dig = (uint32_t)col;
      carry = col >> 32;
      const uint64_t sub = (uint64_t)dig + borrow;  // the result is n_f^2 times a variance, >= 0
      N[j] = nb - (uint32_t)sub;
      borrow = (uint64_t)nb < sub ? 1u : 0u;
    }
    var = div_n2_rn(N, 2 * LIMB_LSB, nf);
  }
  return var;
}

// the mean S1 / n_f of one segment's accumulator (n_f > 0), with S1's sign
__device__ __noinline__ double seg_mean(const TsAcc& acc, uint64_t nf) {
  uint32_t A[NLIMB];
  const bool neg = to_magnitude(acc.limbs[0], A);
  long long mag[NLIMB];
#pragma unroll
  for (int j = 0; j < NLIMB; j++) mag[j] = neg ? -acc.limbs[0][j] : acc.limbs[0][j];
  const double m = limbs_div_rn(mag, nf);
  return neg ? -m : m;
}

// One CTA of four warps per segment: warp 0 the variance, warp 1 the mean,
// warp 2 the two sums, side by side; then the record is written and the
// accumulator cleared for the next call.
constexpr int FIN_THREADS = 128;
__global__ void __launch_bounds__(FIN_THREADS) tstats_finalize(TsParams p) {
  pdl_wait();  // stage 1 complete
  const int64_t s = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5;
  TsAcc& acc = p.acc[s];
  __shared__ double res[4];
  __shared__ VarScratch vs;
  const uint64_t nf = acc.nfin;
  if (warp == 0) {
    const double v = nf ? seg_variance(acc, nf, vs) : 0.0;
    if (tid == 0) res[0] = v;
  }
  if ((tid & 31) == 0) {
    if (warp == 1) res[1] = nf ? seg_mean(acc, nf) : 0.0;
    if (warp == 2) {
      res[2] = limbs_to_double(acc.limbs[0]);
      res[3] = limbs_to_double(acc.limbs[1]);
    }
  }
  __syncthreads();
  if (tid == 0) {
    peat_tstats_t r;
    r.n = (uint64_t)(p.offsets[s + 1] - p.offsets[s]);
    r.n_finite = nf;
    r.n_nan = acc.nnan;
    r.n_inf = acc.ninf;
    r.sum = res[2];
    r.sum_sq = res[3];
    r.mean = res[1];
    r.var = res[0];
    r.min = nf ? key_to_double(~acc.kmin_inv) : 0.0;
    r.max = nf ? key_to_double(acc.kmax) : 0.0;
    p.out[s] = r;
  }
  __syncthreads();
  if (tid < NLIMB) acc.limbs[0][tid] = acc.limbs[1][tid] = 0;
  if (tid == 0) {
    acc.nfin = acc.nnan = acc.ninf = 0;
    acc.kmin_inv = acc.kmax = 0;
  }
}

template <int DT>
constexpr size_t hist_smem() {
  return sizeof(uint32_t) * (size_t)(h16_bins<DT>() + 2);
}

// the dynamic shared memory of the histogram kernel, allowed once per process
cudaError_t hist_prepare() {
  static const cudaError_t e = cudaFuncSetAttribute(tstats_hist<PEAT_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    (int)hist_smem<PEAT_BF16>());
  return e;
}

// Stage 1 by element type: the bit-pattern histogram for bf16 (a window of 32
// of its 254 binades holds nearly every tensor's bulk); the per-thread integer
// window for float32 and fp16 (fp16 has only 30 binades, and the histogram's
// 8-binade window leaves a wide distribution largely to the exact path:
// Laplace-distributed fp16 checkpoint values took 11.9 ms for 355 M elements,
// the register window of 16 binades takes them all but the tiniest)
template <int DT>
cudaError_t launch_t(const TsParams& p, cudaStream_t s) {
  if constexpr (DT != PEAT_BF16) {
    tstats_stage1<DT><<<p.nctas, TB, 0, s>>>(p);
  } else {
    const cudaError_t e = hist_prepare();
    if (e != cudaSuccess) return e;
    tstats_hist<DT><<<p.nctas, TB, hist_smem<DT>(), s>>>(p);
  }
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // a programmatic dependent of stage 1: its launch overlaps stage 1's end
  return launch_dependent(tstats_finalize, (unsigned)p.nseg, FIN_THREADS, 0, s, p);
}

}  // namespace

int tstats_ctas_per_sm(int dtype) {
  struct Occ {
    int v[3];
  };
  static const Occ o = [] {
    Occ r{{1, 1, 1}};
    hist_prepare();
    int a = 0, b = 0, c = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&a, tstats_stage1<PEAT_F32>, TB, 0);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, tstats_stage1<PEAT_F16>, TB, 0);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&c, tstats_hist<PEAT_BF16>, TB, hist_smem<PEAT_BF16>());
    cudaGetLastError();
    if (a > 0) r.v[0] = a;
    if (b > 0) r.v[1] = b;
    if (c > 0) r.v[2] = c;
    return r;
  }();
  return dtype == PEAT_F32 ? o.v[0] : dtype == PEAT_F16 ? o.v[1] : o.v[2];
}

int64_t tstats_vec_elems(int dtype) { return dtype == PEAT_F32 ? 4 : 8; }

cudaError_t launch_tstats(int dtype, const TsParams& p, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return launch_t<PEAT_F32>(p, s);
    case PEAT_F16: return launch_t<PEAT_F16>(p, s);
    case PEAT_BF16: return launch_t<PEAT_BF16>(p, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t register_digit_status_tstats(unsigned int* word) { return set_digit_status_here(word); }

}  // namespace peat
