// Mean of the top errors (Section IV-B-3, "Mean of Top 10% Errors") on sm_103a.
//
// Over the pairs with both operands finite, the k = ceil(n_finite num / den)
// largest |d| = |c - g|: their exact sum and exact mean, rounded once.
//
// key(|d|) is an order-preserving 31-bit key: the bits of RN32(|d|) (RN32 is
// monotone and float bits order like the values), or, when c - g overflows
// float32, the bits of RN32(|d| / 2) plus 2^23 (above every key of the first
// kind).  The key T of the k-th largest |d| is resolved in digits of 10, 11
// and 10 bits, and every |d| whose key is known to lie above T is summed
// exactly on the way:
//   sample  evenly spaced pairs give the digit of key >> 21 where their own
//           top fraction ends; the window [Plo, Phi] is that digit +- 1;
//   pass 1  every pair: those with key >> 21 above the window counted and
//           summed, those inside counted by key >> 10; the last CTA checks
//           that the window holds the k-th largest and resolves P1 = T >> 10;
//   (pass 0 and pass 1 again on the exact digit, only if the window missed)
//   pass 2  every pair: digit histogram of bits 9..0 for key >> 10 = P1, the
//           exact sum of the window's pairs with key >> 10 > P1, and a list
//           of the pairs with key >> 10 = P1 whose |d| is not a float32 value
//           (their rounding errors lo, |d| = value(key) + lo);
//   pass 3  only if that list overflowed: the pairs with key >> 10 = P1 and
//           key > T summed exactly, and T's inexact pairs listed again;
//   pass 4, 5  only if even T's inexact pairs overflow the list: a radix
//           select over the order key of T's rounding errors (16 + 16 bits),
//           summing exactly the errors above the resolved prefix.
// The last CTA to finish a pass selects its digit.  A one-CTA finalize adds
// the P1 range above T from the histogram (every key there is one float32
// value), m value(T) for the m pairs of T's bucket that belong to the top k,
// the listed rounding errors above T and the m largest of T's bucket, and
// rounds sum and mean once.  All sums are exact: float32 values in units of a
// binade floor as 64-bit integers, everything else as fixed-point digits.
// Work on rare pairs is queued per warp and done 32 pairs at a time.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "exact.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

constexpr int TB = 256;                    // threads per CTA
constexpr unsigned KEY_OVF = 0x7F800000u;  // keys from here up: c - g overflowed float32
constexpr int NO_FAST = 1000;              // binade floor that disables the integer path

template <int DT>
struct TK;
template <>
struct TK<PEAT_F32> {
  static constexpr int BYTES = 4, VEC = 4;
  static constexpr uint32_t MAG = 0x7FFFFFFFu, INF = 0x7F800000u;
};
template <>
struct TK<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8;
  static constexpr uint32_t MAG = 0x7FFFu, INF = 0x7C00u;
  static constexpr int MB = 10, EMASK = 0x1F;  // fraction bits, exponent field
};
template <>
struct TK<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8;
  static constexpr uint32_t MAG = 0x7FFFu, INF = 0x7F80u;
  static constexpr int MB = 7, EMASK = 0xFF;
};

// 16-bit operands: c - g may be inexact in float32 only when their exponents
// are more than 23 - MB apart (the difference then spans more than 24 bits);
// a subnormal's exponent field counts as 1
template <int DT>
__device__ __forceinline__ uint32_t maybe_inexact(uint32_t G, uint32_t C) {
  const int eg = max((int)((G >> TK<DT>::MB) & TK<DT>::EMASK), 1);
  const int ec = max((int)((C >> TK<DT>::MB) & TK<DT>::EMASK), 1);
  return (uint32_t)(abs(eg - ec) > 23 - TK<DT>::MB);
}

template <int DT>
__device__ __forceinline__ float tk_f32(uint32_t r) {
  if constexpr (DT == PEAT_F32) return __uint_as_float(r);
  else if constexpr (DT == PEAT_BF16) return __uint_as_float(r << 16);
  else return __half2float(__ushort_as_half((unsigned short)r));
}

template <int DT>
__device__ __forceinline__ bool tk_finite(uint32_t G, uint32_t C) {
  return (G & TK<DT>::MAG) < TK<DT>::INF && (C & TK<DT>::MAG) < TK<DT>::INF;
}

template <int DT>
__device__ __forceinline__ uint32_t tk_lane(const uint4& v, int j) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (TK<DT>::BYTES == 4) return w[j];
  else return (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
}

template <int DT>
__device__ __forceinline__ uint32_t tk_load(const void* base, int64_t i) {
  if constexpr (TK<DT>::BYTES == 4) return __ldg(reinterpret_cast<const uint32_t*>(base) + i);
  else return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(base) + i);
}

__device__ __forceinline__ uint4 tk_vec(const void* base, int64_t byte_off) {
  const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(base) + byte_off);
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(q));
  return v;
}

// the order-preserving key of |c - g| for a finite pair
__device__ __forceinline__ uint32_t tk_key(float gf, float cf) {
  const float s = __fsub_rn(cf, gf);
  if (fabsf(s) < __int_as_float(0x7F800000)) return __float_as_uint(fabsf(s));
  // both operands finite and large: halving them is exact
  const float h = __fsub_rn(__fmul_rn(cf, 0.5f), __fmul_rn(gf, 0.5f));
  return __float_as_uint(fabsf(h)) + (1u << 23);
}

// |d| = (hi + lo) 2^sc exactly (float32 TwoSum, halved when c - g overflows);
// hi is the value of the pair's key
__device__ __forceinline__ void tk_exact(float gf, float cf, float& hi, float& lo, int& sc) {
  float x = cf, y = -gf;
  sc = 0;
  float s = __fadd_rn(x, y);
  if (!(fabsf(s) < __int_as_float(0x7F800000))) {
    x = __fmul_rn(x, 0.5f);
    y = __fmul_rn(y, 0.5f);
    s = __fadd_rn(x, y);
    sc = 1;
  }
  const float yv = __fsub_rn(s, x), xv = __fsub_rn(s, yv);
  const float t = __fadd_rn(__fsub_rn(x, xv), __fsub_rn(y, yv));
  hi = fabsf(s);
  lo = s < 0.0f ? -t : t;
}

// the value a key stands for: v 2^sc
__device__ __forceinline__ float key_value(unsigned key, int& sc) {
  sc = key >= KEY_OVF ? 1 : 0;
  return __uint_as_float(key - (sc ? (1u << 23) : 0u));
}

// the bits of |RN32(c - g)|: the key of a finite pair unless c - g
// overflows; at or above KEY_OVF for a pair with a NaN or an infinity too
template <int DT>
__device__ __forceinline__ uint32_t raw_key(uint32_t G, uint32_t C) {
  return __float_as_uint(__fsub_rn(tk_f32<DT>(C), tk_f32<DT>(G))) & 0x7FFFFFFFu;
}

// one queued pair: both raw operands
template <int DT>
struct QT {
  using T = uint32_t;
};
template <>
struct QT<PEAT_F32> {
  using T = uint2;
};
template <int DT>
__device__ __forceinline__ typename QT<DT>::T q_pack(uint32_t G, uint32_t C) {
  if constexpr (TK<DT>::BYTES == 4) return make_uint2(G, C);
  else return G | (C << 16);
}
template <int DT>
__device__ __forceinline__ void q_unpack(const typename QT<DT>::T& e, uint32_t& G, uint32_t& C) {
  if constexpr (TK<DT>::BYTES == 4) {
    G = e.x;
    C = e.y;
  } else {
    G = e & 0xFFFFu;
    C = e >> 16;
  }
}
template <int DT>
constexpr int ring_cap() {
  return 64 * TK<DT>::VEC;  // at least 31 left over + 32 VEC pushed at once
}

// Every pair once, f(G, C); two vectors per thread in flight.  No
// warp-collective work inside f.
template <int DT, class F>
__device__ __forceinline__ void tk_visit(const TopkParams& p, F&& f) {
  constexpr int VEC = TK<DT>::VEC, B = TK<DT>::BYTES;
  const int64_t stride = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  int64_t v = gt;
  for (; v + stride < p.nvec; v += 2 * stride) {
    const int64_t o0 = (p.p0 + v * VEC) * B, o1 = o0 + stride * VEC * B;
    const uint4 g0 = tk_vec(p.g, o0), c0 = tk_vec(p.c, o0);
    const uint4 g1 = tk_vec(p.g, o1), c1 = tk_vec(p.c, o1);
#pragma unroll
    for (int j = 0; j < VEC; j++) f(tk_lane<DT>(g0, j), tk_lane<DT>(c0, j));
#pragma unroll
    for (int j = 0; j < VEC; j++) f(tk_lane<DT>(g1, j), tk_lane<DT>(c1, j));
  }
  if (v < p.nvec) {
    const int64_t o0 = (p.p0 + v * VEC) * B;
    const uint4 g0 = tk_vec(p.g, o0), c0 = tk_vec(p.c, o0);
#pragma unroll
    for (int j = 0; j < VEC; j++) f(tk_lane<DT>(g0, j), tk_lane<DT>(c0, j));
  }
  // elements outside the vector grid: [0, head) and [tail, n)
  const int64_t head = p.p0 >= 0 ? p.p0 : p.n, tail = p.p0 >= 0 ? p.p0 + p.nvec * VEC : p.n;
  const int64_t ns = head + (p.n - tail);
  for (int64_t idx = gt; idx < ns; idx += stride) {
    const int64_t i = idx < head ? idx : tail + (idx - head);
    f(tk_load<DT>(p.g, i), tk_load<DT>(p.c, i));
  }
}

// Every pair that passes the cheap test isint (a superset of the pairs the
// pass needs) reaches proc(G, C), which makes the exact decision.  Pairs that
// pass are queued in the warp's ring and handed to proc 32 at a time, so the
// rarely taken work runs on full warps.
template <int DT, class Pred, class Proc>
__device__ __forceinline__ void tk_filtered(const TopkParams& p, typename QT<DT>::T* ring, Pred&& isint,
                                            Proc&& proc) {
  constexpr int VEC = TK<DT>::VEC, B = TK<DT>::BYTES, CAP = ring_cap<DT>();
  const uint32_t lane = threadIdx.x & 31;
  uint32_t head = 0, tail = 0;  // the same in every lane
  auto push = [&](const uint4& gv, const uint4& cv, bool ok) {
    uint32_t mask = 0;
#pragma unroll
    for (int j = 0; j < VEC; j++) mask |= isint(tk_lane<DT>(gv, j), tk_lane<DT>(cv, j)) ? (1u << j) : 0u;
    if (!ok) mask = 0;
    if (!__any_sync(0xFFFFFFFFu, mask != 0)) return;
    const uint32_t cnt = __popc(mask);
    uint32_t incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= (uint32_t)o) incl += t;
    }
    const uint32_t total = __shfl_sync(0xFFFFFFFFu, incl, 31);
    uint32_t pos = tail + incl - cnt;
#pragma unroll
    for (int j = 0; j < VEC; j++)
      if (mask & (1u << j)) ring[(pos++) & (CAP - 1)] = q_pack<DT>(tk_lane<DT>(gv, j), tk_lane<DT>(cv, j));
    tail += total;
    __syncwarp();
    while (tail - head >= 32) {
      uint32_t G, C;
      q_unpack<DT>(ring[(head + lane) & (CAP - 1)], G, C);
      head += 32;
      proc(G, C);
    }
    __syncwarp();
  };
  const int64_t stride = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  // rounds of two vectors; every lane of the warp takes every round
  for (int64_t v = gt; __any_sync(0xFFFFFFFFu, v < p.nvec); v += 2 * stride) {
    const bool ok0 = v < p.nvec, ok1 = v + stride < p.nvec;
    const uint4 z = make_uint4(0, 0, 0, 0);
    const int64_t o0 = (p.p0 + v * VEC) * B, o1 = o0 + stride * VEC * B;
    const uint4 g0 = ok0 ? tk_vec(p.g, o0) : z, c0 = ok0 ? tk_vec(p.c, o0) : z;
    const uint4 g1 = ok1 ? tk_vec(p.g, o1) : z, c1 = ok1 ? tk_vec(p.c, o1) : z;
    push(g0, c0, ok0);
    push(g1, c1, ok1);
  }
  if (lane < tail - head) {
    uint32_t G, C;
    q_unpack<DT>(ring[(head + lane) & (CAP - 1)], G, C);
    proc(G, C);
  }
  // elements outside the vector grid: [0, head) and [tail, n)
  const int64_t hd = p.p0 >= 0 ? p.p0 : p.n, tl = p.p0 >= 0 ? p.p0 + p.nvec * VEC : p.n;
  const int64_t ns = hd + (p.n - tl);
  for (int64_t idx = gt; idx < ns; idx += stride) {
    const int64_t i = idx < hd ? idx : tl + (idx - hd);
    const uint32_t G = tk_load<DT>(p.g, i), C = tk_load<DT>(p.c, i);
    if (isint(G, C)) proc(G, C);
  }
}

// A thread's histogram increments, run-length coded: one shared atomic per
// run of equal bins.
struct RunCount {
  uint32_t bin = 0xFFFFFFFFu, cnt = 0;
  __device__ __forceinline__ void add(uint32_t* h, uint32_t b) {
    if (b == bin) {
      cnt++;
      return;
    }
    if (cnt) atomicAdd(&h[bin], cnt);
    bin = b;
    cnt = 1;
  }
  __device__ __forceinline__ void flush(uint32_t* h) {
    if (cnt) atomicAdd(&h[bin], cnt);
  }
};

__device__ __forceinline__ void lim_add(long long* lim, int j, int64_t v) {
  atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v);
}

// +-x 2^sc as digits of the CTA's accumulator
__device__ __forceinline__ void digits_of(long long* lim, float x, int sc) {
  if (x == 0.0f) return;
  int e;
  const uint32_t m = split_float(x, e);
  for_digits(m, e + sc, x < 0.0f, [&](int j, int64_t v) { lim_add(lim, j, v); });
}

// cnt copies of +-x 2^sc as digits of the CTA's accumulator
__device__ __forceinline__ void digits_of_n(long long* lim, float x, int sc, unsigned long long cnt) {
  if (x == 0.0f || cnt == 0) return;
  int e;
  const uint32_t m = split_float(x, e);
  for_digits((unsigned __int128)m * cnt, e + sc, x < 0.0f, [&](int j, int64_t v) { lim_add(lim, j, v); });
}

// A thread's exact sum of |d|: float32 values whose binade is at most 16
// above the floor eb as an integer in units of 2^(eb - 150) (terms below
// 2^40, fewer than 2^24 terms per thread), everything else as digits.
struct ExactAcc {
  uint64_t V = 0;
  int eb;
  long long* lim;
  __device__ __forceinline__ ExactAcc(int eb_, long long* lim_) : eb(eb_), lim(lim_) {}
  __device__ __forceinline__ void add(float gf, float cf) {
    float hi, lo;
    int sc;
    tk_exact(gf, cf, hi, lo, sc);
    if (sc == 0 && lo == 0.0f) {
      const uint32_t b = __float_as_uint(hi);
      const int sh = max((int)(b >> 23), 1) - eb;
      if ((unsigned)sh <= 16u) {
        V += (uint64_t)((b & 0x7FFFFFu) | ((b >> 23) ? 0x800000u : 0u)) << sh;
        return;
      }
    }
    digits_of(lim, hi, sc);
    digits_of(lim, lo, sc);
  }
  // warp sums in 128 bits, added as digits (all lanes of the warp)
  __device__ __forceinline__ void flush() {
    uint64_t lo32 = V & 0xFFFFFFFFull, hi32 = V >> 32;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo32 += __shfl_xor_sync(0xFFFFFFFFu, lo32, o);
      hi32 += __shfl_xor_sync(0xFFFFFFFFu, hi32, o);
    }
    if ((threadIdx.x & 31) == 0 && eb < NO_FAST) {
      const unsigned __int128 S = (unsigned __int128)lo32 + ((unsigned __int128)hi32 << 32);
      if (S) for_digits(S, eb - 150, false, [&](int j, int64_t v) { lim_add(lim, j, v); });
    }
  }
};

// The CTA's shared histogram and digits into the global state; true in the
// last CTA of the grid to get here (which then sees every CTA's totals).
__device__ __forceinline__ bool pass_end(const uint32_t* h, int nb, unsigned long long* gh, const long long* lim,
                                         TopkState* st, int pass, unsigned* last_s) {
  __syncthreads();
  if (h)
    for (int b = threadIdx.x; b < nb; b += TB)
      if (h[b]) atomicAdd(&gh[b], (unsigned long long)h[b]);
  if (lim)
    for (int j = threadIdx.x; j < NLIMB; j += TB)
      if (lim[j]) atomicAdd(reinterpret_cast<unsigned long long*>(&st->limbs[j]), (unsigned long long)lim[j]);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *last_s = atomicAdd(&st->done[pass], 1u) == gridDim.x - 1 ? 1u : 0u;
  __syncthreads();
  const bool last = *last_s != 0;
  if (last) __threadfence();
  return last;
}

__device__ __forceinline__ unsigned long long block_sum(unsigned long long x) {
  __shared__ unsigned long long ws[TB / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = x;
  __syncthreads();
  unsigned long long t = 0;
#pragma unroll
  for (int w = 0; w < TB / 32; w++) t += ws[w];
  return t;
}

// One CTA: the digit d of a histogram of TB PER bins with count(bins above
// d) < krem <= count(bins at or above d); krem becomes krem - count(bins
// above d); the histogram's total is returned.  Thread t owns bins
// [t PER, t PER + PER); every loop is unrolled so the loads go out together.
template <int PER>
__device__ unsigned long long select_digit(const unsigned long long* gh, unsigned long long& krem, unsigned& digit) {
  __shared__ unsigned long long wsum[TB / 32];
  __shared__ unsigned long long sk;
  __shared__ unsigned sd;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int CH = PER < 8 ? PER : 8;  // loads in flight per step
  static_assert(PER % CH == 0, "bins per thread");
  unsigned long long mine = 0;
#pragma unroll 1
  for (int j0 = 0; j0 < PER; j0 += CH) {
#pragma unroll
    for (int j = 0; j < CH; j++) mine += __ldcg(gh + tid * PER + j0 + j);
  }
  // inclusive suffix sum over the lanes of the warp
  unsigned long long suf = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long t = __shfl_down_sync(0xFFFFFFFFu, suf, o);
    if (lane + o < 32) suf += t;
  }
  if (lane == 0) wsum[warp] = suf;
  if (tid == 0) sd = 0;
  __syncthreads();
  unsigned long long above = suf - mine, total = 0;
#pragma unroll
  for (int w = 0; w < TB / 32; w++) {
    total += wsum[w];
    if (w > warp) above += wsum[w];
  }
  const unsigned long long kr = krem;
  if (above < kr && kr <= above + mine) {  // the digit is one of this thread's bins
#pragma unroll 1
    for (int j0 = PER - CH; j0 >= 0; j0 -= CH) {
      unsigned long long c[CH];
#pragma unroll
      for (int j = 0; j < CH; j++) c[j] = __ldcg(gh + tid * PER + j0 + j);
#pragma unroll
      for (int j = CH - 1; j >= 0; j--) {
        if (above < kr && kr <= above + c[j]) {
          sd = (unsigned)(tid * PER + j0 + j);
          sk = kr - above;
        }
        above += c[j];
      }
    }
  }
  __syncthreads();
  digit = sd;
  if (kr >= 1 && kr <= total) krem = sk;
  return total;
}

__device__ __forceinline__ unsigned long long take_count(unsigned long long nfin, const TopkParams& p) {
  return (unsigned long long)(((unsigned __int128)nfin * p.num + p.den - 1) / p.den);
}

// A sample: the digit of key >> 21 where the sample's own top fraction ends,
// and the window of digits around it.  The sample is TK_SAMPLE pairs in
// evenly spaced runs of 32 vectors, one run per warp (evenly spaced single
// pairs when the operands share no vector grid).
template <int DT>
__global__ void __launch_bounds__(TB) topk_sample(TopkParams p) {
  constexpr int VEC = TK<DT>::VEC, B = TK<DT>::BYTES;
  __shared__ uint32_t h[TK_NB0];
  __shared__ unsigned last_s;
  pdl_trigger();
  TopkState* st = p.st;
  for (int b = threadIdx.x; b < TK_NB0; b += TB) h[b] = 0;
  __syncthreads();
  RunCount rc;
  auto count = [&](uint32_t G, uint32_t C) {
    uint32_t key = raw_key<DT>(G, C);
    if (key >= KEY_OVF) {
      if (!tk_finite<DT>(G, C)) return;
      key = tk_key(tk_f32<DT>(G), tk_f32<DT>(C));
    }
    rc.add(h, key >> 21);
  };
  const int64_t nw = (int64_t)gridDim.x * (TB / 32), w = (int64_t)blockIdx.x * (TB / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (p.nvec > 0) {
    const int64_t runs = min((p.nvec + 31) / 32, TK_SAMPLE / (32 * VEC));
    for (int64_t r = w; r < runs; r += nw) {
      const int64_t v = r * p.nvec / runs + lane;  // runs may overlap when nvec is small: a sample all the same
      if (v < p.nvec) {
        const int64_t off = (p.p0 + v * VEC) * B;
        const uint4 gv = tk_vec(p.g, off), cv = tk_vec(p.c, off);
#pragma unroll
        for (int j = 0; j < VEC; j++) count(tk_lane<DT>(gv, j), tk_lane<DT>(cv, j));
      }
    }
  } else {
    const int64_t ns = min(p.n, TK_SAMPLE), step = ns > 0 ? p.n / ns : 1;
    for (int64_t j = w * 32 + lane; j < ns; j += nw * 32) count(tk_load<DT>(p.g, j * step), tk_load<DT>(p.c, j * step));
  }
  rc.flush(h);
  if (!pass_end(h, TK_NB0, st->hist0, nullptr, st, 0, &last_s)) return;
  // the sample's own count of finite pairs is the histogram's total
  unsigned d = 0;
  unsigned long long kr = 0;
  const unsigned long long tot = select_digit<TK_NB0 / TB>(st->hist0, kr, d);
  if (tot > 0) {
    kr = take_count(tot, p);
    select_digit<TK_NB0 / TB>(st->hist0, kr, d);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < TK_NB0; b += TB) st->hist0[b] = 0;
  if (threadIdx.x == 0) {
    st->Plo = d > 0 ? d - 1 : 0;
    st->Phi = min(d + 1, (unsigned)TK_NB0 - 1);
    st->done[0] = 0;
  }
}

// Every pair once: the finite pairs above the window counted and summed
// exactly, those inside it counted by key >> 10, the pairs with a NaN or an
// infinity counted.  The last CTA checks that the window holds the k-th
// largest and, if so, resolves key >> 10.  As the fallback (FB) it runs only
// when the sampled window missed, on the exact window from topk_pass0.
template <int DT, bool FB>
__global__ void __launch_bounds__(TB) topk_pass1(TopkParams p) {
  __shared__ uint32_t h[TK_WIN * TK_NB1];
  __shared__ long long lim[NLIMB];
  __shared__ typename QT<DT>::T ring[(TB / 32) * ring_cap<DT>()];
  __shared__ unsigned long long cnt_s[2];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (FB && st->ok) return;
  for (int b = threadIdx.x; b < TK_WIN * TK_NB1; b += TB) h[b] = 0;
  for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
  if (threadIdx.x < 2) cnt_s[threadIdx.x] = 0;
  __syncthreads();
  const uint32_t Plo = st->Plo, Phi = st->Phi;
  // every key above the window has a biased exponent of at least (Phi + 1) >> 2
  ExactAcc acc(Phi + 1 >= (KEY_OVF >> 21) ? NO_FAST : max((int)((Phi + 1) >> 2), 1), lim);
  RunCount rc;
  uint32_t nab = 0, nnf = 0;
  // 16-bit operands: whether the window's keys all have zero low 10 bits and
  // every window |d| is a float32 value (then pass 1 resolves the last digit)
  uint32_t lowor = 0, inex = 0;
  // a pair whose raw key is below KEY_OVF is finite with that key: inside
  // the window it is only counted, here; everything above the window, and
  // every pair with a NaN, an infinity or an overflow, is queued
  tk_filtered<DT>(
      p, ring + (threadIdx.x >> 5) * ring_cap<DT>(),
      [&](uint32_t G, uint32_t C) {
        const uint32_t u = raw_key<DT>(G, C), k0 = u >> 21;
        if (k0 > Phi || u >= KEY_OVF) return true;
        if (k0 >= Plo) {
          rc.add(h, ((k0 - Plo) << 11) | ((u >> 10) & 0x7FFu));
          if constexpr (TK<DT>::BYTES == 2) {
            lowor |= u & 0x3FFu;
            inex |= maybe_inexact<DT>(G, C);
          }
        }
        return false;
      },
      [&](uint32_t G, uint32_t C) {
        if (!tk_finite<DT>(G, C)) {
          nnf++;
          return;
        }
        const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
        const uint32_t key = tk_key(gf, cf), k0 = key >> 21;
        if (k0 < Plo) return;
        if (k0 > Phi) {
          nab++;
          acc.add(gf, cf);
          return;
        }
        rc.add(h, ((k0 - Plo) << 11) | ((key >> 10) & 0x7FFu));
        if constexpr (TK<DT>::BYTES == 2) {
          lowor |= key & 0x3FFu;
          inex |= maybe_inexact<DT>(G, C);
        }
      });
  rc.flush(h);
  acc.flush();
  nab = __reduce_add_sync(0xFFFFFFFFu, nab);
  nnf = __reduce_add_sync(0xFFFFFFFFu, nnf);
  lowor = __reduce_or_sync(0xFFFFFFFFu, lowor);
  inex = __reduce_or_sync(0xFFFFFFFFu, inex);
  if ((threadIdx.x & 31) == 0) {
    if (nab) atomicAdd(&cnt_s[0], (unsigned long long)nab);
    if (nnf) atomicAdd(&cnt_s[1], (unsigned long long)nnf);
    if (lowor) atomicOr(&st->lowor, lowor);
    if (inex) atomicOr(&st->inexact, inex);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (cnt_s[0]) atomicAdd(&st->above, cnt_s[0]);
    if (cnt_s[1]) atomicAdd(&st->nonfin, cnt_s[1]);
  }
  if (!pass_end(h, TK_WIN * TK_NB1, st->hist1, lim, st, 1, &last_s)) return;
  const unsigned long long nfin = (unsigned long long)p.n - __ldcg(&st->nonfin);
  const unsigned long long k = take_count(nfin, p), above = __ldcg(&st->above);
  // krem in range: the digit is selected as the window's total comes back
  unsigned long long krem = k > above ? k - above : 0;
  unsigned d = 0;
  const unsigned long long wt = select_digit<TK_WIN * TK_NB1 / TB>(st->hist1, krem, d);
  const bool hit = k == 0 || (above < k && k <= above + wt);
  // 16-bit operands whose window keys are all multiples of 2^10 with float32
  // |d|: every window bucket holds one value, so the last digit is 0, the
  // k-th largest is P1 2^10, and the buckets above P1 add count x value
  // exactly; pass 2 (and 3) then have nothing to do
  bool skip = false;
  if constexpr (TK<DT>::BYTES == 2) skip = hit && k > 0 && __ldcg(&st->lowor) == 0 && __ldcg(&st->inexact) == 0;
  if (skip) {
    for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
    __syncthreads();
    for (int b = d + 1 + threadIdx.x; b < TK_WIN * TK_NB1; b += TB) {
      const unsigned long long cnt = __ldcg(&st->hist1[b]);
      if (cnt) {
        int sc;
        const float v = key_value(((Plo << 11) + (uint32_t)b) << 10, sc);
        digits_of_n(lim, v, sc, cnt);
      }
    }
    __syncthreads();
    for (int j = threadIdx.x; j < NLIMB; j += TB)
      if (lim[j]) atomicAdd(reinterpret_cast<unsigned long long*>(&st->limbs[j]), (unsigned long long)lim[j]);
  }
  if (threadIdx.x == 0) {
    st->nfin = nfin;
    st->k = k;
    st->ok = hit ? 1u : 0u;
    if (hit && k > 0) {
      const uint32_t P1 = (Plo << 11) + d;
      st->P1 = P1;
      st->P0 = P1 >> 11;
      st->krem = krem;
      if (skip) {
        st->hist2[0] = __ldcg(&st->hist1[d]);  // P1's bucket: every key is P1 2^10 (last digit 0)
        st->T = P1 << 10;
        st->skip2 = 1u;
      }
    }
    st->done[1] = 0;
  }
}

// Only when the sampled window missed: the exact digit of key >> 21 (k and
// the finite count are exact already), which becomes a window of one digit;
// the accumulators of the missed pass cleared.
template <int DT>
__global__ void __launch_bounds__(TB) topk_pass0(TopkParams p) {
  __shared__ uint32_t h[TK_NB0];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (st->ok) return;
  for (int b = threadIdx.x; b < TK_NB0; b += TB) h[b] = 0;
  __syncthreads();
  RunCount rc;
  tk_visit<DT>(p, [&](uint32_t G, uint32_t C) {
    uint32_t key = raw_key<DT>(G, C);
    if (key >= KEY_OVF) {
      if (!tk_finite<DT>(G, C)) return;
      key = tk_key(tk_f32<DT>(G), tk_f32<DT>(C));
    }
    rc.add(h, key >> 21);
  });
  rc.flush(h);
  if (!pass_end(h, TK_NB0, st->hist0, nullptr, st, 0, &last_s)) return;
  unsigned long long krem = __ldcg(&st->k);
  unsigned d;
  select_digit<TK_NB0 / TB>(st->hist0, krem, d);
  for (int b = threadIdx.x; b < TK_WIN * TK_NB1; b += TB) st->hist1[b] = 0;
  for (int j = threadIdx.x; j < NLIMB; j += TB) st->limbs[j] = 0;
  if (threadIdx.x == 0) {
    st->Plo = st->Phi = d;
    st->above = st->nonfin = 0;
    st->done[0] = 0;
  }
}

template <int DT>
__global__ void __launch_bounds__(TB) topk_pass2(TopkParams p) {
  __shared__ uint32_t h[TK_NB2];
  __shared__ long long lim[NLIMB];
  __shared__ typename QT<DT>::T ring[(TB / 32) * ring_cap<DT>()];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (st->k == 0 || st->skip2) return;
  for (int b = threadIdx.x; b < TK_NB2; b += TB) h[b] = 0;
  for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
  __syncthreads();
  // the window's pairs above P1 (those above the window are summed already)
  const uint32_t Phi = st->Phi, P1 = st->P1;
  const uint32_t span = ((Phi + 1) << 11) - P1;  // values of key >> 10 from P1 to the end of the window
  ExactAcc acc(P1 >= (KEY_OVF >> 10) ? NO_FAST : max((int)(P1 >> 13), 1), lim);
  RunCount rc;
  // queued: the pairs to sum, those of P1's range (for their rounding
  // errors) and every pair with a NaN, an infinity or an overflow; a zero
  // key (|d| = 0 exactly) is only counted, here
  tk_filtered<DT>(
      p, ring + (threadIdx.x >> 5) * ring_cap<DT>(),
      [&](uint32_t G, uint32_t C) {
        const uint32_t u = raw_key<DT>(G, C);
        if (u == 0) {
          if (P1 == 0) rc.add(h, 0);
          return false;
        }
        return u >= KEY_OVF || (u >> 10) - P1 < span;
      },
      [&](uint32_t G, uint32_t C) {
        if (!tk_finite<DT>(G, C)) return;
        const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
        const uint32_t key = tk_key(gf, cf), k1 = key >> 10;
        if ((key >> 21) > Phi || k1 < P1) return;
        if (k1 > P1) {
          acc.add(gf, cf);
          return;
        }
        rc.add(h, key & 0x3FFu);
        float hi, lo;
        int sc;
        tk_exact(gf, cf, hi, lo, sc);
        if (lo != 0.0f) {
          const unsigned i = atomicAdd(&st->nlist, 1u);
          if (i < TK_LCAP) p.list[i] = TopkListEntry{lo, key};
        }
      });
  rc.flush(h);
  acc.flush();
  if (!pass_end(h, TK_NB2, st->hist2, lim, st, 2, &last_s)) return;
  unsigned long long krem = __ldcg(&st->krem);
  unsigned d;
  select_digit<TK_NB2 / TB>(st->hist2, krem, d);
  if (threadIdx.x == 0) {
    st->T = (P1 << 10) | d;
    st->krem = krem;
    st->done[2] = 0;
  }
}

__device__ __forceinline__ uint32_t order_key(float x) {
  const uint32_t b = __float_as_uint(x);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float from_order_key(uint32_t u) {
  return __uint_as_float((u & 0x80000000u) ? (u & 0x7FFFFFFFu) : ~u);
}

// Only when the list of the last pass overflowed: the pairs with key >> 10 =
// P1 above T summed exactly, and T's pairs whose |d| is not a float32 listed.
template <int DT>
__global__ void __launch_bounds__(TB) topk_pass3(TopkParams p) {
  __shared__ long long lim[NLIMB];
  __shared__ typename QT<DT>::T ring[(TB / 32) * ring_cap<DT>()];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (st->k == 0 || st->skip2 || st->nlist <= TK_LCAP) return;
  for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
  __syncthreads();
  const uint32_t P1 = st->P1, T = st->T;
  const uint32_t span = ((P1 + 1) << 10) - T;  // keys from T to the end of P1's range
  ExactAcc acc(T >= KEY_OVF ? NO_FAST : max((int)(T >> 23), 1), lim);
  tk_filtered<DT>(
      p, ring + (threadIdx.x >> 5) * ring_cap<DT>(),
      [&](uint32_t G, uint32_t C) {
        const uint32_t u = raw_key<DT>(G, C);
        return u >= KEY_OVF || u - T < span;
      },
      [&](uint32_t G, uint32_t C) {
        if (!tk_finite<DT>(G, C)) return;
        const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
        const uint32_t key = tk_key(gf, cf);
        if ((key >> 10) != P1 || key < T) return;
        if (key > T) {
          acc.add(gf, cf);
          return;
        }
        float hi, lo;
        int sc;
        tk_exact(gf, cf, hi, lo, sc);
        if (lo != 0.0f) {
          const unsigned i = atomicAdd(&st->nlist2, 1u);
          if (i < TK_LCAP) p.list[i] = TopkListEntry{lo, key};
        }
      });
  acc.flush();
  if (pass_end(nullptr, 0, nullptr, lim, st, 2, &last_s) && threadIdx.x == 0) st->done[2] = 0;
}

// Only when pass 3 found more than TK_LCAP pairs of T's bucket whose |d| is
// not a float32 value, so that their rounding errors lo (|d| = (vT + lo)
// 2^scT) cannot all be listed: the m largest lo of the bucket (m = krem, its
// pairs inside the top k), by a radix select on order_key(lo) in two 16-bit
// digits.  Pairs whose |d| is a float32 value take part with lo = 0.
// Pass 4 counts the bucket by the high digit; the last CTA selects it.
template <int DT>
__global__ void __launch_bounds__(TB) topk_pass4(TopkParams p) {
  __shared__ typename QT<DT>::T ring[(TB / 32) * ring_cap<DT>()];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (st->k == 0 || st->skip2 || st->nlist2 <= TK_LCAP) return;
  const uint32_t T = st->T;
  tk_filtered<DT>(
      p, ring + (threadIdx.x >> 5) * ring_cap<DT>(),
      [&](uint32_t G, uint32_t C) {
        const uint32_t u = raw_key<DT>(G, C);
        return u >= KEY_OVF || u == T;
      },
      [&](uint32_t G, uint32_t C) {
        if (!tk_finite<DT>(G, C)) return;
        const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
        if (tk_key(gf, cf) != T) return;
        float hi, lo;
        int sc;
        tk_exact(gf, cf, hi, lo, sc);
        atomicAdd(&st->histl[0][order_key(lo) >> 16], 1ull);
      });
  if (!pass_end(nullptr, 0, nullptr, nullptr, st, 2, &last_s)) return;
  unsigned long long krem = __ldcg(&st->krem);
  unsigned d;
  select_digit<TK_NBL / TB>(st->histl[0], krem, d);
  if (threadIdx.x == 0) {
    st->dl[0] = d;
    st->kreml[0] = krem;
    st->done[2] = 0;
  }
}

// Pass 5: the bucket's lo above the high digit summed exactly, those at it
// counted by the low digit; the last CTA selects the low digit.  Every bin of
// the low digit stands for one float32 value of lo.
template <int DT>
__global__ void __launch_bounds__(TB) topk_pass5(TopkParams p) {
  __shared__ typename QT<DT>::T ring[(TB / 32) * ring_cap<DT>()];
  __shared__ long long lim[NLIMB];
  __shared__ unsigned last_s;
  pdl_wait();
  pdl_trigger();
  TopkState* st = p.st;
  if (st->k == 0 || st->skip2 || st->nlist2 <= TK_LCAP) return;
  for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
  __syncthreads();
  const uint32_t T = st->T, dh = st->dl[0];
  int scT;
  key_value(T, scT);
  tk_filtered<DT>(
      p, ring + (threadIdx.x >> 5) * ring_cap<DT>(),
      [&](uint32_t G, uint32_t C) {
        const uint32_t u = raw_key<DT>(G, C);
        return u >= KEY_OVF || u == T;
      },
      [&](uint32_t G, uint32_t C) {
        if (!tk_finite<DT>(G, C)) return;
        const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
        if (tk_key(gf, cf) != T) return;
        float hi, lo;
        int sc;
        tk_exact(gf, cf, hi, lo, sc);
        const uint32_t u = order_key(lo);
        if ((u >> 16) > dh) digits_of(lim, lo, scT);
        else if ((u >> 16) == dh) atomicAdd(&st->histl[1][u & 0xFFFFu], 1ull);
      });
  if (!pass_end(nullptr, 0, nullptr, lim, st, 2, &last_s)) return;
  unsigned long long krem = __ldcg(&st->kreml[0]);
  unsigned d;
  select_digit<TK_NBL / TB>(st->histl[1], krem, d);
  if (threadIdx.x == 0) {
    st->dl[1] = d;
    st->kreml[1] = krem;
    st->done[2] = 0;
  }
}

// The P1 range, T's bucket, the rounding, the output; the state cleared for
// the next call.  One CTA.
__global__ void __launch_bounds__(TB) topk_finalize(TopkParams p) {
  pdl_wait();
  TopkState* st = p.st;
  __shared__ long long lim[NLIMB];
  const int tid = threadIdx.x;
  const unsigned long long k = st->k;
  peat_topk_t r;
  r.n_finite = st->nfin;
  r.k = k;
  r.threshold = r.sum = r.mean = 0.0;
  r.exact = 1;  // every field is exact as defined, always
  r.reserved = 0;
  if (k > 0) {
    for (int j = tid; j < NLIMB; j += TB) lim[j] = st->limbs[j];
    __syncthreads();
    const uint32_t T = st->T, P1 = st->P1, d2 = T & 0x3FFu;
    const unsigned long long m = st->krem, nbT = st->hist2[d2];
    const bool ovf = st->nlist > TK_LCAP;
    const bool radix = ovf && st->nlist2 > TK_LCAP;  // T's bucket resolved by passes 4 and 5
    const unsigned L = radix ? 0u : ovf ? st->nlist2 : st->nlist;
    int scT;
    const float vT = key_value(T, scT);
    if (!ovf) {
      // keys of the P1 range above T: each one float32 value, count copies
      for (unsigned b = d2 + 1 + tid; b < (unsigned)TK_NB2; b += TB) {
        int sc;
        const float v = key_value((P1 << 10) | b, sc);
        digits_of_n(lim, v, sc, st->hist2[b]);
      }
      // their rounding errors
      for (unsigned i = tid; i < L; i += TB) {
        const TopkListEntry e = p.list[i];
        if (e.key > T) digits_of(lim, e.lo, e.key >= KEY_OVF ? 1 : 0);
      }
    }
    if (tid == 0) digits_of_n(lim, vT, scT, m);
    // T's bucket: its pairs are vT + lo (times 2^scT); the m largest lo count,
    // where the listed pairs carry their lo and the other nbT - LT pairs lo = 0
    unsigned lt = 0;
    for (unsigned i = tid; i < L; i += TB) lt += p.list[i].key == T ? 1u : 0u;
    const unsigned long long LT = block_sum(lt);
    float vstar = 0.0f;
    if (radix) {
      // the bucket's lo above the selected low digit: one float32 value per
      // bin; the m-th largest lo is the selected bin's value
      const uint32_t dh = st->dl[0], dlow = st->dl[1];
      for (unsigned b = dlow + 1 + tid; b < (unsigned)TK_NBL; b += TB) {
        const unsigned long long c = st->histl[1][b];
        if (c) digits_of_n(lim, from_order_key((dh << 16) | b), scT, c);
      }
      vstar = from_order_key((dh << 16) | dlow);
      if (tid == 0) digits_of_n(lim, vstar, scT, st->kreml[1]);
    } else if (LT > 0) {
      const unsigned long long Z = nbT - LT;
      // u*: the largest order key with count(order key >= u*) >= m
      uint32_t u = 0;
      for (int bit = 31; bit >= 0; bit--) {
        const uint32_t cand = u | (1u << bit);
        unsigned c = 0;
        for (unsigned i = tid; i < L; i += TB) {
          const TopkListEntry e = p.list[i];
          c += (e.key == T && order_key(e.lo) >= cand) ? 1u : 0u;
        }
        const unsigned long long tot = block_sum(c) + (cand <= 0x80000000u ? Z : 0ull);
        if (tot >= m) u = cand;
      }
      vstar = from_order_key(u);
      unsigned c = 0;
      for (unsigned i = tid; i < L; i += TB) {
        const TopkListEntry e = p.list[i];
        if (e.key == T && order_key(e.lo) > u) {
          c++;
          digits_of(lim, e.lo, scT);
        }
      }
      const unsigned long long gt = block_sum(c) + (u < 0x80000000u ? Z : 0ull);
      if (tid == 0) digits_of_n(lim, vstar, scT, m - gt);
    }
    __syncthreads();
    __shared__ double mean_s;
    r.threshold = __dadd_rn((double)vT, (double)vstar) * (scT ? 2.0 : 1.0);
    if (tid == 0) r.sum = limbs_to_double(lim);
    if (tid == 32) mean_s = limbs_div_rn(lim, k);
    __syncthreads();
    r.mean = mean_s;
  }
  if (tid == 0) *p.out = r;
  __syncthreads();
  // clear the state
  for (int j = tid; j < TK_NB0; j += TB) st->hist0[j] = 0;
  for (int j = tid; j < TK_WIN * TK_NB1; j += TB) st->hist1[j] = 0;
  for (int j = tid; j < TK_NB2; j += TB) st->hist2[j] = 0;
  for (int j = tid; j < NLIMB; j += TB) st->limbs[j] = 0;
  if (st->nlist > TK_LCAP && st->nlist2 > TK_LCAP)  // the radix passes ran: clear their counts
    for (int j = tid; j < 2 * TK_NBL; j += TB) (&st->histl[0][0])[j] = 0;
  __syncthreads();
  if (tid == 0) {
    st->nonfin = st->above = st->nfin = st->k = st->krem = 0;
    st->kreml[0] = st->kreml[1] = 0;
    st->dl[0] = st->dl[1] = 0;
    st->Plo = st->Phi = st->P0 = st->P1 = st->T = 0;
    st->ok = 0;
    st->nlist = st->nlist2 = 0;
    st->lowor = st->inexact = st->skip2 = 0;
  }
}

template <class K>
int occ(K kernel) {
  int b = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, TB, 0) != cudaSuccess) return 1;
  return b;
}

template <int DT>
int ctas_per_sm_t() {
  const int a = std::min(occ(topk_pass1<DT, false>), occ(topk_pass1<DT, true>));
  const int b = std::min(std::min(occ(topk_pass0<DT>), occ(topk_pass2<DT>)),
                         std::min(occ(topk_pass3<DT>), std::min(occ(topk_pass4<DT>), occ(topk_pass5<DT>))));
  return std::max(1, std::min(a, b));
}

template <int DT>
cudaError_t launch_t(const TopkParams& p, int nctas, cudaStream_t s) {
  // one warp per run of 32 vectors (or per 32 single pairs)
  const int64_t units = p.nvec > 0 ? std::min<int64_t>((p.nvec + 31) / 32, TK_SAMPLE / (32 * TK<DT>::VEC))
                                   : (std::min<int64_t>(p.n, TK_SAMPLE) + 31) / 32;
  const int sctas = (int)std::max<int64_t>(1, std::min<int64_t>(nctas, (units + TB / 32 - 1) / (TB / 32)));
  // the sample waits for everything before it on the stream; each later pass
  // is a programmatic dependent of the one before (its launch overlaps the
  // previous pass, its first access waits for it), which hides the launch
  // latency of the passes that find nothing to do
  topk_sample<DT><<<sctas, TB, 0, s>>>(p);
  cudaError_t e = cudaGetLastError();
  const unsigned g = (unsigned)nctas;
  if (e == cudaSuccess) e = launch_dependent(topk_pass1<DT, false>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass0<DT>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass1<DT, true>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass2<DT>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass3<DT>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass4<DT>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_pass5<DT>, g, TB, 0, s, p);
  if (e == cudaSuccess) e = launch_dependent(topk_finalize, 1u, TB, 0, s, p);
  return e;
}

}  // namespace

int topk_max_ctas(int nsm) {
  static const int per_sm = [] {
    const int v = std::min(ctas_per_sm_t<PEAT_F32>(),
                           std::min(ctas_per_sm_t<PEAT_F16>(), ctas_per_sm_t<PEAT_BF16>()));
    cudaGetLastError();
    return v;
  }();
  return std::max(1, per_sm * nsm);
}

cudaError_t launch_topk(int dtype, const TopkParams& p, int nctas, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return launch_t<PEAT_F32>(p, nctas, s);
    case PEAT_F16: return launch_t<PEAT_F16>(p, nctas, s);
    case PEAT_BF16: return launch_t<PEAT_BF16>(p, nctas, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t register_digit_status_topk(unsigned int* word) { return set_digit_status_here(word); }

}  // namespace peat
