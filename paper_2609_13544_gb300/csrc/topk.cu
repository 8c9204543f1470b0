// Mean of the top errors (Section IV-B-3, "Mean of Top 10% Errors") on sm_103a.
//
// Over the pairs with both operands finite, the k = ceil(n_finite num / den)
// largest |d| = |c - g|: their exact sum and exact mean, rounded once.
//
// key(|d|) is an order-preserving 32-bit key: the bits of RN32(|d|) (RN32 is
// monotone and float bits order like the values), or, when c - g overflows
// float32, the bits of RN32(|d| / 2) plus 2^23 (above every key of the first
// kind).  A radix select over the key -- three streaming passes with 11-, 11-
// and 10-bit digit histograms, each followed by a one-CTA select -- finds the
// key T of the k-th largest |d| and how many of the pairs with key T belong to
// the top k.  A fourth pass adds every |d| above T exactly (integers in units
// of T's float32 step where |d| is a float32 value not far above T, integer
// digits of a fixed-point accumulator otherwise), counts the pairs with key T
// and lists those among them whose |d| is not a float32 value; a one-CTA
// finalize orders that bucket exactly, adds its share and rounds.
#include <cuda_fp16.h>

#include <cstdint>

#include "exact.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

constexpr int TB = 256;  // threads per CTA

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
};
template <>
struct TK<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8;
  static constexpr uint32_t MAG = 0x7FFFu, INF = 0x7F80u;
};

template <int DT>
__device__ __forceinline__ float tk_f32(uint32_t r) {
  if constexpr (DT == PEAT_F32) return __uint_as_float(r);
  else if constexpr (DT == PEAT_BF16) return __uint_as_float(r << 16);
  else return __half2float(__ushort_as_half((unsigned short)r));
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

// |d| = (hi + lo) 2^sc exactly (float32 TwoSum, halved when c - g overflows)
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

// Every pair, in rounds that all threads of the grid run the same number of
// times (so warp-collective work inside f is safe): f(G, C, valid).
template <int DT, class F>
__device__ __forceinline__ void tk_visit(const TopkParams& p, F&& f) {
  constexpr int VEC = TK<DT>::VEC;
  const int64_t nthreads = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  const int64_t rounds = (p.nvec + nthreads - 1) / nthreads;
  for (int64_t r = 0; r < rounds; r++) {
    const int64_t v = r * nthreads + gt;
    const bool ok = v < p.nvec;
    uint4 gv = make_uint4(0, 0, 0, 0), cv = gv;
    if (ok) {
      const int64_t off = (p.p0 + v * VEC) * TK<DT>::BYTES;
      gv = tk_vec(p.g, off);
      cv = tk_vec(p.c, off);
    }
#pragma unroll
    for (int j = 0; j < VEC; j++) f(tk_lane<DT>(gv, j), tk_lane<DT>(cv, j), ok);
  }
  // elements outside the vector grid: [0, head) and [tail, n)
  const int64_t head = p.p0 >= 0 ? p.p0 : p.n, tail = p.p0 >= 0 ? p.p0 + p.nvec * VEC : p.n;
  const int64_t ns = head + (p.n - tail);
  const int64_t srounds = (ns + nthreads - 1) / nthreads;
  for (int64_t r = 0; r < srounds; r++) {
    const int64_t idx = r * nthreads + gt;
    const bool ok = idx < ns;
    uint32_t G = 0, C = 0;
    if (ok) {
      const int64_t i = idx < head ? idx : tail + (idx - head);
      G = tk_load<DT>(p.g, i);
      C = tk_load<DT>(p.c, i);
    }
    f(G, C, ok);
  }
}

// one count for `bin` from every active lane, one shared atomic per distinct bin
__device__ __forceinline__ void hist_add(uint32_t* h, uint32_t bin, bool act) {
  const uint32_t m = __ballot_sync(0xFFFFFFFFu, act);
  if (m == 0u) return;
  if (act) {
    const uint32_t peers = __match_any_sync(m, bin);
    if ((int)(threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&h[bin], (uint32_t)__popc(peers));
  }
}

// digit pass LEVEL (0, 1, 2) of the radix select
template <int DT, int LEVEL>
__global__ void __launch_bounds__(TB) topk_hist(TopkParams p) {
  using T = TK<DT>;
  __shared__ uint32_t h[TK_BINS];
  __shared__ unsigned long long nf_s;
  TopkState* st = p.st;
  if (LEVEL > 0 && st->k == 0) return;  // no finite pair
  for (int b = threadIdx.x; b < TK_BINS; b += TB) h[b] = 0;
  if (threadIdx.x == 0) nf_s = 0;
  __syncthreads();
  const uint32_t prefix = LEVEL > 0 ? st->prefix : 0u;
  uint32_t nf = 0;
  tk_visit<DT>(p, [&](uint32_t G, uint32_t C, bool ok) {
    const bool fin = ok && (G & T::MAG) < T::INF && (C & T::MAG) < T::INF;
    const uint32_t key = fin ? tk_key(tk_f32<DT>(G), tk_f32<DT>(C)) : 0u;
    bool act;
    uint32_t bin;
    if constexpr (LEVEL == 0) {
      act = fin;
      bin = key >> 21;
      nf += fin ? 1u : 0u;
    } else if constexpr (LEVEL == 1) {
      act = fin && (key >> 21) == prefix;
      bin = (key >> 10) & 0x7FFu;
    } else {
      act = fin && (key >> 10) == prefix;
      bin = key & 0x3FFu;
    }
    hist_add(h, bin, act);
  });
  if (LEVEL == 0) {
    const uint32_t w = __reduce_add_sync(0xFFFFFFFFu, nf);
    if ((threadIdx.x & 31) == 0 && w) atomicAdd(&nf_s, (unsigned long long)w);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < TK_BINS; b += TB)
    if (h[b]) atomicAdd(&st->hist[LEVEL][b], (unsigned long long)h[b]);
  if (LEVEL == 0 && threadIdx.x == 0 && nf_s) atomicAdd(&st->nfin, nf_s);
}

// After digit pass `level`: the digit d of the k-th largest key (counting from
// the top, krem to go): count(keys above d within the prefix) < krem <=
// count(keys at or above d).  One CTA.
__global__ void __launch_bounds__(TB) topk_select(TopkParams p, int level) {
  TopkState* st = p.st;
  __shared__ unsigned long long part[TB];
  if (level == 0 && threadIdx.x == 0) {
    const unsigned __int128 prod = (unsigned __int128)st->nfin * p.num;
    const unsigned long long k = (unsigned long long)((prod + p.den - 1) / p.den);
    st->k = k;
    st->krem = k;
  }
  __syncthreads();
  if (st->k == 0) return;
  const unsigned long long krem = st->krem;
  constexpr int PER = TK_BINS / TB;  // bins per thread, thread t owns [t PER, t PER + PER)
  const unsigned long long* h = st->hist[level];
  unsigned long long mine = 0;
#pragma unroll
  for (int j = 0; j < PER; j++) mine += h[threadIdx.x * PER + j];
  part[threadIdx.x] = mine;
  __syncthreads();
  // counts strictly above this thread's bins (threads with higher bins), a serial
  // suffix over 256 partial sums per thread is cheap for one CTA
  unsigned long long above = 0;
  for (int t = threadIdx.x + 1; t < TB; t++) above += part[t];
  for (int j = PER - 1; j >= 0; j--) {
    const int b = threadIdx.x * PER + j;
    const unsigned long long hb = h[b];
    if (above < krem && krem <= above + hb) {
      const int bits = level == 2 ? 10 : 11;
      st->prefix = level == 0 ? (unsigned int)b : (st->prefix << bits) | (unsigned int)b;
      st->krem = krem - above;
    }
    above += hb;
  }
}

// the exact sum of the |d| above T; the pairs with key T counted and listed
template <int DT>
__global__ void __launch_bounds__(TB) topk_sum(TopkParams p) {
  using T = TK<DT>;
  TopkState* st = p.st;
  __shared__ long long lim[NLIMB];
  __shared__ unsigned long long nb_s;
  if (st->k == 0) return;
  for (int j = threadIdx.x; j < NLIMB; j += TB) lim[j] = 0;
  if (threadIdx.x == 0) nb_s = 0;
  __syncthreads();
  const uint32_t K = st->prefix;
  const bool Ksc = K >= 0x7F800000u;                        // T itself overflowed float32
  const int eT = Ksc ? 255 : max((int)(K >> 23), 1);         // T's binade (subnormal: 1)
  // |d| a float32 value with binade e: |d| = m 2^(e - 150) = (m << (e - eT)) 2^(eT - 150)
  uint64_t V = 0;  // this thread's sum, in units of 2^(eT - 150); terms below 2^40
  uint32_t nb = 0;
  auto exact_digits = [&](float x, int sc) {
    if (x == 0.0f) return;
    int e;
    const uint32_t m = split_float(x, e);
    for_digits(m, e + sc, x < 0.0f, [&](int j, int64_t v) { atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v); });
  };
  tk_visit<DT>(p, [&](uint32_t G, uint32_t C, bool ok) {
    if (!ok || (G & T::MAG) >= T::INF || (C & T::MAG) >= T::INF) return;
    const float gf = tk_f32<DT>(G), cf = tk_f32<DT>(C);
    const uint32_t key = tk_key(gf, cf);
    if (key < K) return;
    float hi, lo;
    int sc;
    tk_exact(gf, cf, hi, lo, sc);
    if (key == K) {
      nb++;
      if (lo != 0.0f) {
        const unsigned idx = atomicAdd(&st->nlist, 1u);
        if (idx < TK_LCAP) p.list[idx] = TopkListEntry{lo, sc};
      }
      return;
    }
    if (!Ksc && sc == 0 && lo == 0.0f) {
      const uint32_t b = __float_as_uint(hi);
      const int e = max((int)(b >> 23), 1);
      const int sh = e - eT;  // >= 0: hi > T
      if (sh <= 16) {
        V += (uint64_t)((b & 0x7FFFFFu) | ((b >> 23) ? 0x800000u : 0u)) << sh;
        return;
      }
    }
    exact_digits(hi, sc);
    exact_digits(lo, sc);
  });
  // the integer sums: warp sums in 128 bits, added as digits
  {
    uint64_t lo32 = V & 0xFFFFFFFFull, hi32 = V >> 32;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo32 += __shfl_xor_sync(0xFFFFFFFFu, lo32, o);
      hi32 += __shfl_xor_sync(0xFFFFFFFFu, hi32, o);
    }
    const uint32_t w = __reduce_add_sync(0xFFFFFFFFu, nb);
    if ((threadIdx.x & 31) == 0) {
      const unsigned __int128 S = (unsigned __int128)lo32 + ((unsigned __int128)hi32 << 32);
      if (S) for_digits(S, eT - 150, false, [&](int j, int64_t v) { atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v); });
      if (w) atomicAdd(&nb_s, (unsigned long long)w);
    }
  }
  __syncthreads();
  for (int j = threadIdx.x; j < NLIMB; j += TB)
    if (lim[j]) atomicAdd(reinterpret_cast<unsigned long long*>(&st->limbs[j]), (unsigned long long)lim[j]);
  if (threadIdx.x == 0 && nb_s) atomicAdd(&st->nbucket, nb_s);
}

// The bucket's share, the rounding, the output; the state cleared for the next
// call.  One CTA.
__global__ void __launch_bounds__(TB) topk_finalize(TopkParams p) {
  TopkState* st = p.st;
  __shared__ long long lim[NLIMB];
  __shared__ float thr_lo;
  const int tid = threadIdx.x;
  const unsigned long long k = st->k;
  if (k > 0) {
    for (int j = tid; j < NLIMB; j += TB) lim[j] = st->limbs[j];
    if (tid == 0) thr_lo = 0.0f;
    __syncthreads();
    const uint32_t K = st->prefix;
    const int scT = K >= 0x7F800000u ? 1 : 0;
    const float hT = __uint_as_float(K - (scT ? (1u << 23) : 0u));  // bucket values: (hT + lo) 2^scT
    const unsigned long long m = st->krem, nb = st->nbucket;
    const unsigned L = min(st->nlist, TK_LCAP);
    // m hT, exactly
    if (tid == 0 && hT != 0.0f) {
      int e;
      const uint32_t mant = split_float(hT, e);
      for_digits((unsigned __int128)mant * m, e + scT, false,
                 [&](int j, int64_t v) { atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v); });
    }
    // listed members (lo != 0) in exact order: rank = listed members with a
    // larger lo, ties by list position; members with lo = 0 sit between the
    // positive and the negative ones
    const unsigned long long Z = nb - L;  // members whose |d| is hT exactly
    for (unsigned i = tid; i < L; i += TB) {
      const float li = p.list[i].lo;
      unsigned r = 0;
      for (unsigned j = 0; j < L; j++) {
        const float lj = p.list[j].lo;
        r += (lj > li || (lj == li && j < i)) ? 1u : 0u;
      }
      const unsigned long long pos = li > 0.0f ? r : r + Z;  // place among all bucket members
      if (pos < m) {
        int e;
        const uint32_t mant = split_float(li, e);
        for_digits(mant, e + scT, li < 0.0f,
                   [&](int j, int64_t v) { atomicAdd(reinterpret_cast<unsigned long long*>(&lim[j]), (unsigned long long)v); });
      }
      if (pos == m - 1) thr_lo = li;
    }
    __syncthreads();
    if (tid == 0) {
      peat_topk_t r;
      r.n_finite = st->nfin;
      r.k = k;
      r.threshold = __dadd_rn((double)hT, (double)thr_lo) * (scT ? 2.0 : 1.0);
      r.sum = limbs_to_double(lim);
      r.mean = limbs_div_rn(lim, k);
      r.exact = st->nlist <= TK_LCAP ? 1u : 0u;
      r.reserved = 0;
      *p.out = r;
    }
  } else if (tid == 0) {
    peat_topk_t r;
    r.n_finite = st->nfin;
    r.k = 0;
    r.threshold = r.sum = r.mean = 0.0;
    r.exact = 1;
    r.reserved = 0;
    *p.out = r;
  }
  __syncthreads();
  // clear the state
  for (int j = tid; j < 3 * TK_BINS; j += TB) (&st->hist[0][0])[j] = 0;
  for (int j = tid; j < NLIMB; j += TB) st->limbs[j] = 0;
  if (tid == 0) {
    st->nfin = st->k = st->krem = st->nbucket = 0;
    st->prefix = 0;
    st->nlist = 0;
  }
}

template <int DT>
cudaError_t launch_t(const TopkParams& p, int nctas, cudaStream_t s) {
  topk_hist<DT, 0><<<nctas, TB, 0, s>>>(p);
  topk_select<<<1, TB, 0, s>>>(p, 0);
  topk_hist<DT, 1><<<nctas, TB, 0, s>>>(p);
  topk_select<<<1, TB, 0, s>>>(p, 1);
  topk_hist<DT, 2><<<nctas, TB, 0, s>>>(p);
  topk_select<<<1, TB, 0, s>>>(p, 2);
  topk_sum<DT><<<nctas, TB, 0, s>>>(p);
  topk_finalize<<<1, TB, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_topk(int dtype, const TopkParams& p, int nctas, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return launch_t<PEAT_F32>(p, nctas, s);
    case PEAT_F16: return launch_t<PEAT_F16>(p, nctas, s);
    case PEAT_BF16: return launch_t<PEAT_BF16>(p, nctas, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace peat
