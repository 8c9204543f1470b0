// torch.isclose pass counts over a grid of tolerances (Section III-A, whose
// Fig. 5 reports the share of output elements isclose accepts for FP16-FP32
// and FP32-FP64 pairs as rtol and atol vary): for every rtol_i (ascending)
// and atol_j, the number of pairs the compare classes EXACT or WITHIN_TOL
// under that tolerance, i.e. both operands the same NaN/infinity class or
// |c - g| <= atol_j + rtol_i |g| exactly.  One read of both tensors.
//
// Acceptance grows with rtol and with atol, so a pair is described by
// f(j) = the first rtol index accepting it at atol_j (0 for an EXACT pair,
// nr for none), and f does not increase along the atols sorted ascending.
// Exact pairs are counted per thread.  A warp queues its differing finite
// pairs in shared memory and takes them 32 at a time: each lane finds f(j)
// for the atols in ascending order by a binary search bounded by f(j - 1)
// (each test one fma with a float32 margin; the integer digits of
// a - atol - rtol |g| decide the close calls), and the warp adds each atol's
// f values to a shared histogram, one atomic per distinct value.  Cell
// (i, j) is the histogram's prefix over f <= i.
#include <cuda_fp16.h>

#include <cstdint>

#include "exact.cuh"
#include "peat_internal.h"
#include "tol_exact.cuh"

namespace peat {
namespace {

using namespace tolx;

constexpr int TB = 256;

template <int DT>
struct IC;
template <>
struct IC<PEAT_F32> {
  static constexpr int BYTES = 4, VEC = 4;
  static constexpr uint32_t MAG = 0x7FFFFFFFu, INF = 0x7F800000u;
};
template <>
struct IC<PEAT_F16> {
  static constexpr int BYTES = 2, VEC = 8;
  static constexpr uint32_t MAG = 0x7FFFu, INF = 0x7C00u;
};
template <>
struct IC<PEAT_BF16> {
  static constexpr int BYTES = 2, VEC = 8;
  static constexpr uint32_t MAG = 0x7FFFu, INF = 0x7F80u;
};
template <>
struct IC<PEAT_F8E5M2> {  // IEEE-like: infinities and NaNs at the all-ones exponent
  static constexpr int BYTES = 1, VEC = 16;
  static constexpr uint32_t MAG = 0x7Fu, INF = 0x7Cu;
};
template <>
struct IC<PEAT_F8E4M3> {  // no infinities: 0x7F (either sign) is the only NaN
  static constexpr int BYTES = 1, VEC = 16;
  static constexpr uint32_t MAG = 0x7Fu, INF = 0x7Fu;
};

// magnitude bits: not finite / NaN
template <int DT>
__device__ __forceinline__ bool ic_nonfinite(uint32_t m) { return m >= IC<DT>::INF; }
template <int DT>
__device__ __forceinline__ bool ic_nan(uint32_t m) {
  if constexpr (DT == PEAT_F8E4M3) return m == 0x7Fu;
  else return m > IC<DT>::INF;
}

// the value of a finite pattern (exact in float32)
template <int DT>
__device__ __forceinline__ float ic_f32(uint32_t r) {
  if constexpr (DT == PEAT_F32) {
    return __uint_as_float(r);
  } else if constexpr (DT == PEAT_BF16) {
    return __uint_as_float(r << 16);
  } else if constexpr (DT == PEAT_F16) {
    return __half2float(__ushort_as_half((unsigned short)r));
  } else if constexpr (DT == PEAT_F8E5M2) {
    return __half2float(__ushort_as_half((unsigned short)(r << 8)));  // the top byte of a binary16
  } else {
    // E4M3: exponent bias 7, 3 fraction bits; subnormals m 2^-9
    const uint32_t e = (r >> 3) & 0xFu, m = r & 7u;
    const float v = e ? __uint_as_float(((e + 120u) << 23) | (m << 20)) : __fmul_rn(__uint2float_rn(m), 0x1p-9f);
    return (r & 0x80u) ? -v : v;
  }
}

template <int DT>
__device__ __forceinline__ uint32_t ic_lane(const uint4& v, int j) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (IC<DT>::BYTES == 4) return w[j];
  else if constexpr (IC<DT>::BYTES == 2) return (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
  else return (w[j >> 2] >> (8 * (j & 3))) & 0xFFu;
}

template <int DT>
__device__ __forceinline__ uint32_t ic_load(const void* base, int64_t i) {
  if constexpr (IC<DT>::BYTES == 4) return __ldg(reinterpret_cast<const uint32_t*>(base) + i);
  else if constexpr (IC<DT>::BYTES == 2) return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(base) + i);
  else return (uint32_t)__ldg(reinterpret_cast<const unsigned char*>(base) + i);
}

__device__ __forceinline__ uint4 ic_vec(const void* base, int64_t byte_off) {
  const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(base) + byte_off);
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(q));
  return v;
}

constexpr int NW = TB / 32;
constexpr int QCAP = 64;  // a warp's queue: at most 31 left over plus 32 new pairs
constexpr int NBIN = 2 * ISC_MAX;  // na (nr + 1) <= nr na + na <= 128

struct QEntry {
  float hi, lo, ag;
  int sc;
};

struct IscSmem {
  float R[ISC_MAX], A[ISC_MAX];  // rtols ascending, atols ascending
  unsigned H[NBIN];              // H[j (nr + 1) + f]: pairs whose first accepting rtol at atol j is f
  QEntry q[NW][QCAP];
};

// The lane's pair: kind 0 accepted by every tolerance (EXACT), 1 by none,
// 2 finite and different: |c - g| = (hi + lo) 2^sc, ag = |g|.
template <int DT>
__device__ __forceinline__ int classify(uint32_t G, uint32_t C, float& hi, float& lo, int& sc, float& ag) {
  using T = IC<DT>;
  if (G == C) return 0;
  const uint32_t mg = G & T::MAG, mc = C & T::MAG;
  if (ic_nonfinite<DT>(mg) || ic_nonfinite<DT>(mc)) return (ic_nan<DT>(mg) && ic_nan<DT>(mc)) ? 0 : 1;  // both NaN: EXACT
  const float gf = ic_f32<DT>(G), cf = ic_f32<DT>(C);
  if (gf == cf) return 0;  // +0 and -0
  abs_diff(gf, cf, hi, lo, sc);
  ag = fabsf(gf);
  return 2;
}

// One batch of the warp's queue: lane takes entry e (valid: it holds one).
__device__ __forceinline__ void run_batch(const IscParams& p, IscSmem& sm, const QEntry& e, bool valid) {
  const int nb = p.nr + 1;
  int prev = valid ? p.nr : 0;  // f(j - 1); invalid lanes carry 0 and add nothing
  for (int j = 0; j < p.na; j++) {
    const unsigned vmask = __ballot_sync(0xFFFFFFFFu, valid && prev > 0);
    if (vmask == 0u) {
      // every valid lane is accepted at rtol_0 from here on: f = 0 for the remaining atols
      const int nvalid = __popc(__ballot_sync(0xFFFFFFFFu, valid));
      if ((threadIdx.x & 31) == 0)
        for (int jj = j; jj < p.na; jj++) atomicAdd(&sm.H[jj * nb], (unsigned)nvalid);
      return;
    }
    int f = prev;
    if (valid && prev > 0) {
      int a = 0, b = prev;
      const float at = sm.A[j];
      while (a < b) {
        const int mid = (a + b) >> 1;
        if (close_test(e.hi, e.lo, e.sc, e.ag, sm.R[mid], at)) b = mid;
        else a = mid + 1;
      }
      f = a;
    }
    prev = f;
    const int key = valid ? f : -1;
    const unsigned grp = __match_any_sync(0xFFFFFFFFu, key);
    if (valid && (threadIdx.x & 31) == __ffs(grp) - 1) atomicAdd(&sm.H[j * nb + f], (unsigned)__popc(grp));
  }
}

// Queue the lane's pair if it needs a search; take a batch once 32 wait.
// Every lane of the warp calls it (ok: this lane holds a pair).
template <int DT>
__device__ __forceinline__ void ic_pair(const IscParams& p, IscSmem& sm, uint32_t G, uint32_t C, bool ok, int& qn,
                                        uint32_t& nexact) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float hi = 0.0f, lo = 0.0f, ag = 0.0f;
  int sc = 0;
  const int kind = ok ? classify<DT>(G, C, hi, lo, sc, ag) : 1;
  nexact += kind == 0;
  const unsigned m = __ballot_sync(0xFFFFFFFFu, kind == 2);
  if (m == 0u) return;
  if (kind == 2) sm.q[warp][qn + __popc(m & ((1u << lane) - 1u))] = QEntry{hi, lo, ag, sc};
  qn += __popc(m);
  if (qn < 32) return;
  __syncwarp();
  const QEntry e = sm.q[warp][lane];
  __syncwarp();
  if (lane < qn - 32) sm.q[warp][lane] = sm.q[warp][32 + lane];
  qn -= 32;
  __syncwarp();
  run_batch(p, sm, e, true);
}

template <int DT>
__global__ void __launch_bounds__(TB) isclose_grid(IscParams p) {
  constexpr int VEC = IC<DT>::VEC, B = IC<DT>::BYTES;
  __shared__ IscSmem sm;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < ISC_MAX; i += TB) {
    sm.R[i] = i < p.nr ? p.rtol[i] : 0.0f;
    sm.A[i] = i < p.na ? p.atol[i] : 0.0f;
  }
  for (int i = threadIdx.x; i < NBIN; i += TB) sm.H[i] = 0u;
  __syncthreads();
  const int64_t stride = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  int qn = 0;            // this warp's queue length (the same in every lane)
  uint32_t nexact = 0;   // this thread's EXACT pairs (below 2^32: the host bounds the elements per CTA)
  // rounds of one vector per thread, whole warps in every round
  for (int64_t v = gt; __any_sync(0xFFFFFFFFu, v < p.nvec); v += stride) {
    const bool ok = v < p.nvec;
    uint4 gv = make_uint4(0, 0, 0, 0), cv = gv;
    if (ok) {
      const int64_t off = (p.p0 + v * VEC) * B;
      gv = ic_vec(p.g, off);
      cv = ic_vec(p.c, off);
    }
    if (__all_sync(0xFFFFFFFFu, !ok || (gv.x == cv.x && gv.y == cv.y && gv.z == cv.z && gv.w == cv.w))) {
      nexact += ok ? VEC : 0;  // a warp slot of bitwise-equal vectors
      continue;
    }
#pragma unroll
    for (int j = 0; j < VEC; j++) ic_pair<DT>(p, sm, ic_lane<DT>(gv, j), ic_lane<DT>(cv, j), ok, qn, nexact);
  }
  // elements outside the vector grid, in whole-warp rounds as well
  const int64_t head = p.p0 >= 0 ? p.p0 : p.n, tail = p.p0 >= 0 ? p.p0 + p.nvec * VEC : p.n;
  const int64_t ns = head + (p.n - tail);
  const int64_t wbase = gt - lane;
  for (int64_t r = wbase; r < ns; r += stride) {
    const int64_t idx = r + lane;
    const bool ok = idx < ns;
    uint32_t G = 0, C = 0;
    if (ok) {
      const int64_t i = idx < head ? idx : tail + (idx - head);
      G = ic_load<DT>(p.g, i);
      C = ic_load<DT>(p.c, i);
    }
    ic_pair<DT>(p, sm, G, C, ok, qn, nexact);
  }
  // the rest of the queue
  if (qn > 0) {
    __syncwarp();
    const QEntry e = sm.q[warp][lane < qn ? lane : 0];
    run_batch(p, sm, e, lane < qn);
  }
  // exact pairs: f = 0 at every atol
  const uint32_t ne = __reduce_add_sync(0xFFFFFFFFu, nexact);
  if (lane == 0 && ne)
    for (int j = 0; j < p.na; j++) atomicAdd(&sm.H[j * (p.nr + 1)], ne);
  __syncthreads();
  // cell (i, j) = pairs with f(j) <= i, into the caller's cell order
  for (int c = threadIdx.x; c < p.ncells; c += TB) {
    const int i = c / p.na, j = c - i * p.na;
    unsigned long long cnt = 0;
    for (int f = 0; f <= i; f++) cnt += sm.H[j * (p.nr + 1) + f];
    if (cnt) atomicAdd(p.counts + i * p.na + p.aperm[j], cnt);
  }
}

template <int DT>
cudaError_t launch_t(const IscParams& p, int nctas, cudaStream_t s) {
  isclose_grid<DT><<<nctas, TB, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_isclose(int dtype, const IscParams& p, int nctas, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return launch_t<PEAT_F32>(p, nctas, s);
    case PEAT_F16: return launch_t<PEAT_F16>(p, nctas, s);
    case PEAT_BF16: return launch_t<PEAT_BF16>(p, nctas, s);
    case PEAT_F8E4M3: return launch_t<PEAT_F8E4M3>(p, nctas, s);
    case PEAT_F8E5M2: return launch_t<PEAT_F8E5M2>(p, nctas, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t register_digit_status_isclose(unsigned int* word) { return set_digit_status_here(word); }

}  // namespace peat
