// torch.isclose pass counts over a grid of tolerances (Section III-A, whose
// Fig. 5 reports the share of output elements isclose accepts for FP16-FP32
// and FP32-FP64 pairs as rtol and atol vary): for every rtol_i (ascending)
// and atol_j, the number of pairs the compare classes EXACT or WITHIN_TOL
// under that tolerance, i.e. both operands the same NaN/infinity class or
// |c - g| <= atol_j + rtol_i |g| exactly.  One read of both tensors.
//
// Per pair and atol_j, the first rtol index i* that accepts the pair (0 for
// an EXACT pair, nr for one no tolerance accepts) comes from a binary search
// (acceptance grows with rtol); each test is one fma with a float32 margin,
// and the integer digits of a - atol - rtol |g| decide the rare close calls.
// A warp counts cell (i, j) as the population of the ballot i*_j <= i; lane
// c % 32 keeps cell c's count in a register.
#include <cuda_fp16.h>

#include <cstdint>

#include "exact.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

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

template <int DT>
__device__ __forceinline__ float ic_f32(uint32_t r) {
  if constexpr (DT == PEAT_F32) return __uint_as_float(r);
  else if constexpr (DT == PEAT_BF16) return __uint_as_float(r << 16);
  else return __half2float(__ushort_as_half((unsigned short)r));
}

template <int DT>
__device__ __forceinline__ uint32_t ic_lane(const uint4& v, int j) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (IC<DT>::BYTES == 4) return w[j];
  else return (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
}

template <int DT>
__device__ __forceinline__ uint32_t ic_load(const void* base, int64_t i) {
  if constexpr (IC<DT>::BYTES == 4) return __ldg(reinterpret_cast<const uint32_t*>(base) + i);
  else return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(base) + i);
}

__device__ __forceinline__ uint4 ic_vec(const void* base, int64_t byte_off) {
  const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(base) + byte_off);
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(q));
  return v;
}

// sign of (hi + lo) 2^sc - atol - rtol ag, exactly (integer digits)
__device__ __noinline__ int excess_sign(float hi, float lo, int sc, float ag, float rtol, float atol) {
  int64_t d[NLIMB];
#pragma unroll
  for (int j = 0; j < NLIMB; j++) d[j] = 0;
  auto add = [&](int j, int64_t v) { d[j] += v; };
  int e;
  if (hi != 0.0f) {
    const uint32_t m = split_float(hi, e);
    for_digits(m, e + sc, false, add);
  }
  if (lo != 0.0f) {
    const uint32_t m = split_float(lo, e);
    for_digits(m, e + sc, lo < 0.0f, add);
  }
  if (atol != 0.0f) {
    const uint32_t m = split_float(atol, e);
    for_digits(m, e, true, add);
  }
  if (rtol != 0.0f && ag != 0.0f) {
    int er, eg;
    const uint32_t mr = split_float(rtol, er), mg = split_float(ag, eg);
    for_digits((uint64_t)mr * mg, er + eg, true, add);
  }
  int64_t carry = 0;
#pragma unroll
  for (int j = 0; j < NLIMB - 1; j++) {
    const int64_t v = d[j] + carry;
    carry = v >> 32;
    d[j] = v & 0xFFFFFFFFll;
  }
  d[NLIMB - 1] += carry;
  if (d[NLIMB - 1] != 0) return d[NLIMB - 1] < 0 ? -1 : 1;
  bool nz = false;
#pragma unroll
  for (int j = 0; j < NLIMB - 1; j++) nz |= d[j] != 0;
  return nz ? 1 : 0;
}

// a = (hi + lo) 2^sc <= atol + rtol ag, exactly
__device__ __forceinline__ bool close_test(float hi, float lo, int sc, float ag, float rtol, float atol) {
  const float thr = __fmaf_rn(rtol, ag, atol);
  if (sc == 0 && hi >= 1e-30f && thr >= 1e-30f) {
    // |lo| <= 2^-24 hi and thr is within 2^-24 of the exact bound: margins of 2^-21
    if (__fmul_rn(hi, 1.0000005f) < __fmul_rn(thr, 0.9999995f)) return true;
    if (__fmul_rn(hi, 0.9999995f) > __fmul_rn(thr, 1.0000005f)) return false;
  }
  return excess_sign(hi, lo, sc, ag, rtol, atol) <= 0;
}

// |d| = (hi + lo) 2^sc exactly (float32 TwoSum, halved when c - g overflows)
__device__ __forceinline__ void abs_diff(float gf, float cf, float& hi, float& lo, int& sc) {
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

// One pair slot of a warp (every lane calls it; ok: this lane holds a pair):
// the first accepting rtol index per atol, then one ballot per cell.
template <int DT>
__device__ __forceinline__ void ic_pair(const IscParams& p, const float* R, const float* A, uint32_t G, uint32_t C,
                                        bool ok, uint32_t& c0, uint32_t& c1) {
  using T = IC<DT>;
  const int lane = threadIdx.x & 31;
  // kind 0: accepted by every tolerance; 1: by none; 2: search
  int kind = 1;
  float hi = 0.0f, lo = 0.0f, ag = 0.0f;
  int sc = 0;
  if (ok) {
    if (G == C) {
      kind = 0;
    } else {
      const uint32_t mg = G & T::MAG, mc = C & T::MAG;
      if (mg >= T::INF || mc >= T::INF) {
        // both NaN, or the same infinity (G == C handled above): EXACT
        kind = (mg > T::INF && mc > T::INF) ? 0 : 1;
      } else {
        const float gf = ic_f32<DT>(G), cf = ic_f32<DT>(C);
        if (gf == cf) {
          kind = 0;  // +0 and -0
        } else {
          abs_diff(gf, cf, hi, lo, sc);
          ag = fabsf(gf);
          kind = 2;
        }
      }
    }
  }
  if (__all_sync(0xFFFFFFFFu, kind == 0)) {  // a whole slot of EXACT pairs: every cell
    if (lane < p.ncells) c0 += 32u;
    if (lane + 32 < p.ncells) c1 += 32u;
    return;
  }
  for (int j = 0; j < p.na; j++) {
    int first = kind == 0 ? 0 : p.nr;
    if (kind == 2) {
      int a = 0, b = p.nr;
      while (a < b) {
        const int mid = (a + b) >> 1;
        if (close_test(hi, lo, sc, ag, R[mid], A[j])) b = mid;
        else a = mid + 1;
      }
      first = a;
    }
    for (int i = 0; i < p.nr; i++) {
      const int cell = i * p.na + j;
      const uint32_t cnt = __popc(__ballot_sync(0xFFFFFFFFu, first <= i));
      if (lane == (cell & 31)) {
        if (cell < 32) c0 += cnt;
        else c1 += cnt;
      }
    }
  }
}

template <int DT>
__global__ void __launch_bounds__(TB) isclose_grid(IscParams p) {
  constexpr int VEC = IC<DT>::VEC, B = IC<DT>::BYTES;
  __shared__ float R[ISC_MAX], A[ISC_MAX];
  const int lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < ISC_MAX; i += TB) {
    R[i] = i < p.nr ? p.rtol[i] : 0.0f;
    A[i] = i < p.na ? p.atol[i] : 0.0f;
  }
  __syncthreads();
  const int64_t stride = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  uint32_t c0 = 0, c1 = 0;  // cells lane and lane + 32 (those below ncells)
  // rounds of one vector per thread, whole warps in every round
  for (int64_t v = gt; __any_sync(0xFFFFFFFFu, v < p.nvec); v += stride) {
    const bool ok = v < p.nvec;
    uint4 gv = make_uint4(0, 0, 0, 0), cv = gv;
    if (ok) {
      const int64_t off = (p.p0 + v * VEC) * B;
      gv = ic_vec(p.g, off);
      cv = ic_vec(p.c, off);
    }
#pragma unroll
    for (int j = 0; j < VEC; j++) ic_pair<DT>(p, R, A, ic_lane<DT>(gv, j), ic_lane<DT>(cv, j), ok, c0, c1);
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
    ic_pair<DT>(p, R, A, G, C, ok, c0, c1);
  }
  if (c0 && lane < p.ncells) atomicAdd(p.counts + lane, (unsigned long long)c0);
  if (c1 && lane + 32 < p.ncells) atomicAdd(p.counts + 32 + lane, (unsigned long long)c1);
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
  }
  return cudaErrorInvalidValue;
}

}  // namespace peat
