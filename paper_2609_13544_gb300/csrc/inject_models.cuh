// Element-wise pseudo-error models (the Inject step of Alg. 1 and Alg. 2;
// Section IV-A: FP16 cast; Section II-B: random NaN; plus Gaussian noise,
// bias, BF16 casts and sign flips), one element at a time: shared by the
// injector (in-place passes) and the fused inject-and-compare (the candidate
// generated from the golden tile and never stored).  Randomness is
// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, SC'11), counter = (element
// index, model index, stream tag), key = the seed, so element i of model m
// always sees the same four words.  Gaussian variates use Box-Muller with a
// natural log (atanh series after reduction to [sqrt(1/2), sqrt(2)]) and
// cos(2 pi u) (quadrant reduction on u, Taylor series on [-pi/4, pi/4]),
// every float32 operation written as an explicit correctly rounded intrinsic
// so the sequence of roundings is fixed.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>

#include "peat.h"

namespace peat {
namespace inj {

constexpr uint32_t PHILOX_M0 = 0xD2511F53u, PHILOX_M1 = 0xCD9E8D57u;
constexpr uint32_t PHILOX_W0 = 0x9E3779B9u, PHILOX_W1 = 0xBB67AE85u;
constexpr uint32_t TAG_ELEM = 0x454C454Du;

__device__ __forceinline__ uint4 philox(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; r++) {
    if (r) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    uint32_t lo0 = PHILOX_M0 * c.x, hi0 = __umulhi(PHILOX_M0, c.x);
    uint32_t lo1 = PHILOX_M1 * c.z, hi1 = __umulhi(PHILOX_M1, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

__device__ __forceinline__ float log_series(float x) {
  const float C3 = 0x1.555556p-2f, C5 = 0x1.99999ap-3f, C7 = 0x1.24924ap-3f;
  const float C9 = 0x1.c71c72p-4f, C11 = 0x1.745d18p-4f;
  const float LN2_HI = 0x1.62ep-1f, LN2_LO = 0x1.0bfbe8p-15f, SQRT2 = 0x1.6a09e6p+0f;
  uint32_t b = __float_as_uint(x);
  int e = (int)(b >> 23) - 127;
  float m = __uint_as_float((b & 0x7FFFFFu) | 0x3F800000u);
  if (m > SQRT2) {
    m = __fmul_rn(m, 0.5f);
    e += 1;
  }
  float f = __fdiv_rn(__fsub_rn(m, 1.0f), __fadd_rn(m, 1.0f));
  float f2 = __fmul_rn(f, f);
  float p = __fmaf_rn(f2, C11, C9);
  p = __fmaf_rn(f2, p, C7);
  p = __fmaf_rn(f2, p, C5);
  p = __fmaf_rn(f2, p, C3);
  float tf = __fadd_rn(f, f);
  float tf3 = __fmul_rn(tf, f2);
  float lm = __fmaf_rn(tf3, p, tf);
  float ef = __int2float_rn(e);
  return __fmaf_rn(ef, LN2_HI, __fmaf_rn(ef, LN2_LO, lm));
}

__device__ __forceinline__ float cos_2pi(float u) {
  const float TWO_PI = 0x1.921fb6p+2f;
  const float I2 = 0x1p-1f, I4 = 0x1.555556p-5f, I6 = 0x1.6c16c2p-10f, I8 = 0x1.a01a02p-16f,
              I10 = 0x1.27e4fcp-22f;
  const float I3 = 0x1.555556p-3f, I5 = 0x1.111112p-7f, I7 = 0x1.a01a02p-13f, I9 = 0x1.71de3ap-19f;
  float q = rintf(__fmul_rn(u, 4.0f));
  float r = __fsub_rn(u, __fmul_rn(q, 0.25f));
  float x = __fmul_rn(r, TWO_PI);
  float x2 = __fmul_rn(x, x);
  float cp = __fmaf_rn(x2, -I10, I8);
  cp = __fmaf_rn(x2, cp, -I6);
  cp = __fmaf_rn(x2, cp, I4);
  cp = __fmaf_rn(x2, cp, -I2);
  float cosx = __fmaf_rn(x2, cp, 1.0f);
  float sp = __fmaf_rn(x2, I9, -I7);
  sp = __fmaf_rn(x2, sp, I5);
  sp = __fmaf_rn(x2, sp, -I3);
  float x3 = __fmul_rn(x, x2);
  float sinx = __fmaf_rn(x3, sp, x);
  int j = (int)q & 3;
  return j == 0 ? cosx : (j == 1 ? -sinx : (j == 2 ? -cosx : sinx));
}

__device__ __forceinline__ float normal_from(uint32_t w0, uint32_t w1) {
  float u1 = __fmul_rn(__uint2float_rn((w0 >> 8) + 1u), 0x1p-24f);
  float u2 = __fmul_rn(__uint2float_rn(w1 >> 8), 0x1p-24f);
  float l = log_series(u1);
  float r = __fsqrt_rn(__fmul_rn(-2.0f, l));
  return __fmul_rn(r, cos_2pi(u2));
}

template <int DT>
__device__ __forceinline__ uint32_t ld_bits(const void* p, int64_t i) {
  if constexpr (DT == PEAT_F32) return reinterpret_cast<const uint32_t*>(p)[i];
  else return reinterpret_cast<const unsigned short*>(p)[i];
}
template <int DT>
__device__ __forceinline__ void st_bits(void* p, int64_t i, uint32_t v) {
  if constexpr (DT == PEAT_F32) reinterpret_cast<uint32_t*>(p)[i] = v;
  else reinterpret_cast<unsigned short*>(p)[i] = (unsigned short)v;
}
template <int DT>
__device__ __forceinline__ bool finite_bits(uint32_t b) {
  if constexpr (DT == PEAT_F32) return (b & 0x7FFFFFFFu) < 0x7F800000u;
  else if constexpr (DT == PEAT_F16) return (b & 0x7FFFu) < 0x7C00u;
  else return (b & 0x7FFFu) < 0x7F80u;
}
template <int DT>
__device__ __forceinline__ float bits_to_f32(uint32_t b) {
  if constexpr (DT == PEAT_F32) return __uint_as_float(b);
  else if constexpr (DT == PEAT_F16) return __half2float(__ushort_as_half((unsigned short)b));
  else return __uint_as_float(b << 16);
}
template <int DT>
__device__ __forceinline__ uint32_t f32_to_bits(float y) {  // round to nearest even
  if constexpr (DT == PEAT_F32) return __float_as_uint(y);
  else if constexpr (DT == PEAT_F16) return __half_as_ushort(__float2half_rn(y));
  else return __bfloat16_as_ushort(__float2bfloat16_rn(y));
}


// Model `kind` (index `model` in its list) applied to element i with raw bits
// b; fired: the model changed (or, for NaN/Inf and sign flips, drew) the
// element.  Noise, bias and casts pass NaN and infinities through.
template <int DT>
__device__ __forceinline__ uint32_t apply_model(uint32_t b, int64_t i, int kind, uint32_t model, uint64_t threshold,
                                                float x, uint32_t k0, uint32_t k1, bool& fired) {
  fired = false;
  const bool bern = kind == PEAT_INJ_NAN_INF || kind == PEAT_INJ_SIGNFLIP;
  const bool gauss = kind == PEAT_INJ_REL_GAUSS || kind == PEAT_INJ_ADD_GAUSS;
  uint4 w = make_uint4(0, 0, 0, 0);
  if (bern || gauss) w = philox(make_uint4((uint32_t)i, (uint32_t)((uint64_t)i >> 32), model, TAG_ELEM), k0, k1);
  if (bern) {
    if ((uint64_t)w.x >= threshold) return b;
    fired = true;
    if (kind == PEAT_INJ_SIGNFLIP) return b ^ (DT == PEAT_F32 ? 0x80000000u : 0x8000u);
    const uint32_t sel = w.y >> 30;
    if constexpr (DT == PEAT_F32) return sel < 2 ? 0x7FC00000u : (sel == 2 ? 0x7F800000u : 0xFF800000u);
    else if constexpr (DT == PEAT_F16) return sel < 2 ? 0x7E00u : (sel == 2 ? 0x7C00u : 0xFC00u);
    else return sel < 2 ? 0x7FC0u : (sel == 2 ? 0x7F80u : 0xFF80u);
  }
  if (!finite_bits<DT>(b)) return b;
  fired = true;
  const float v = bits_to_f32<DT>(b);
  float y;
  if (kind == PEAT_INJ_REL_GAUSS) {
    y = __fmul_rn(v, __fmaf_rn(x, normal_from(w.x, w.y), 1.0f));
  } else if (kind == PEAT_INJ_ADD_GAUSS) {
    y = __fmaf_rn(x, normal_from(w.x, w.y), v);
  } else if (kind == PEAT_INJ_BIAS) {
    y = __fmaf_rn(x, fabsf(v), v);
  } else if (kind == PEAT_INJ_CAST_F16_RNE) {
    y = __half2float(__float2half_rn(v));
  } else if (kind == PEAT_INJ_CAST_F16_RTZ) {
    y = __half2float(__float2half_rz(v));
  } else if (kind == PEAT_INJ_CAST_BF16_RNE) {
    y = __bfloat162float(__float2bfloat16_rn(v));
  } else {
    y = __bfloat162float(__float2bfloat16_rz(v));
  }
  return f32_to_bits<DT>(y);
}

}  // namespace inj
}  // namespace peat
