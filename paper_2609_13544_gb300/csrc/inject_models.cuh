// Element-wise pseudo-error models (the Inject step of Alg. 1 and Alg. 2;
// Section IV-A: FP16 cast; Section II-B: random NaN; plus Gaussian noise,
// bias, BF16 casts and sign flips): shared by the injector (in-place passes)
// and the fused inject-and-compare (the candidate generated from the golden
// tile and never stored).  Randomness is Philox4x32-10 (Salmon, Moraes, Dror
// and Shaw, SC'11) keyed by the seed.  One draw, counter (d, model, tag),
// serves the block of four elements 4d .. 4d+3: element i takes word i mod 4
// (rate models), or the normal of its word pair (Gaussian models: the pair
// (w0, w1) gives elements 4d and 4d+1 the Box-Muller pair r cos, r sin; the
// pair (w2, w3) elements 4d+2 and 4d+3).  A fired NaN/Inf element draws its
// class from a counter of its own.  Box-Muller uses a natural log (atanh
// series after reduction to [sqrt(1/2), sqrt(2)]) and cos/sin(2 pi u)
// (quadrant reduction on u, Taylor series on [-pi/4, pi/4]), every float32
// operation written as an explicit correctly rounded intrinsic so the
// sequence of roundings is fixed.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>
#include <type_traits>

#include "peat.h"

namespace peat {
namespace inj {

constexpr uint32_t PHILOX_M0 = 0xD2511F53u, PHILOX_M1 = 0xCD9E8D57u;
constexpr uint32_t PHILOX_W0 = 0x9E3779B9u, PHILOX_W1 = 0xBB67AE85u;
constexpr uint32_t TAG_ELEM = 0x454C454Du, TAG_CLASS = 0x434C5353u;

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

// sin and cos of 2 pi u, u in [0, 1): u = q/4 + r exactly, x = 2 pi r, then
// (cos, sin)(x + q pi/2) from the two series
__device__ __forceinline__ void sincos_2pi(float u, float& s, float& c) {
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
  const int j = (int)q & 3;
  const bool swap = j & 1, neg_c = j == 1 || j == 2, neg_s = j >= 2;
  const float cc = swap ? sinx : cosx, ss = swap ? cosx : sinx;
  c = neg_c ? -cc : cc;
  s = neg_s ? -ss : ss;
}

// the Box-Muller pair of two words: r cos(2 pi u2), r sin(2 pi u2)
__device__ __forceinline__ void normal_pair(uint32_t w0, uint32_t w1, float& z0, float& z1) {
  float u1 = __fmul_rn(__uint2float_rn((w0 >> 8) + 1u), 0x1p-24f);
  float u2 = __fmul_rn(__uint2float_rn(w1 >> 8), 0x1p-24f);
  float l = log_series(u1);
  float r = __fsqrt_rn(__fmul_rn(-2.0f, l));
  float sn, cs;
  sincos_2pi(u2, sn, cs);
  z0 = __fmul_rn(r, cs);
  z1 = __fmul_rn(r, sn);
}

__device__ __forceinline__ uint4 block_draw(int64_t d, uint32_t model, uint32_t k0, uint32_t k1) {
  return philox(make_uint4((uint32_t)d, (uint32_t)((uint64_t)d >> 32), model, TAG_ELEM), k0, k1);
}
__device__ __forceinline__ uint32_t word_of(const uint4& w, int j) {
  return j == 0 ? w.x : (j == 1 ? w.y : (j == 2 ? w.z : w.w));
}
template <int K>
constexpr bool rate_kind = K == PEAT_INJ_NAN_INF || K == PEAT_INJ_SIGNFLIP;
template <int K>
constexpr bool gauss_kind = K == PEAT_INJ_REL_GAUSS || K == PEAT_INJ_ADD_GAUSS;

// f(std::integral_constant<int, kind>) for an element-wise kind (the kind is
// uniform over a launch or a chunk: one branch, then code without any)
template <class F>
__device__ __forceinline__ void with_kind(int kind, F&& f) {
  switch (kind) {
    case PEAT_INJ_NAN_INF: f(std::integral_constant<int, PEAT_INJ_NAN_INF>{}); break;
    case PEAT_INJ_SIGNFLIP: f(std::integral_constant<int, PEAT_INJ_SIGNFLIP>{}); break;
    case PEAT_INJ_REL_GAUSS: f(std::integral_constant<int, PEAT_INJ_REL_GAUSS>{}); break;
    case PEAT_INJ_ADD_GAUSS: f(std::integral_constant<int, PEAT_INJ_ADD_GAUSS>{}); break;
    case PEAT_INJ_BIAS: f(std::integral_constant<int, PEAT_INJ_BIAS>{}); break;
    case PEAT_INJ_CAST_F16_RNE: f(std::integral_constant<int, PEAT_INJ_CAST_F16_RNE>{}); break;
    case PEAT_INJ_CAST_F16_RTZ: f(std::integral_constant<int, PEAT_INJ_CAST_F16_RTZ>{}); break;
    case PEAT_INJ_CAST_BF16_RNE: f(std::integral_constant<int, PEAT_INJ_CAST_BF16_RNE>{}); break;
    case PEAT_INJ_CAST_BF16_RTZ: f(std::integral_constant<int, PEAT_INJ_CAST_BF16_RTZ>{}); break;
    default: break;
  }
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


// the class of a fired NaN/Inf element: 0, 1 NaN; 2 +Inf; 3 -Inf (rare: out of line)
static __device__ __noinline__ uint32_t nan_class(int64_t i, uint32_t model, uint32_t k0, uint32_t k1) {
  return philox(make_uint4((uint32_t)i, (uint32_t)((uint64_t)i >> 32), model, TAG_CLASS), k0, k1).x >> 30;
}

// Model K (index `model` in its list) applied to element i with raw bits b,
// given the element's word and normal; fired: the model changed (or, for
// NaN/Inf and sign flips, drew) the element.  Noise, bias and casts pass NaN
// and infinities through.
template <int DT, int K>
__device__ __forceinline__ uint32_t model_apply(uint32_t b, int64_t i, uint32_t model, uint64_t threshold, float x,
                                                uint32_t word, float z, uint32_t k0, uint32_t k1, bool& fired) {
  if constexpr (rate_kind<K>) {
    fired = (uint64_t)word < threshold;
    if (!fired) return b;
    if constexpr (K == PEAT_INJ_SIGNFLIP) {
      return b ^ (DT == PEAT_F32 ? 0x80000000u : 0x8000u);
    } else {
      const uint32_t sel = nan_class(i, model, k0, k1);
      if constexpr (DT == PEAT_F32) return sel < 2 ? 0x7FC00000u : (sel == 2 ? 0x7F800000u : 0xFF800000u);
      else if constexpr (DT == PEAT_F16) return sel < 2 ? 0x7E00u : (sel == 2 ? 0x7C00u : 0xFC00u);
      else return sel < 2 ? 0x7FC0u : (sel == 2 ? 0x7F80u : 0xFF80u);
    }
  } else {
    fired = finite_bits<DT>(b);
    const float v = bits_to_f32<DT>(b);
    float y;
    if constexpr (K == PEAT_INJ_REL_GAUSS) y = __fmul_rn(v, __fmaf_rn(x, z, 1.0f));
    else if constexpr (K == PEAT_INJ_ADD_GAUSS) y = __fmaf_rn(x, z, v);
    else if constexpr (K == PEAT_INJ_BIAS) y = __fmaf_rn(x, fabsf(v), v);
    else if constexpr (K == PEAT_INJ_CAST_F16_RNE) y = __half2float(__float2half_rn(v));
    else if constexpr (K == PEAT_INJ_CAST_F16_RTZ) y = __half2float(__float2half_rz(v));
    else if constexpr (K == PEAT_INJ_CAST_BF16_RNE) y = __bfloat162float(__float2bfloat16_rn(v));
    else y = __bfloat162float(__float2bfloat16_rz(v));
    return fired ? f32_to_bits<DT>(y) : b;
  }
}

// One element on its own (its block's draw made for it alone).
template <int DT, int K>
__device__ __forceinline__ uint32_t apply_one(uint32_t b, int64_t i, uint32_t model, uint64_t threshold, float x,
                                              uint32_t k0, uint32_t k1, bool& fired) {
  const int j = (int)(i & 3);
  uint32_t word = 0;
  float z = 0.0f;
  if constexpr (rate_kind<K> || gauss_kind<K>) {
    const uint4 w = block_draw(i >> 2, model, k0, k1);
    word = word_of(w, j);
    if constexpr (gauss_kind<K>) {
      float z0, z1;
      if (j < 2) normal_pair(w.x, w.y, z0, z1);
      else normal_pair(w.z, w.w, z0, z1);
      z = (j & 1) ? z1 : z0;
    }
  }
  return model_apply<DT, K>(b, i, model, threshold, x, word, z, k0, k1, fired);
}

// The same with the kind known only at run time (the rare scalar paths).
template <int DT>
__device__ __forceinline__ uint32_t apply_model(uint32_t b, int64_t i, int kind, uint32_t model, uint64_t threshold,
                                                float x, uint32_t k0, uint32_t k1, bool& fired) {
  uint32_t r = b;
  fired = false;
  with_kind(kind, [&](auto k) { r = apply_one<DT, decltype(k)::value>(b, i, model, threshold, x, k0, k1, fired); });
  return r;
}

// NB whole blocks e[0 .. 4 NB) = elements i0 .. i0 + 4 NB - 1, i0 a multiple
// of 4: the NB draws first, then the normals, then the model, so that the
// blocks' independent chains can overlap.  Returns how many elements fired;
// bit j of *mask (if given) marks element j.
template <int DT, int K, int NB>
__device__ __forceinline__ uint32_t apply_blocks(uint32_t (&e)[4 * NB], int64_t i0, uint32_t model,
                                                 uint64_t threshold, float x, uint32_t k0, uint32_t k1,
                                                 uint32_t* mask = nullptr) {
  uint4 w[NB];
  float z[4 * NB];
#pragma unroll
  for (int q = 0; q < NB; q++)
    w[q] = (rate_kind<K> || gauss_kind<K>) ? block_draw((i0 >> 2) + q, model, k0, k1) : make_uint4(0, 0, 0, 0);
#pragma unroll
  for (int j = 0; j < 4 * NB; j++) z[j] = 0.0f;
  if constexpr (gauss_kind<K>) {
#pragma unroll
    for (int q = 0; q < NB; q++) {
      normal_pair(w[q].x, w[q].y, z[4 * q], z[4 * q + 1]);
      normal_pair(w[q].z, w[q].w, z[4 * q + 2], z[4 * q + 3]);
    }
  }
  uint32_t n = 0, mk = 0;
#pragma unroll
  for (int j = 0; j < 4 * NB; j++) {
    bool f;
    e[j] = model_apply<DT, K>(e[j], i0 + j, model, threshold, x, word_of(w[j >> 2], j & 3), z[j], k0, k1, f);
    n += f;
    mk |= (uint32_t)f << j;
  }
  if (mask) *mask = mk;
  return n;
}

}  // namespace inj
}  // namespace peat
