// The exact tolerance test |c - g| <= atol + rtol |g| on float32 operands
// (the WITHIN_TOL condition of the compare, and the isclose acceptance of
// Section III-A): |d| as an exact float32 TwoSum pair, one fma with a margin
// deciding all but the close calls, and the integer digits of
// |d| - atol - rtol |g| deciding those.
#pragma once
#include <cstdint>

#include "exact.cuh"

namespace peat {
namespace tolx {

// sign of (hi + lo) 2^sc - atol - rtol ag, exactly (integer digits)
static __device__ __noinline__ int excess_sign(float hi, float lo, int sc, float ag, float rtol, float atol) {
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

}  // namespace tolx
}  // namespace peat
