// Exact integer digits shared by the library's kernels: values split into
// integer significands, signed 32-bit digits of a fixed-point accumulator
// (digit j weighs 2^(32 j + LIMB_LSB)), and the one rounding of such an
// accumulator to binary64.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

#include "peat_internal.h"

namespace peat {

// x = m * 2^e with m an integer (x finite, nonzero); float32 and binary64
__device__ __forceinline__ uint32_t split_float(float x, int& e) {
  uint32_t b = __float_as_uint(x) & 0x7FFFFFFFu;
  uint32_t be = b >> 23, m = b & 0x7FFFFFu;
  if (be == 0) {
    e = -149;
    return m;
  }
  e = (int)be - 150;
  return m | 0x800000u;
}
__device__ __forceinline__ uint64_t split_double(double x, int& e) {
  uint64_t b = (uint64_t)__double_as_longlong(x) & 0x7FFFFFFFFFFFFFFFull;
  int be = (int)(b >> 52);
  uint64_t m = b & 0xFFFFFFFFFFFFFull;
  if (be == 0) {
    e = -1074;
    return m;
  }
  e = be - 1075;
  return m | (1ull << 52);
}

// Where a digit outside an accumulator's range is reported: a mapped host
// word shared by the whole library (bit STATUS_DIGIT_RANGE; the handle calls
// return PEAT_ERR_INTERNAL once they see it).  Every source file that
// includes this header has its own copy of the pointer, set on each device
// by register_digit_status before its kernels run (null: not reported).
static __device__ unsigned int* g_digit_status = nullptr;
static inline cudaError_t set_digit_status_here(unsigned int* word) {
  return cudaMemcpyToSymbol(g_digit_status, &word, sizeof(word));
}
#ifdef PEAT_CHECKED
__device__ __forceinline__ bool check_ok(bool c) {
  if (!c && g_digit_status) atomicOr(g_digit_status, STATUS_CHECK);
  return c;
}
#define PEAT_CHECK(cond) (::peat::check_ok(cond))
#else
#define PEAT_CHECK(cond) true
#endif

// the host side of for_digits (only the index check of the test hook runs there)
static thread_local bool t_host_digit_dropped = false;

#pragma nv_exec_check_disable
__host__ __device__ __forceinline__ void digit_dropped() {
#ifdef __CUDA_ARCH__
  if (g_digit_status) atomicOr(g_digit_status, STATUS_DIGIT_RANGE);
#else
  t_host_digit_dropped = true;
#endif
}

// Signed 32-bit digits of +-m * 2^e (m < 2^128), delivered to f(digit, value).
// Every value that occurs is a multiple of 2^LIMB_LSB and below 2^352, so
// every digit index lies in [0, NLIMB); a digit outside it (an internal
// error) is not written out of bounds but reported through the status word.
#pragma nv_exec_check_disable
template <class F>
__host__ __device__ __forceinline__ void for_digits(unsigned __int128 m, int e, bool neg, F&& f) {
  if (m == 0) return;
  int p = e - LIMB_LSB;
  int j = p >> 5, r = p & 31;
  uint32_t md[4] = {(uint32_t)m, (uint32_t)(m >> 32), (uint32_t)(m >> 64), (uint32_t)(m >> 96)};
  uint32_t out[5];
  out[0] = md[0] << r;
#pragma unroll
  for (int k = 1; k < 4; k++) out[k] = (md[k] << r) | (r ? (md[k - 1] >> (32 - r)) : 0u);
  out[4] = r ? (md[3] >> (32 - r)) : 0u;
#pragma unroll
  for (int k = 0; k < 5; k++) {
    if (!out[k]) continue;
    if ((unsigned)(j + k) < (unsigned)NLIMB) f(j + k, neg ? -(int64_t)out[k] : (int64_t)out[k]);
    else digit_dropped();
  }
}

// RN-even binary64 of the exact value of NLIMB carry-save digits (digit j
// weighs 2^(32 j + LIMB_LSB)).  Loops are unrolled with constant indices so
// the digits stay in registers.
__device__ inline double limbs_to_double(const long long* src) {
  int64_t d[NLIMB];
#pragma unroll
  for (int j = 0; j < NLIMB; j++) d[j] = src[j];
  // carry-propagate: digits 0..NLIMB-2 into [0, 2^32), the top digit signed
  int64_t carry = 0;
#pragma unroll
  for (int j = 0; j < NLIMB - 1; j++) {
    const int64_t v = d[j] + carry;
    carry = v >> 32;
    d[j] = v & 0xFFFFFFFFll;
  }
  d[NLIMB - 1] += carry;
  const bool neg = d[NLIMB - 1] < 0;
  if (neg) {
    carry = 0;
#pragma unroll
    for (int j = 0; j < NLIMB - 1; j++) {
      const int64_t v = -d[j] + carry;
      carry = v >> 32;
      d[j] = v & 0xFFFFFFFFll;
    }
    d[NLIMB - 1] = -d[NLIMB - 1] + carry;
  }
  // the top nonzero digit, the two below it, and a sticky bit for the rest
  int top = -1;
#pragma unroll
  for (int j = 0; j < NLIMB; j++)
    if (d[j] != 0) top = j;
  if (top < 0) return 0.0;
  uint64_t w2 = 0, w1 = 0, w0 = 0;
  bool sticky = false;
#pragma unroll
  for (int j = 0; j < NLIMB; j++) {
    if (j == top) w2 = (uint64_t)d[j];
    if (j == top - 1) w1 = (uint64_t)d[j];
    if (j == top - 2) w0 = (uint64_t)d[j];
    if (j < top - 2 && d[j] != 0) sticky = true;
  }
  // after normalisation every digit is below 2^32 (the sums stay below 2^352):
  // W = w2 2^64 + w1 2^32 + w0 < 2^96, value = W 2^(32 (top - 2) + LIMB_LSB)
  const int b = 31 - __clz((uint32_t)w2);  // leading one of w2
  const unsigned __int128 W = ((unsigned __int128)w2 << 64) | ((unsigned __int128)w1 << 32) | w0;
  const int shift = b + 1;                 // W >> shift has its leading one at bit 63
  const uint64_t m = (uint64_t)(W >> shift);
  if ((W & (((unsigned __int128)1 << shift) - 1)) != 0) sticky = true;
  uint64_t mant = m >> 11;
  const uint64_t rbits = m & 0x7FFull;
  if (rbits > 0x400ull || (rbits == 0x400ull && (sticky || (mant & 1ull)))) mant++;
  const int e = 11 + shift + 32 * (top - 2) + LIMB_LSB;
  const double r = ldexp((double)mant, e);
  return neg ? -r : r;
}

// RN-even binary64 of (exact value of the digits) / k, for a non-negative
// value and k >= 1.  The value's leading 128 bits W (the rest only decides
// whether anything below is nonzero) divided by k give a quotient of at least
// 64 bits; with the remainder and the dropped bits as the sticky bit, that
// quotient rounds exactly as the full quotient does.
__device__ inline double limbs_div_rn(const long long* src, uint64_t k) {
  uint32_t d[NLIMB];
  int64_t carry = 0;
#pragma unroll
  for (int j = 0; j < NLIMB; j++) {  // carry-propagate into base-2^32 digits
    const int64_t v = src[j] + carry;
    carry = v >> 32;
    d[j] = (uint32_t)(v & 0xFFFFFFFFll);
  }
  int top = -1;
#pragma unroll
  for (int j = 0; j < NLIMB; j++)
    if (d[j] != 0) top = j;
  if (top < 0) return 0.0;
  uint32_t w4 = 0, w3 = 0, w2 = 0, w1 = 0, w0 = 0;
  bool sticky = false;
#pragma unroll
  for (int j = 0; j < NLIMB; j++) {
    if (j == top) w4 = d[j];
    if (j == top - 1) w3 = d[j];
    if (j == top - 2) w2 = d[j];
    if (j == top - 3) w1 = d[j];
    if (j == top - 4) w0 = d[j];
    if (j < top - 4 && d[j] != 0) sticky = true;
  }
  // the 160-bit window w4..w0 shifted so that its leading one is bit 127 of W
  const int lz = __clz(w4);
  const unsigned __int128 win = ((unsigned __int128)w4 << 96) | ((unsigned __int128)w3 << 64) |
                                ((unsigned __int128)w2 << 32) | w1;
  const unsigned __int128 W = lz ? ((win << lz) | (w0 >> (32 - lz))) : win;
  if ((lz ? (uint32_t)(w0 << lz) : w0) != 0) sticky = true;
  // value = W 2^E + (below), E the weight of W's last bit
  const int E = 32 * (top - 3) - lz + LIMB_LSB;
  const unsigned __int128 q = W / k;
  if (W - q * k != 0) sticky = true;
  const uint64_t qh = (uint64_t)(q >> 64);
  const int qlz = qh ? __clzll(qh) : 64 + __clzll((uint64_t)q);
  const int shift = 64 - qlz;  // q >= 2^63: bits of q below its leading 64
  const uint64_t m = (uint64_t)(q >> shift);
  if (shift > 0 && (q & (((unsigned __int128)1 << shift) - 1)) != 0) sticky = true;
  uint64_t mant = m >> 11;
  const uint64_t rbits = m & 0x7FFull;
  if (rbits > 0x400ull || (rbits == 0x400ull && (sticky || (mant & 1ull)))) mant++;
  return ldexp((double)mant, 11 + shift + E);
}

}  // namespace peat
