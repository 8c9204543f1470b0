// The paper's "Mean of Errors" and "Variance of Errors" scores (Section
// IV-B-3) from exact sums: with S1 = sum |d| and S2 = sum d^2 over the n_f
// pairs whose operands are both finite,
//     mean = S1 / n_f,     var = (n_f S2 - S1^2) / n_f^2   (population variance),
// each the exact value rounded once to binary64 (round to nearest even,
// subnormal and overflowing results included).  The compare kernels of every
// operand width hand their exact sums to mean_var_block; only the digit
// counts and the weight of the last digit differ between them.
#pragma once
#include <cstdint>

namespace peat {

// RN-even binary64 of (W + f) 2^E, with W the integer of the NWD base-2^32
// digits w (least significant first) and 0 <= f < 1, f > 0 exactly when
// sticky is set.  When sticky is set W must have at least 55 significant bits,
// so that every bit that decides the rounding is a bit of W.
template <int NWD>
__device__ double digits_rn(const uint32_t (&w)[NWD], int E, bool sticky) {
  int top = -1;  // position of W's leading one
  for (int j = NWD - 1; j >= 0 && top < 0; j--)
    if (w[j]) top = 32 * j + 31 - __clz(w[j]);
  if (top < 0) return 0.0;
  if (top + E > 1023) return __longlong_as_double(0x7FF0000000000000ll);  // at least 2^1024
  int p = top - 52;                  // last kept bit of a normal result
  if (p + E < -1074) p = -1074 - E;  // or of the subnormal grid
  auto bit = [&](int k) -> uint64_t {
    return (k < 0 || k >= 32 * NWD) ? 0ull : (uint64_t)((w[k >> 5] >> (k & 31)) & 1u);
  };
  uint64_t mant = 0;
  for (int k = top; k >= p; k--) mant = (mant << 1) | bit(k);
  const uint64_t half = bit(p - 1);
  bool below = sticky;
  for (int k = p - 2; k >= 0 && !below; k--) below = bit(k) != 0;
  if (half && (below || (mant & 1ull))) mant++;
  return ldexp((double)mant, p + E);  // exact: mant <= 2^53 on the binary64 grid (or +inf)
}

// RN-even binary64 of N 2^scale / k^times (k >= 1, times 1 or 2), N the
// magnitude of nd base-2^32 digits.  N's leading eight digits (W, 256 bits,
// top digit nonzero) are divided by k, times times, by long division; the
// digits below them and the remainders only set the sticky bit.  As floor
// (floor(W / k) / k) = floor(W / k^2) and W >= 2^224, the quotient keeps at
// least 96 significant bits, so it rounds as the exact quotient does.
__device__ inline double digits_div_rn(const uint32_t* N, int nd, uint64_t k, int times, int scale) {
  int top = nd - 1;
  while (top >= 0 && N[top] == 0) top--;
  if (top < 0) return 0.0;
  uint32_t w[8];
  bool sticky = false;
  for (int j = 0; j < 8; j++) {
    const int i = top - 7 + j;
    w[j] = i >= 0 ? N[i] : 0u;
  }
  for (int i = 0; i < top - 7; i++)
    if (N[i]) sticky = true;
  const int E = scale + 32 * (top - 7);  // weight of W's last bit
  for (int t = 0; t < times; t++) {
    uint64_t rem = 0;  // below k, so every partial quotient fits 32 bits
    for (int j = 7; j >= 0; j--) {
      const unsigned __int128 cur = ((unsigned __int128)rem << 32) | w[j];
      const unsigned __int128 q = cur / k;
      rem = (uint64_t)(cur - q * k);
      w[j] = (uint32_t)q;
    }
    if (rem) sticky = true;
  }
  return digits_rn(w, E, sticky);
}

// Shared scratch of mean_var_block: S1 = A 2^e1 (NA digits) and
// S2 = B 2^(2 e1 + 32 SHB) (NB digits), both non-negative magnitudes.
template <int NA, int NB, int SHB>
struct MeanVarScratch {
  static constexpr int ND = (2 * NA > NB + SHB + 2 ? 2 * NA : NB + SHB + 2) + 1;
  uint32_t A[NA], B[NB];
  unsigned __int128 col[2 * NA];  // column sums of A * A
  uint32_t N[ND];
  double mean, var;
};

// Non-negative carry-save digits (signed 64-bit, digit j weighs 2^(32 j)
// times a common unit) to n + 2 base-2^32 digits of the same value (the last
// carry, non-negative and below 2^63, takes two digits).
__device__ inline void carry_to_digits(const long long* src, int n, uint32_t* out) {
  long long carry = 0;
  for (int j = 0; j < n; j++) {
    const long long v = src[j] + carry;
    carry = v >> 32;
    out[j] = (uint32_t)(v & 0xFFFFFFFFll);
  }
  out[n] = (uint32_t)carry;
  out[n + 1] = (uint32_t)((unsigned long long)carry >> 32);
}

// Called by every thread of the block once s.A and s.B hold S1 and S2 (and
// the writes are visible to the block); leaves s.mean and s.var for every
// thread.  n_f S2 - S1^2 is never negative (Cauchy-Schwarz over the n_f
// values |d|), so the subtraction below ends without a borrow.
template <int NA, int NB, int SHB>
__device__ void mean_var_block(MeanVarScratch<NA, NB, SHB>& s, uint64_t nf, int e1) {
  constexpr int ND = MeanVarScratch<NA, NB, SHB>::ND;
  __syncthreads();
  for (int c = threadIdx.x; c < 2 * NA - 1; c += blockDim.x) {
    unsigned __int128 acc = 0;
    const int i0 = c < NA ? 0 : c - NA + 1, i1 = c < NA ? c : NA - 1;
    for (int i = i0; i <= i1; i++) acc += (unsigned __int128)((uint64_t)s.A[i] * s.A[c - i]);
    s.col[c] = acc;
  }
  if (threadIdx.x == 0) s.col[2 * NA - 1] = 0;
  __syncthreads();
  if (threadIdx.x == 0) {
    if (nf == 0) {
      s.mean = s.var = 0.0;
    } else {
      // N = n_f B 2^(32 SHB) - A^2, digit by digit: the minuend's digit x
      // from the running product, the subtrahend's digit y from the column
      // sums with their carries, and the borrow
      unsigned __int128 prod = 0, carry = 0;
      uint32_t borrow = 0;
      for (int j = 0; j < ND; j++) {
        if (j >= SHB && j < SHB + NB) prod += (unsigned __int128)s.B[j - SHB] * nf;
        const uint32_t x = (uint32_t)prod;
        prod >>= 32;
        unsigned __int128 cs = carry;
        if (j < 2 * NA) cs += s.col[j];
        const uint32_t y = (uint32_t)cs;
        carry = cs >> 32;
        const uint64_t sub = (uint64_t)y + borrow;
        s.N[j] = x - (uint32_t)sub;
        borrow = (uint64_t)x < sub ? 1u : 0u;
      }
      s.mean = digits_div_rn(s.A, NA, nf, 1, e1);
      s.var = digits_div_rn(s.N, ND, nf, 2, 2 * e1);
    }
  }
  __syncthreads();
}

}  // namespace peat
