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
#include <cstring>

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
static __device__ __noinline__ double digits_div_rn(const uint32_t* N, int nd, uint64_t k, int times, int scale) {
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

// host and device spellings of the few bit operations used below
__host__ __device__ inline int clz64(uint64_t x) {
#ifdef __CUDA_ARCH__
  return __clzll((long long)x);
#else
  return x ? __builtin_clzll(x) : 64;
#endif
}
__host__ __device__ inline double bits_to_double(uint64_t b) {
#ifdef __CUDA_ARCH__
  return __longlong_as_double((long long)b);
#else
  double d;
  memcpy(&d, &b, sizeof(d));
  return d;
#endif
}

// floor(W / Dn) and W mod Dn for W < 2^128 and Dn in [2^63, 2^64): the
// quotient is built from digits of about 20 bits, each estimated in float32
// from the remainder's leading 24 bits and Dn's leading 24 bits, scaled down
// by 1 - 2^-20 so that it never exceeds the true digit (the estimate is
// within 3 2^-24 of rem / Dn), and each removed from the remainder exactly;
// a digit that comes out as 0 while rem >= Dn is taken as 1.  Every step
// shrinks the remainder by about 2^20 (a digit is at least 2^-19 short of
// the true quotient only in relative terms), so five or six steps reach
// rem < Dn; the loops are bounded all the same.
__host__ __device__ inline void divmod_128_64(unsigned __int128 W, uint64_t Dn, unsigned __int128& Q, uint64_t& R) {
  const float rd = 1.0f / (float)(uint32_t)(Dn >> 40);  // Dn >> 40 in [2^23, 2^24): exact in float32
  unsigned __int128 rem = W, q = 0;
  for (int it = 0; it < 16 && rem >= Dn; it++) {
    const uint64_t rh64 = (uint64_t)(rem >> 64);
    const int lz = rh64 ? clz64(rh64) : 64 + clz64((uint64_t)rem);
    const int s = 104 - lz;  // rem's leading 24 bits are rem >> s
    const uint32_t top = (uint32_t)(rem >> s);
    // rem / Dn ~ top 2^s / (dtop 2^40) with dtop = Dn >> 40: est 2^(s - 40)
    // with est = top rd in (1/2, 2), taken as the 25-bit integer est 2^24
    const uint64_t e24 = (uint64_t)((float)top * rd * (1.0f - 9.5367431640625e-7f) * 16777216.0f);  // (1 - 2^-20) 2^24
    // rem >= Dn >= 2^63 has at least 64 bits, so k = s - 40 >= 0
    const int k = s - 40 - 24;
    unsigned __int128 t = k >= 0 ? (unsigned __int128)e24 << k : (unsigned __int128)(e24 >> -k);
    if (t == 0) t = 1;  // rem >= Dn: at least one more
    rem -= t * Dn;      // t Dn <= rem: never below zero
    q += t;
  }
  for (int it = 0; it < 4 && rem >= Dn; it++) {  // not reached: the loop above ends with rem < Dn
    rem -= Dn;
    q += 1;
  }
  Q = q;
  R = (uint64_t)rem;
}

// RN-even binary64 of X = (W + f) 2^E / D for W >= 2^127 (its top bit
// set), 0 <= f < 1 (f > 0 exactly when sticky) and 1 <= D < 2^64, in integer
// and float32 arithmetic only: with Dn = D 2^z normalised to [2^63, 2^64),
// Q = floor(W / Dn) (2^63 <= Q < 2^65) and X = (Q + e) 2^(E + z), 0 <= e < 1,
// e > 0 exactly when the remainder or f is nonzero.  Q keeps at least 63
// bits, more than the 53 + 1 the rounding reads, so the remainder only
// enters as the sticky bit.  The binary64 bits are assembled directly
// (normal, subnormal, or +inf past the largest double).
__host__ __device__ inline double quot_rn(unsigned __int128 W, bool sticky, int E, uint64_t D) {
  const int z = clz64(D);
  const uint64_t Dn = D << z;
  unsigned __int128 Q;
  uint64_t rem;
  divmod_128_64(W, Dn, Q, rem);
  sticky = sticky || rem != 0;
  const int t = (uint64_t)(Q >> 64) ? 64 : 63;  // Q's leading one
  const int P = E + z, lead = t + P;
  if (lead >= 1024) return bits_to_double(0x7FF0000000000000ull);
  const bool normal = lead >= -1022;
  const int pos = normal ? t - 52 : -1074 - P;  // Q's bit of the result's last place (>= 1)
  uint64_t m = 0;
  bool half = false, below = sticky || Q != 0;
  if (pos < 128) {
    m = (uint64_t)(Q >> pos);
    half = ((Q >> (pos - 1)) & 1) != 0;
    below = sticky || (pos >= 2 && (Q << (129 - pos)) != 0);
  }
  if (half && (below || (m & 1ull))) m++;
  // normal: the implicit bit of m carries into the exponent field (and a
  // rounding to 2^53 moves it up one); subnormal: m itself (2^52 is 2^-1022)
  const uint64_t bits = normal ? ((uint64_t)(lead + 1022) << 52) + m : m;
  if (bits >= 0x7FF0000000000000ull) return bits_to_double(0x7FF0000000000000ull);
  return bits_to_double(bits);
}

// RN-even binary64 of N 2^scale / D for the nd-digit magnitude N and
// 1 <= D < 2^64: N's leading 128 bits as W (top bit set), the rest as the
// sticky bit, then quot_rn.
// Out of line: the mean and the variance share one copy of the code (it runs
// once per call, so a second copy would be a second cold fetch).
static __host__ __device__ __noinline__ double digits_quot_rn(const uint32_t* N, int nd, uint64_t D, int scale) {
  int top = nd - 1;
  while (top >= 0 && N[top] == 0) top--;
  if (top < 0) return 0.0;
  const int lz = clz64(N[top]) - 32;
  auto dig = [&](int i) -> uint32_t { return i >= 0 ? N[i] : 0u; };
  const unsigned __int128 win = ((unsigned __int128)dig(top) << 96) | ((unsigned __int128)dig(top - 1) << 64) |
                                ((unsigned __int128)dig(top - 2) << 32) | dig(top - 3);
  const uint32_t next = dig(top - 4);
  const unsigned __int128 W = lz ? (win << lz) | (next >> (32 - lz)) : win;
  bool sticky = lz ? (uint32_t)(next << lz) != 0 : next != 0;
  for (int i = top - 5; i >= 0 && !sticky; i--) sticky = N[i] != 0;  // usually stops at once
  return quot_rn(W, sticky, scale + 32 * (top - 3) - lz, D);
}

// Shared scratch of mean_var_block: S1 = A 2^e1 (NA digits) and
// S2 = B 2^(2 e1 + 32 SHB) (NB digits), both non-negative magnitudes.
template <int NA, int NB, int SHB>
struct MeanVarScratch {
  static constexpr int ND = (2 * NA > NB + SHB + 2 ? 2 * NA : NB + SHB + 2) + 1;
  uint32_t A[NA], B[NB];
  unsigned __int128 col[2 * NA];  // column sums of A * A
  long long t[ND];                // N as signed carry-save digits
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

// A barrier of nt threads (a multiple of 32): the block's own barrier for
// id 0, else the named barrier id (only the group's threads take part).
__device__ __forceinline__ void group_sync(int id, int nt) {
  if (id == 0) __syncthreads();
  else asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nt) : "memory");
}

// Called by every thread of a group of nt threads (t = 0 .. nt - 1, barrier
// id bar) once s.A and s.B hold S1 and S2 (written by threads of the group);
// leaves s.mean and s.var for every thread of the group.  n_f S2 - S1^2 is
// never negative (Cauchy-Schwarz over the n_f values |d|), so the carry
// propagation below ends without a borrow.  The mean (thread 32) and the
// carries and the variance (thread 0) run side by side on two warps.
template <int NA, int NB, int SHB>
__device__ void mean_var_group(MeanVarScratch<NA, NB, SHB>& s, uint64_t nf, int e1, int t, int nt, int bar) {
  constexpr int ND = MeanVarScratch<NA, NB, SHB>::ND;
  group_sync(bar, nt);
  // the nonzero digit ranges: the loops below skip the zeros around them
  int la = NA, ta = -1, lb = NB, tb = -1;
  for (int i = 0; i < NA; i++)
    if (s.A[i]) {
      la = min(la, i);
      ta = i;
    }
  for (int i = 0; i < NB; i++)
    if (s.B[i]) {
      lb = min(lb, i);
      tb = i;
    }
  for (int c = 2 * la + t; c <= 2 * ta; c += nt) {
    unsigned __int128 acc = 0;
    const int i0 = max(la, c - ta), i1 = min(ta, c - la);
    for (int i = i0; i <= i1; i++) acc += (unsigned __int128)((uint64_t)s.A[i] * s.A[c - i]);
    s.col[c] = acc;  // below 2^(64 + 8): three digits
  }
  // N = n_f B 2^(32 SHB) - A^2 as signed carry-save digits, every digit on
  // its own thread: the three 32-bit parts of the products B[k] n_f that
  // land on digit j, minus those of the column sums (each part below 2^32,
  // so |t[j]| < 2^34).  Digits below j0 are zero, and so are those from j1
  // on (past the last carry).
  const int j0 = ta < 0 ? 0 : (tb >= 0 ? min(2 * la, SHB + lb) : 2 * la);
  const int j1 = ta < 0 ? 0 : min(ND, max(2 * ta + 4, tb >= 0 ? SHB + tb + 4 : 0));
  group_sync(bar, nt);
  for (int j = j0 + t; j < j1; j += nt) {
    long long v = 0;
#pragma unroll
    for (int q = 0; q < 3; q++) {
      const int k = j - SHB - q;  // B[k] n_f contributes its part q to digit j
      if (k >= lb && k <= tb) v += (long long)(uint32_t)(((unsigned __int128)s.B[k] * nf) >> (32 * q));
      const int c = j - q;  // so does the column sum c
      if (c >= 2 * la && c <= 2 * ta) v -= (long long)(uint32_t)(s.col[c] >> (32 * q));
    }
    s.t[j] = v;
  }
  group_sync(bar, nt);
  const int tmean = nt > 32 ? 32 : 0;
  if (t == tmean) s.mean = (nf == 0 || ta < 0) ? 0.0 : digits_quot_rn(s.A, ta + 1, nf, e1);
  if (t == 0) {
    if (nf == 0 || ta < 0) {
      s.var = 0.0;
    } else {
      // carry propagation (64-bit arithmetic shifts; the final carry is 0 as N >= 0)
      for (int j = 0; j < j0; j++) s.N[j] = 0;
      long long carry = 0;
      for (int j = j0; j < j1; j++) {
        const long long v = s.t[j] + carry;
        s.N[j] = (uint32_t)v;
        carry = v >> 32;
      }
      for (int j = j1; j < ND; j++) s.N[j] = 0;
      s.var = nf < (1ull << 32) ? digits_quot_rn(s.N, j1, nf * nf, 2 * e1) : digits_div_rn(s.N, j1, nf, 2, 2 * e1);
    }
  }
  group_sync(bar, nt);
}

// the same with the whole block as the group (every thread calls it)
template <int NA, int NB, int SHB>
__device__ void mean_var_block(MeanVarScratch<NA, NB, SHB>& s, uint64_t nf, int e1) {
  mean_var_group(s, nf, e1, (int)threadIdx.x, (int)blockDim.x, 0);
}

}  // namespace peat
