// Exact binary64 arithmetic shared by the binary64 compare and isclose grid:
// doubles as integer terms m 2^e, the exact sign of a short sum of such
// terms (32-bit digits over the whole range of products of two doubles), the
// exact difference of two doubles as a TwoSum pair, and the exact tolerance
// test |d| <= atol + rtol |g|.
#pragma once
#include <cstdint>

namespace peat {
namespace x64 {

using u128 = unsigned __int128;

// a finite double as m 2^e, m an integer below 2^53 (m = 0 for zero)
__device__ __forceinline__ void split_d(double x, uint64_t& m, int& e) {
  const uint64_t b = (uint64_t)__double_as_longlong(x) & 0x7FFFFFFFFFFFFFFFull;
  const int ex = (int)(b >> 52);
  const uint64_t f = b & 0xFFFFFFFFFFFFFull;
  if (ex == 0) {
    m = f;
    e = -1074;
  } else {
    m = f | (1ull << 52);
    e = ex - 1075;
  }
}

struct XTerm {
  u128 m;
  int e;
  bool neg;
};

// digits of 32 bits from 2^XLSB: every product of two doubles (down to 2^-2148,
// with 53 + 53 bits) and every term below 2^2080
constexpr int XLSB = -2272;
constexpr int XL = 136;

// sign of sum (neg ? -m : m) 2^e over n terms, exactly (rare paths: out of line)
static __device__ __noinline__ int xsign(const XTerm* t, int n) {
  long long d[XL];
  for (int j = 0; j < XL; j++) d[j] = 0;
  for (int k = 0; k < n; k++) {
    if (t[k].m == 0) continue;
    const int p = t[k].e - XLSB;
    const int limb = p >> 5, sh = p & 31;
    const u128 lo = t[k].m << sh;
    const unsigned long long hi = sh ? (unsigned long long)(t[k].m >> (128 - sh)) : 0ull;
    for (int q = 0; q < 5; q++) {
      const unsigned long long dig =
          q < 4 ? (unsigned long long)(lo >> (32 * q)) & 0xFFFFFFFFull : hi & 0xFFFFFFFFull;
      const int j = limb + q;
      if (dig && j >= 0 && j < XL) d[j] += t[k].neg ? -(long long)dig : (long long)dig;
    }
  }
  long long carry = 0;
  bool nz = false;
  for (int j = 0; j < XL; j++) {
    const long long v = d[j] + carry;
    carry = v >> 32;
    nz |= (v & 0xFFFFFFFFll) != 0;
  }
  if (carry != 0) return carry < 0 ? -1 : 1;
  return nz ? 1 : 0;
}

// the term m1 m2 2^(e1 + e2 + sc) of a product of two doubles
__device__ __forceinline__ XTerm prod_term(double x, double y, int sc, bool neg) {
  uint64_t mx, my;
  int ex, ey;
  split_d(x, mx, ex);
  split_d(y, my, ey);
  return XTerm{(u128)mx * my, ex + ey + sc, neg};
}
__device__ __forceinline__ XTerm dbl_term(double x, int sc, bool neg) {
  uint64_t m;
  int e;
  split_d(x, m, e);
  return XTerm{(u128)m, e + sc, neg};
}

// |d| = (hi + lo) 2^sc with hi = RN64(|d| / 2^sc) >= 0 and lo signed
struct Mag {
  double hi, lo;
  int sc;
};

// d = c - g exactly (both finite); returns |d| and the sign of d
__device__ __forceinline__ Mag diff64(double g, double c, bool& dneg) {
  double x = c, y = -g;
  int sc = 0;
  double s = __dadd_rn(x, y);
  if (!(fabs(s) <= 1.7976931348623157e308)) {
    x = __dmul_rn(x, 0.5);
    y = __dmul_rn(y, 0.5);
    s = __dadd_rn(x, y);
    sc = 1;
  }
  const double yv = __dsub_rn(s, x), xv = __dsub_rn(s, yv);
  const double t = __dadd_rn(__dsub_rn(x, xv), __dsub_rn(y, yv));
  dneg = s < 0.0;
  return Mag{fabs(s), dneg ? -t : t, sc};
}

// a > b exactly (lexicographic on the scale, then hi, then lo: hi is the
// rounding of the exact value, so a larger hi means a larger value)
__device__ __forceinline__ bool mag_gt(const Mag& a, const Mag& b) {
  if (a.sc != b.sc) return a.sc > b.sc;
  if (a.hi != b.hi) return a.hi > b.hi;
  return a.lo > b.lo;
}

// a <= atol + rtol ag exactly (a > 0)
static __device__ bool within64(const Mag& a, double ag, double rtol, double atol) {
  const double thr = __fma_rn(rtol, ag, atol);
  if (a.sc == 0 && a.hi >= 0x1p-900 && thr >= 0x1p-900 && thr <= 0x1p+1000) {
    if (__dmul_rn(a.hi, 1.0 + 0x1p-50) < __dmul_rn(thr, 1.0 - 0x1p-50)) return true;
    if (__dmul_rn(a.hi, 1.0 - 0x1p-50) > __dmul_rn(thr, 1.0 + 0x1p-50)) return false;
  }
  XTerm t[4] = {dbl_term(a.hi, a.sc, false), dbl_term(fabs(a.lo), a.sc, a.lo < 0.0), dbl_term(atol, 0, true),
                prod_term(rtol, ag, 0, true)};
  return xsign(t, 4) <= 0;
}

}  // namespace x64
}  // namespace peat
