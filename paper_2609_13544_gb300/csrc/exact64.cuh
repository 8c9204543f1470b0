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

constexpr uint64_t MAG64 = 0x7FFFFFFFFFFFFFFFull, INF64 = 0x7FF0000000000000ull;
__device__ __forceinline__ uint64_t bits64(double x) { return (uint64_t)__double_as_longlong(x); }
__device__ __forceinline__ double from_bits64(uint64_t b) { return __longlong_as_double((long long)b); }

// d = c - g exactly (both finite); returns |d| and the sign of d.  The
// operands are ordered by magnitude (their bit patterns order as their
// values), so Fast2Sum's three operations give the exact error term
// (Dekker: s = RN(x + y), t = y - RN(s - x) when |x| >= |y|).
__device__ __forceinline__ Mag diff64(double g, double c, bool& dneg) {
  double x = c, y = from_bits64(bits64(g) ^ 0x8000000000000000ull);
  if ((bits64(x) & MAG64) < (bits64(y) & MAG64)) {
    const double t = x;
    x = y;
    y = t;
  }
  int sc = 0;
  double s = __dadd_rn(x, y);
  if ((bits64(s) & MAG64) >= INF64) {  // the difference overflows: halve both (exact at this size)
    x = __dmul_rn(x, 0.5);
    y = __dmul_rn(y, 0.5);
    s = __dadd_rn(x, y);
    sc = 1;
  }
  const double t = __dsub_rn(y, __dsub_rn(s, x));
  dneg = (bits64(s) >> 63) != 0;
  // the error term of |d| (sign of d folded in); a zero is +0: -0 and +0 would order apart below
  const uint64_t lb = bits64(t) ^ (dneg ? 0x8000000000000000ull : 0ull);
  return Mag{from_bits64(bits64(s) & MAG64), from_bits64((lb & MAG64) ? lb : 0ull), sc};
}

// x < 0 on the bits (x is never -0 here: see diff64)
__device__ __forceinline__ bool neg64(double x) { return (bits64(x) >> 63) != 0; }

// order-preserving key of a double (as an unsigned integer)
__device__ __forceinline__ uint64_t okey64(double x) {
  const uint64_t b = bits64(x);
  return (b >> 63) ? ~b : (b | 0x8000000000000000ull);
}

// a > b exactly (lexicographic on the scale, then hi, then lo: hi is the
// rounding of the exact value, so a larger hi means a larger value)
__device__ __forceinline__ bool mag_gt(const Mag& a, const Mag& b) {
  if (a.sc != b.sc) return a.sc > b.sc;
  const uint64_t ha = bits64(a.hi), hb = bits64(b.hi);  // both >= 0: the bits order as the values
  if (ha != hb) return ha > hb;
  return okey64(a.lo) > okey64(b.lo);
}

// a <= atol + rtol ag exactly (a > 0)
__device__ __forceinline__ bool within64(const Mag& a, double ag, double rtol, double atol) {
  const double thr = __fma_rn(rtol, ag, atol);
  // margin test on the bit patterns (positive normal doubles): 16 patterns apart
  // is at least 16 units in the last place of the smaller, more than the
  // rounding of thr and the |lo| <= ulp(hi) / 2 of a together
  const uint64_t hb = bits64(a.hi), tb = bits64(thr);
  const uint64_t LO = 0x07B0000000000000ull, HI = 0x7E70000000000000ull;  // 2^-900, 2^1000
  if (a.sc == 0 && hb >= LO && tb >= LO && tb <= HI) {
    if (hb + 16 < tb) return true;
    if (hb > tb + 16) return false;
  }
  XTerm t[4] = {dbl_term(a.hi, a.sc, false), dbl_term(a.lo, a.sc, neg64(a.lo)), dbl_term(atol, 0, true),
                prod_term(rtol, ag, 0, true)};
  return xsign(t, 4) <= 0;
}

}  // namespace x64
}  // namespace peat
