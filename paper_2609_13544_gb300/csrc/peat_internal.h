// Internal declarations shared by the library's translation units.
#pragma once
#include <cstdint>

#include <cuda_runtime.h>

#include "peat.h"

namespace peat {

// Exact sums are carried as NLIMB signed 64-bit digits; digit j weighs
// 2^(32 j + LIMB_LSB).  Every term that occurs (products of two float32
// values, or of a binary64 difference and a float32 value) is a multiple of
// 2^-416, and every sum stays below 2^352.
constexpr int NLIMB = 24;
constexpr int LIMB_LSB = -416;
constexpr int NSUM = 3;  // 0: sum d, 1: sum |d|, 2: sum d^2

constexpr int BLOCK = 256;    // threads per compare CTA
constexpr int HBINS = 128;    // 64 rel bins + 64 ULP bins

// Exact maxima records.  abs: |d| = hi + lo (binary64 pair, hi = RN(|d|)).
// rel: (hi + lo) / g with g = |golden| (g = 0 means +inf).  idx = -1: none.
struct MaxAbs {
  double hi, lo;
  int64_t idx;
};
struct MaxRel {
  double hi, lo, g;
  int64_t idx;
};
struct MaxUlp {
  uint64_t u;
  int64_t idx;
};

// One CTA's contribution to one segment.  Element indices are global.
struct Partial {
  uint64_t cnt[PEAT_NCLASS];
  uint64_t nonfinite;  // pairs with a NaN or Inf operand
  uint64_t n;
  uint64_t hist[HBINS];
  MaxAbs mabs;
  MaxRel mrel;
  MaxUlp mulp;         // only u > 0 is recorded
  int64_t first_fin;   // lowest index of a finite pair (-1 none)
  int64_t first_ulp;   // lowest index of a pair without NaN (-1 none)
  int64_t limbs[NSUM][NLIMB];  // normalised: digits 0..NLIMB-2 in [0, 2^32), top signed
};

struct CompareParams {
  const void* g;
  const void* c;
  int64_t n_total;
  const int64_t* offsets;  // device copy, nseg + 1 entries
  int64_t nseg;
  int64_t p0;              // first element index of the aligned vector grid; -1: scalar only
  int nctas;
  Partial* partials;       // nseg + nctas slots; slot s + b holds CTA b's part of segment s
  float rtol, atol;        // float32 tolerances
  peat_stats_t* stats;
  uint64_t* hist;          // may be null
};

// Host-side launchers (compare.cu / inject.cu).
cudaError_t launch_compare(int dtype, const CompareParams& p, cudaStream_t s);
int compare_ctas_per_sm();
size_t compare_partial_bytes();

struct InjectElemParams {
  void* dst;
  const void* src;
  int64_t n;
  int kind;
  uint32_t model;
  uint64_t seed;
  uint64_t threshold;   // Bernoulli threshold on a 32-bit word (up to 2^32)
  float x;              // sigma / alpha, float32
  unsigned long long* count;
};
struct InjectScatterParams {
  void* dst;
  const void* src;
  int64_t n;
  int kind;
  const int64_t* pos;   // k positions
  const int64_t* from;  // RV: source values (bit patterns), gathered before any model ran
  const uint32_t* bit;  // BITFLIP bit indices
  int64_t k;
};
cudaError_t launch_inject_elem(int dtype, const InjectElemParams& p, cudaStream_t s);
cudaError_t launch_inject_scatter(int dtype, const InjectScatterParams& p, cudaStream_t s);
cudaError_t launch_gather(int dtype, const void* src, const int64_t* from, int64_t* out, int64_t k,
                          cudaStream_t s);

}  // namespace peat
