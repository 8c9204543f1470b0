// Internal declarations shared by the library's translation units.
#pragma once
#include <cstdint>

#include <cuda_runtime.h>

#include "peat.h"

namespace peat {

#ifdef __CUDACC__
// Programmatic dependent launch (PTX griddepcontrol, sm_90 and later). A
// kernel started by launch_dependent may begin while the kernel before it on
// the stream is still running, so it calls pdl_wait() before its first access
// to anything that kernel (or any earlier one) writes; pdl_wait() returns once
// the previous kernel has completed and its memory operations are visible,
// and at once in a kernel launched the ordinary way. pdl_trigger() lets the
// next dependent kernel start launching; without it that happens when this
// kernel completes. A dependent's blocks only occupy resources that the
// previous grid's finished blocks gave back, since the launch waits for every
// block of the previous grid to trigger or exit.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
template <typename... KA, typename... A>
inline cudaError_t launch_dependent(void (*kernel)(KA...), unsigned grid, unsigned block, size_t smem,
                                    cudaStream_t s, A... args) {
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}
#endif

// Exact sums are carried as NLIMB signed 64-bit digits; digit j weighs
// 2^(32 j + LIMB_LSB).  Every term that occurs (products of two float32
// values, or of a binary64 difference and a float32 value) is a multiple of
// 2^-416, and every sum stays below 2^352.
constexpr int NLIMB = 24;
constexpr int LIMB_LSB = -416;
constexpr int NSUM = 3;  // 0: sum d, 1: sum |d|, 2: sum d^2

constexpr int BLOCK = 256;    // threads per compare CTA
constexpr int GCAP = 16384;   // general-path pairs a CTA lists per segment piece (more: the piece is rescanned)
constexpr int HBINS = 128;    // 64 rel bins + 64 ULP bins

// Exact maxima of one CTA piece (element indices are global).  |d| is kept
// as (hi + lo) * 2^sc with hi = RN32(|d| 2^-sc), |lo| at most half a float32
// step of hi, and sc = 1 only when |d| exceeds the float32 range.  The rel
// record is (hi + lo) 2^sc / g with g = |golden| (g = 0: +inf).  idx = -1:
// no record.  Only strictly positive errors and ULP distances are recorded;
// first_fin / first_ulp give the argmax when every error is zero.
struct Partial {
  float abs_hi, abs_lo;
  int32_t abs_sc, pad0;
  int64_t abs_idx;
  float rel_hi, rel_lo, rel_g;
  int32_t rel_sc;
  int64_t rel_idx;
  uint64_t ulp;
  int64_t ulp_idx;
  int64_t first_fin;  // lowest index of a finite pair (-1 none)
  int64_t first_ulp;  // lowest index of a pair without NaN (-1 none)
};

// Integer totals of one segment: every CTA piece of the segment adds into
// them with atomics (all integers, so the order does not matter); the CTA that
// finishes the segment's last piece reads and clears them.  cnt: 0 EXACT,
// 1 window pairs, 2 window pairs within tol, 3 non-finite pairs, 4 general
// within, 5 general mismatch, 6 NaN/Inf asymmetric, 7 sign flip.  limbs:
// carry-save digits of the three exact sums.  done: pieces finished so far.
struct SegAcc {
  unsigned long long hist[HBINS];
  unsigned long long cnt[8];
  long long limbs[NSUM][NLIMB];
  unsigned int done;
  unsigned int pad;
};

// One element-wise pseudo-error model of a fused inject-and-compare call.
constexpr int INJ_MAX = 8;
struct InjStep {
  int kind;            // PEAT_INJ_* (element-wise kinds only)
  uint32_t model;      // its index in the caller's list (Philox counter word)
  uint64_t threshold;  // Bernoulli threshold on a 32-bit word (rates)
  float x;             // sigma, alpha or rate parameter in float32
};

// the element-wise model kinds (those a fused call can generate per element)
inline bool inj_elementwise(int kind) {
  return kind == PEAT_INJ_NAN_INF || kind == PEAT_INJ_SIGNFLIP || kind == PEAT_INJ_REL_GAUSS ||
         kind == PEAT_INJ_ADD_GAUSS || kind == PEAT_INJ_BIAS || kind == PEAT_INJ_CAST_F16_RNE ||
         kind == PEAT_INJ_CAST_F16_RTZ || kind == PEAT_INJ_CAST_BF16_RNE || kind == PEAT_INJ_CAST_BF16_RTZ;
}

struct CompareParams {
  const void* g;
  const void* c;           // unused when inj_n > 0
  // fused injection: the candidate is the golden after inj[0..inj_n) applied
  // in order, generated in the tiles and never stored (inj_n = 0: c is read)
  int inj_n;
  uint32_t inj_k0, inj_k1;  // the seed
  InjStep inj[INJ_MAX];
  int64_t n_total;
  const int64_t* offsets;  // device copy, nseg + 1 entries
  const int64_t* bounds;   // device copy, nctas + 1 CTA range boundaries
  int64_t nseg;
  int64_t p0;              // first element index of the aligned vector grid; -1: scalar only
  int nctas;
  Partial* partials;       // nseg + nctas slots; slot s + b holds CTA b's part of segment s
  SegAcc* acc;             // nseg accumulators, all zero between calls
  uint32_t* glist;         // nctas * GCAP offsets: each CTA's general pairs of the current piece
  int has_empty;           // some segment is empty (CTA 0 writes the outputs of the empty segments)
  unsigned int* status;    // device-visible error word (bit 0: a bounded wait expired)
  unsigned int wait_limit; // iteration bound of a pipeline wait (0: give up at once, for tests)
  float rtol, atol;        // float32 tolerances
  peat_stats_t* stats;
  uint64_t* hist;          // may be null
  void* stage1_event;      // host side only: a cudaEvent_t recorded after the stage-1 launch (or null)
};

// Host-side launchers (compare.cu / inject.cu).
cudaError_t launch_compare(int dtype, const CompareParams& p, cudaStream_t s);
int compare_ctas_per_sm();
cudaError_t compare_prepare();
// CTA b of a grid of nctas owns elements [bound(b), bound(b+1)); boundaries
// lie on the 16-byte vector grid that starts at element p0 (p0 < 0: none)
int64_t compare_cta_bound(int dtype, int64_t b, int nctas, int64_t n, int64_t p0);
size_t compare_partial_bytes();
size_t compare_segacc_bytes();
// offsets {0, n} and the nctas + 1 CTA bounds of a one-tensor call, computed
// by a one-CTA kernel (for the caller that has no host staging buffer)
cudaError_t launch_bounds_on_device(int dtype, int64_t* offsets, int64_t* bounds, int nctas, int64_t n, int64_t p0,
                                    unsigned int* status, cudaStream_t s);

// ---- mean of the top errors (topk.cu) ----
// key(|d|) is an order-preserving 31-bit key of |c - g|.  A sample picks a
// window of TK_WIN digits of key >> 21 (TK_NB0 values); a streaming pass
// counts exactly and resolves key >> 10 inside the window (TK_NB1 = 2048
// values per digit); a second one resolves the last 10 bits (TK_NB2).  Should
// the window miss, an exact pass over key >> 21 replaces the sample.
constexpr int TK_NB0 = 1024, TK_NB1 = 2048, TK_NB2 = 1024, TK_WIN = 3;
constexpr int64_t TK_SAMPLE = 1 << 18;  // pairs in the sample
constexpr unsigned TK_LCAP = 65536;     // listed pairs whose |d| is not a float32 value
constexpr int TK_NBL = 65536;           // bins of each 16-bit digit of the order key of a rounding error

// Device state of one peat_topk_mean call, zero between calls.
struct TopkState {
  unsigned long long hist0[TK_NB0], hist1[TK_WIN * TK_NB1], hist2[TK_NB2];
  unsigned long long nonfin;    // pairs with a NaN or an infinity
  unsigned long long above;     // pairs with key >> 21 above the window
  unsigned long long nfin;      // finite pairs
  unsigned long long k;         // pairs taken
  unsigned long long krem;      // of them, still to place inside the resolved prefix
  unsigned int Plo, Phi;        // the window of key >> 21
  unsigned int P0, P1, T;       // key >> 21, key >> 10, and the key of the k-th largest |d|
  unsigned int ok;              // the window held the k-th largest
  unsigned int done[3];         // CTAs finished, per pass
  unsigned int nlist, nlist2;   // list entries from the last pass and the optional extra one
  unsigned int lowor, inexact;  // over the window pairs of pass 1: OR of the keys' low 10 bits, any |d| not a float32
  unsigned int skip2;           // pass 1 resolved the last digit itself (passes 2 and 3 return at once)
  long long limbs[NLIMB];       // exact sum of the |d| resolved above the prefix
  // only when T's bucket has more than TK_LCAP pairs whose |d| is not a
  // float32 value: a radix select over the order key of their rounding
  // errors, high and low 16 bits (counts zero between calls)
  unsigned long long histl[2][TK_NBL];
  unsigned long long kreml[2];  // the rank left inside the selected high digit, then inside the low one
  unsigned int dl[2];           // the selected high and low digits
};
struct TopkListEntry {
  float lo;      // |d| = (value of key + lo), the value of key taken as in the key's definition
  unsigned key;
};
struct TopkParams {
  const void* g;
  const void* c;
  int64_t n;
  int64_t p0;     // first element of the 16-byte vector grid; -1: none
  int64_t nvec;   // vectors on the grid
  uint64_t num, den;
  TopkState* st;
  TopkListEntry* list;
  peat_topk_t* out;
};
// CTAs of the streaming passes that fit on the device at once
int topk_max_ctas(int nsm);
cudaError_t launch_topk(int dtype, const TopkParams& p, int nctas, cudaStream_t s);

// ---- context statistics (tstats.cu) ----
struct TsAcc {  // per segment, zero between calls
  long long limbs[2][NLIMB];      // exact sum and sum of squares of the finite elements
  unsigned long long nfin, nnan, ninf;
  unsigned int kmin_inv, kmax;    // order keys: ~(smallest finite), largest finite
};
struct TsParams {
  const void* x;
  int64_t n_total;
  int64_t p0;               // first element of the 16-byte vector grid; -1: none
  int64_t nseg;
  const int64_t* offsets;   // device, nseg + 1
  const int64_t* bounds;    // device, nctas + 1
  int nctas;
  TsAcc* acc;               // nseg accumulators
  peat_tstats_t* out;       // device, nseg records
};
int tstats_ctas_per_sm(int dtype);  // resident CTAs of the element type's stage 1
cudaError_t launch_tstats(int dtype, const TsParams& p, cudaStream_t s);

// ---- isclose pass counts over a tolerance grid (isclose.cu) ----
constexpr int ISC_MAX = 64;  // cells (nr * na) at most; nr, na at most as many
struct IscParams {
  const void* g;
  const void* c;
  int64_t n;
  int64_t p0;     // first element of the 16-byte vector grid; -1: none
  int64_t nvec;   // vectors on the grid
  int nr, na, ncells;
  float rtol[ISC_MAX], atol[ISC_MAX];  // float32 tolerances, both ascending
  int aperm[ISC_MAX];                  // the caller's index of the j-th smallest atol
  unsigned long long* counts;          // device, ncells (cell i * na + caller's j), zero before the launch
};
cudaError_t launch_isclose(int dtype, const IscParams& p, int nctas, cudaStream_t s);
cudaError_t launch_isclose64(const IscParams& p, int nctas, cudaStream_t s);  // binary64 operands

// 8-bit formats: one item's totals (sums in units of 2^-S, 2^-2S)
struct Part8 {
  unsigned long long cnt[PEAT_NCLASS], nfin;
  unsigned long long s1lo, s1hi, s2lo, s2hi, sdlo, sdhi;
  unsigned long long ma;
  long long ia;
  unsigned long long ra, rb;
  long long ir;
  unsigned long long mu;
  long long iu;
};
struct Cmp8Params {
  const void* g;
  const void* c;
  const int64_t* offsets;    // nseg + 1
  const int64_t* item_b;     // work items: [item_b, item_e) within segment item_seg
  const int64_t* item_e;
  const int64_t* item_seg;
  const int64_t* seg_first;  // items of segment s: [seg_first[s], seg_first[s + 1])
  int64_t nitems, nseg;
  float rtol, atol;
  // amax[m]: the largest |c - g| 2^S the tolerance accepts for a golden of magnitude bits m,
  // floor(rtol |g| 2^S + atol 2^S) (2^40 when it exceeds every possible difference)
  unsigned long long amax[128];
  int vec;                   // both bases 16-byte aligned
  Part8* parts;              // nitems
  peat_stats_t* stats;       // nseg
  unsigned long long* hist;  // nseg x 128, zero before the launch; NULL: none
};
cudaError_t launch_compare8(int dtype, const Cmp8Params& p, int nctas, cudaStream_t s);

// binary64: one item's maxima and counts, and its three sums as normalised
// 32-bit digits from 2^-2272 (the top limb signed)
struct Part64Rec {
  unsigned long long cnt[PEAT_NCLASS], nfin;
  double ahi, alo;  // max |d| = (ahi + alo) 2^asc at ia
  int asc;
  long long ia;
  double rhi, rlo, rg;  // max |d| / |g| = (rhi + rlo) 2^rsc / rg (rkind 0: zero, 1: finite, 2: +inf) at ir
  int rsc, rkind;
  int rle;              // its log2, approximately: rle + rlf (rle exact, rlf within 2^-20)
  float rlf;
  long long ir;
  unsigned long long mu;  // max ULP distance at iu
  long long iu;
};
constexpr int P64_LIMBS = 136;
struct Part64 {
  Part64Rec rec;
  long long limbs[3 * P64_LIMBS];  // sum d, sum |d|, sum d^2
};
struct Cmp64Params {
  const void* g;
  const void* c;
  const int64_t* offsets;
  const int64_t* item_b;
  const int64_t* item_e;
  const int64_t* item_seg;
  const int64_t* seg_first;
  int64_t nitems, nseg;
  double rtol, atol;  // the float32 tolerances
  int vec;            // both bases 16-byte aligned
  Part64* parts;
  peat_stats_t* stats;
  unsigned long long* hist;
};
cudaError_t launch_compare64(const Cmp64Params& p, int nctas, cudaStream_t s);

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

// The range check of the exact accumulators (for_digits): each kernel source
// sets bit STATUS_DIGIT_RANGE of a library-wide word when a digit would fall
// outside its accumulator (an internal error: the bounds on the terms exclude
// it); each
// kernel source reports to `word` (a device pointer of a mapped host word),
// set per device.
constexpr unsigned int STATUS_DIGIT_RANGE = 2u;
// The checked build (compiled with -DPEAT_CHECKED): index and range
// assertions in the compare kernels.  A failed one sets STATUS_CHECK in the
// same word and its guarded access is skipped; nothing traps.  Without the
// macro every check is the constant true and compiles away.
constexpr unsigned int STATUS_CHECK = 4u;
cudaError_t register_digit_status_compare(unsigned int* word);
cudaError_t register_digit_status_topk(unsigned int* word);
cudaError_t register_digit_status_tstats(unsigned int* word);
cudaError_t register_digit_status_isclose(unsigned int* word);
int test_for_digits(uint64_t m_lo, uint64_t m_hi, int e, int neg, int64_t* out);
double test_quot_rn(uint64_t w_hi, uint64_t w_lo, int sticky, int e, uint64_t d);

}  // namespace peat
