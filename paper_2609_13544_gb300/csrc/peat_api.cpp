// Host runtime behind the C ABI declared in include/peat.h: handles,
// workspace, argument checks, launch planning and error reporting.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <unordered_set>
#include <vector>

#include "peat.h"
#include "peat_internal.h"

struct peat_handle_s {
  int device = 0;
  int nsm = 0;
  int64_t max_segments = 4096;
  int max_ctas = 0;
  // compare workspace
  peat::Partial* partials = nullptr;
  peat::SegAcc* acc = nullptr;   // per-segment integer totals, zero between calls
  uint32_t* glist = nullptr;      // per-CTA lists of general-path pairs (stage 1 scratch)
  unsigned int* status_host = nullptr;  // mapped pinned error word written by the kernels
  unsigned int* status_dev = nullptr;
  unsigned int wait_limit = 1u << 24;   // polls before a pipeline wait gives up
  void* stage1_event = nullptr;         // profiling aid: recorded after each compare's stage-1 launch
  int64_t* d_offsets = nullptr;  // offsets (nseg + 1) then CTA bounds (nctas + 1)
  int64_t* h_offsets = nullptr;  // pinned staging of the same
  int64_t* d_single = nullptr;   // one-tensor calls: {0, n} then CTA bounds, written on the device
  // what d_single holds: the key of its last write (dtype, n, p0, nctas, stream)
  bool single_valid = false;
  int single_dtype = -1, single_nctas = 0;
  int64_t single_n = -1, single_p0 = 0;
  cudaStream_t single_stream = nullptr;
  cudaEvent_t staged = nullptr;  // the last staging copy has been consumed
  bool staged_pending = false;
  // mean-of-top-errors workspace, zero between calls
  peat::TopkState* topk = nullptr;
  peat::TopkListEntry* topk_list = nullptr;
  // context-statistics accumulators (one per segment), zero between calls
  peat::TsAcc* tsacc = nullptr;
  // injector staging (grown on demand)
  int64_t* d_inj = nullptr;
  int64_t* h_inj = nullptr;
  size_t inj_cap = 0;  // in int64 elements
  // 8-bit compare: pinned staging of offsets and work items, device copy plus item records
  int64_t* h_f8 = nullptr;
  void* d_f8 = nullptr;
  size_t f8_hcap = 0, f8_dcap = 0;  // bytes
  std::string err;
};

namespace {

thread_local std::string g_create_error;
// text of the last peat_compare_noalloc error on this thread (fixed storage:
// that entry point allocates nothing, host memory included)
thread_local char g_noalloc_error[192];
thread_local bool g_null_error_is_noalloc = false;

struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

peat_status_t fail(peat_handle_t h, peat_status_t st, const std::string& msg) {
  if (h) h->err = msg;
  return st;
}

peat_status_t cuda_fail(peat_handle_t h, cudaError_t e, const char* what) {
  cudaGetLastError();  // clear a sticky non-fatal error state
  return fail(h, PEAT_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// The library-wide word of the exact accumulators' range check (bit
// peat::STATUS_DIGIT_RANGE): one mapped, portable host word, allocated with
// the first handle (or the first allocation-free call) and registered with
// every kernel source once per device.
std::mutex g_digit_mu;
unsigned int* g_digit_host = nullptr;
uint64_t g_digit_devices = 0;  // ordinals below 64 whose kernels report to it

cudaError_t register_digit_status(int dev) {
  std::lock_guard<std::mutex> lk(g_digit_mu);
  if (dev >= 0 && dev < 64 && (g_digit_devices >> dev) & 1) return cudaSuccess;
  cudaError_t e = cudaSuccess;
  if (!g_digit_host) {
    e = cudaHostAlloc((void**)&g_digit_host, sizeof(unsigned int), cudaHostAllocMapped | cudaHostAllocPortable);
    if (e != cudaSuccess) {
      g_digit_host = nullptr;
      return e;
    }
    *(volatile unsigned int*)g_digit_host = 0;
  }
  unsigned int* dptr = nullptr;
  e = cudaHostGetDevicePointer((void**)&dptr, g_digit_host, 0);
  if (e == cudaSuccess) e = peat::register_digit_status_compare(dptr);
  if (e == cudaSuccess) e = peat::register_digit_status_topk(dptr);
  if (e == cudaSuccess) e = peat::register_digit_status_tstats(dptr);
  if (e == cudaSuccess) e = peat::register_digit_status_isclose(dptr);
  if (e == cudaSuccess && dev >= 0 && dev < 64) g_digit_devices |= 1ull << dev;
  return e;
}

// true (and the word cleared) if a kernel reported a lost digit, or a failed
// assertion of the checked build, since the last look; DIGIT_FAULT says which
const char* g_digit_what = "";
bool digit_fault_pending() {
  if (!g_digit_host) return false;
  const unsigned int w = __atomic_exchange_n(g_digit_host, 0u, __ATOMIC_RELAXED);
  if (!w) return false;
  g_digit_what = (w & peat::STATUS_DIGIT_RANGE)
                     ? "an exact accumulator needed a digit outside its range in an earlier call (an internal "
                       "error): the outputs of the calls since the previous check are invalid"
                     : "an index or range assertion of the checked build failed in an earlier call: the outputs "
                       "of the calls since the previous check are invalid";
  return true;
}
#define DIGIT_FAULT g_digit_what


// the element types of the main kernels (the 8-bit formats have their own compare)
int dtype_bytes(int dt) { return dt == PEAT_F32 ? 4 : (dt == PEAT_F16 || dt == PEAT_BF16 ? 2 : 0); }
bool is_fp8(int dt) { return dt == PEAT_F8E4M3 || dt == PEAT_F8E5M2; }
// the element types with a compare of their own (and no other entry point but the isclose grid for 8 bits)
bool own_compare(int dt) { return is_fp8(dt) || dt == PEAT_F64; }
const char* const FP8_ONLY =
    "8-bit and binary64 operands: peat_compare, peat_compare_segmented and peat_isclose_grid only";

bool round_tol(peat_tol_t tol, float* r, float* a) {
  if (!(tol.rtol >= 0.0) || !(tol.atol >= 0.0)) return false;  // rejects NaN too
  *r = (float)tol.rtol;
  *a = (float)tol.atol;
  return std::isfinite(*r) && std::isfinite(*a);
}

// CTA ranges of a segmented call.  A CTA pays for its elements and, per
// segment piece it meets, a fixed CTA-wide merge worth about PIECE_COST
// elements.  For a capacity C, a greedy walk over the segments gives the
// fewest CTAs with cost <= C each (cutting a segment where a CTA fills up);
// a bisection on C finds the smallest capacity that fits in max_ctas CTAs,
// i.e. one wave.  Writes out[0..nctas] and returns nctas (0: no split fits).
constexpr int64_t PIECE_COST = 8192;

int greedy_split(const int64_t* off, int64_t nseg, int64_t n, int64_t C, int cap, int64_t* out) {
  int nct = 0;
  out[0] = 0;
  int64_t cost = 0;
  for (int64_t s = 0; s < nseg; s++) {
    int64_t pos = off[s];
    const int64_t s1 = off[s + 1];
    while (pos < s1) {
      if (cost > 0 && cost + PIECE_COST >= C) {  // no room for another piece: close the CTA
        if (nct == cap) return 0;
        out[++nct] = pos;
        cost = 0;
      }
      const int64_t take = std::min(s1 - pos, std::max<int64_t>(1, C - cost - PIECE_COST));
      cost += PIECE_COST + take;
      pos += take;
      if (pos < s1) {  // the segment goes on in the next CTA
        if (nct == cap) return 0;
        out[++nct] = pos;
        cost = 0;
      }
    }
  }
  if (out[nct] < n) {
    if (nct == cap) return 0;
    out[++nct] = n;
  }
  return nct;
}

int segment_split(const int64_t* off, int64_t nseg, int64_t n, int max_ctas, int64_t* out) {
  int64_t lo = n / max_ctas, hi = n + (nseg + 1) * PIECE_COST;  // hi always fits in one CTA
  for (int it = 0; it < 40 && lo + 1 < hi; it++) {
    const int64_t mid = lo + (hi - lo) / 2;
    if (greedy_split(off, nseg, n, mid, max_ctas, out) > 0) hi = mid;
    else lo = mid;
  }
  return greedy_split(off, nseg, n, hi, max_ctas, out);
}

// wait until the pinned staging buffers may be rewritten
peat_status_t wait_staging(peat_handle_t h) {
  if (h->staged_pending) {
    cudaError_t e = cudaEventSynchronize(h->staged);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventSynchronize");
    h->staged_pending = false;
  }
  return PEAT_OK;
}

// d_single for a one-tensor call: offsets {0, n} and the CTA bounds, written
// by a one-CTA kernel only when they differ from its last write on the same
// stream (stream order then makes the earlier write visible; calls on one
// handle do not overlap on the GPU)
static cudaError_t single_bounds(peat_handle_t h, int dtype, int nctas, int64_t n, int64_t p0, cudaStream_t st) {
  if (h->single_valid && h->single_dtype == dtype && h->single_n == n && h->single_p0 == p0 &&
      h->single_nctas == nctas && h->single_stream == st)
    return cudaSuccess;
  h->single_valid = false;
  cudaError_t e = peat::launch_bounds_on_device(dtype, h->d_single, h->d_single + 2, nctas, n, p0, nullptr, st);
  if (e != cudaSuccess) return e;
  h->single_valid = true;
  h->single_dtype = dtype;
  h->single_n = n;
  h->single_p0 = p0;
  h->single_nctas = nctas;
  h->single_stream = st;
  return cudaSuccess;
}

// Work items for the 8-bit and binary64 compares: runs of at most `ch`
// elements within one segment (about four per SM for one tensor), staged
// with the offsets into the handle's workspace, followed by one record of
// `part_bytes` per item.  Fills the item fields of p (any of the two
// parameter structs) and returns the device base of the records.
struct Items {
  const int64_t *offsets, *item_b, *item_e, *item_seg, *seg_first;
  int64_t nitems;
  void* parts;
};
static peat_status_t stage_items(peat_handle_t h, const int64_t* offsets, int64_t nseg, size_t part_bytes,
                                 cudaStream_t st, Items* out) {
  const int64_t n = offsets[nseg];
  int64_t ch = (n + 4 * (int64_t)h->nsm - 1) / (4 * (int64_t)h->nsm);
  ch = std::min<int64_t>(std::max<int64_t>((ch + 15) / 16 * 16, 4096), (int64_t)1 << 22);
  int64_t nitems = 0;
  for (int64_t s = 0; s < nseg; s++) nitems += (offsets[s + 1] - offsets[s] + ch - 1) / ch;
  // staging: offsets (nseg + 1), item_b, item_e, item_seg (nitems each), seg_first (nseg + 1)
  const size_t nwords = (size_t)(nseg + 1) * 2 + 3 * (size_t)nitems;
  const size_t hbytes = nwords * sizeof(int64_t);
  const size_t pbase = (hbytes + 255) / 256 * 256;
  const size_t dbytes = pbase + (size_t)std::max<int64_t>(nitems, 1) * part_bytes;
  peat_status_t ps = wait_staging(h);  // the pinned staging is free
  if (ps != PEAT_OK) return ps;
  if (hbytes > h->f8_hcap || dbytes > h->f8_dcap) {
    if (h->h_f8) cudaFreeHost(h->h_f8);
    if (h->d_f8) cudaFree(h->d_f8);
    h->h_f8 = nullptr;
    h->d_f8 = nullptr;
    h->f8_hcap = h->f8_dcap = 0;
    const size_t hc = std::max(hbytes, (size_t)65536), dc = std::max(dbytes, (size_t)1 << 20);
    if (cudaMallocHost(&h->h_f8, hc) != cudaSuccess || cudaMalloc(&h->d_f8, dc) != cudaSuccess) {
      cudaGetLastError();
      return fail(h, PEAT_ERR_ALLOC, "compare workspace allocation failed");
    }
    h->f8_hcap = hc;
    h->f8_dcap = dc;
  }
  int64_t* ho = h->h_f8;
  int64_t* hb = ho + (nseg + 1);
  int64_t* he = hb + nitems;
  int64_t* hs = he + nitems;
  int64_t* hf = hs + nitems;
  std::memcpy(ho, offsets, sizeof(int64_t) * (size_t)(nseg + 1));
  int64_t it = 0;
  for (int64_t s = 0; s < nseg; s++) {
    hf[s] = it;
    for (int64_t x = offsets[s]; x < offsets[s + 1]; x += ch, it++) {
      hb[it] = x;
      he[it] = std::min(offsets[s + 1], x + ch);
      hs[it] = s;
    }
  }
  hf[nseg] = it;
  int64_t* d = static_cast<int64_t*>(h->d_f8);
  cudaError_t e = cudaMemcpyAsync(d, ho, hbytes, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(items)");
  e = cudaEventRecord(h->staged, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventRecord");
  h->staged_pending = true;
  out->offsets = d;
  out->item_b = d + (nseg + 1);
  out->item_e = out->item_b + nitems;
  out->item_seg = out->item_e + nitems;
  out->seg_first = out->item_seg + nitems;
  out->nitems = nitems;
  out->parts = reinterpret_cast<char*>(h->d_f8) + pbase;
  return PEAT_OK;
}

// floor(mx 2^ex + my 2^ey) for mx, my < 2^57, saturated at 2^40.  The
// fractional parts are added in 128-bit fixed point with unit 2^-120, exact
// for exponents down to -120; a term below that is under 2^-64 and cannot
// complete a carry, since the other term's fraction is then at most
// 1 - 2^-57.
static uint64_t floor_dyadic_sum(uint64_t mx, int ex, uint64_t my, int ey) {
  const uint64_t CAP = 1ull << 40;
  uint64_t fl = 0;
  unsigned __int128 fr = 0;
  const uint64_t ms[2] = {mx, my};
  const int es[2] = {ex, ey};
  for (int t = 0; t < 2; t++) {
    const uint64_t m = ms[t];
    const int e = es[t];
    if (m == 0 || e < -120) continue;
    if (e >= 0) {
      if (e >= 40 || (m >> (40 - e)) != 0) return CAP;
      fl += m << e;
    } else {
      const int k = -e;
      if (k < 64) {
        fl += m >> k;
        fr += (unsigned __int128)(m & ((1ull << k) - 1)) << (120 - k);
      } else {
        fr += (unsigned __int128)m << (120 - k);
      }
    }
  }
  if (fr >> 120) fl += 1;
  return std::min(fl, CAP);
}

// x = m 2^e with m a 24-bit integer (x a finite float32 >= 0; m = 0 for 0)
static void split_f32(float x, uint64_t* m, int* e) {
  if (x == 0.0f) {
    *m = 0;
    *e = 0;
    return;
  }
  int ex;
  const float fr = std::frexp(x, &ex);  // x = fr 2^ex, fr in [0.5, 1)
  *m = (uint64_t)std::ldexp(fr, 24);    // exact: 24 significant bits
  *e = ex - 24;
}

// The 8-bit formats: items of one segment each, one record per item, merged per segment.
static peat_status_t compare8_impl(peat_handle_t h, const void* g, const void* c, const int64_t* offsets,
                                   int64_t nseg, int dtype, float rtol, float atol, peat_stats_t* stats,
                                   uint64_t* hist, cudaStream_t st) {
  Items it;
  peat_status_t ps = stage_items(h, offsets, nseg, sizeof(peat::Part8), st, &it);
  if (ps != PEAT_OK) return ps;
  cudaError_t e;
  if (hist) {
    e = cudaMemsetAsync(hist, 0, sizeof(uint64_t) * PEAT_HIST_BINS * (size_t)nseg, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(hist)");
  }
  peat::Cmp8Params p;
  std::memset(&p, 0, sizeof(p));
  p.g = g;
  p.c = c;
  p.offsets = it.offsets;
  p.item_b = it.item_b;
  p.item_e = it.item_e;
  p.item_seg = it.item_seg;
  p.seg_first = it.seg_first;
  p.nitems = it.nitems;
  p.nseg = nseg;
  p.rtol = rtol;
  p.atol = atol;
  {
    // the tolerance as one integer bound per golden magnitude: |d| 2^S <= rtol K + atol 2^S
    const int S = dtype == PEAT_F8E4M3 ? 9 : 16, MB = dtype == PEAT_F8E4M3 ? 3 : 2;
    uint64_t mr, ma;
    int er, ea;
    split_f32(rtol, &mr, &er);
    split_f32(atol, &ma, &ea);
    for (uint32_t mag = 0; mag < 128; mag++) {
      const uint32_t ee = mag >> MB, mm = mag & ((1u << MB) - 1u);
      const uint64_t K = ee == 0 ? mm : ((uint64_t)(mm | (1u << MB)) << (ee - 1));  // |g| 2^S (unused past the finite range)
      p.amax[mag] = floor_dyadic_sum(mr * K, er, ma, ea + S);
    }
  }
  p.vec = (reinterpret_cast<uintptr_t>(g) % 16 == 0 && reinterpret_cast<uintptr_t>(c) % 16 == 0) ? 1 : 0;
  p.parts = static_cast<peat::Part8*>(it.parts);
  p.stats = stats;
  p.hist = reinterpret_cast<unsigned long long*>(hist);
  const int nctas = (int)std::max<int64_t>(1, std::min<int64_t>(it.nitems, 2 * (int64_t)h->nsm));
  e = peat::launch_compare8(dtype, p, nctas, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "8-bit compare launch");
  return PEAT_OK;
}

// binary64: the same item structure, records with the three sums as digits.
static peat_status_t compare64_impl(peat_handle_t h, const void* g, const void* c, const int64_t* offsets,
                                    int64_t nseg, float rtol, float atol, peat_stats_t* stats, uint64_t* hist,
                                    cudaStream_t st) {
  Items it;
  peat_status_t ps = stage_items(h, offsets, nseg, sizeof(peat::Part64), st, &it);
  if (ps != PEAT_OK) return ps;
  cudaError_t e;
  if (hist) {
    e = cudaMemsetAsync(hist, 0, sizeof(uint64_t) * PEAT_HIST_BINS * (size_t)nseg, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(hist)");
  }
  peat::Cmp64Params p;
  std::memset(&p, 0, sizeof(p));
  p.g = g;
  p.c = c;
  p.offsets = it.offsets;
  p.item_b = it.item_b;
  p.item_e = it.item_e;
  p.item_seg = it.item_seg;
  p.seg_first = it.seg_first;
  p.nitems = it.nitems;
  p.nseg = nseg;
  p.rtol = (double)rtol;
  p.atol = (double)atol;
  p.vec = (reinterpret_cast<uintptr_t>(g) % 16 == 0 && reinterpret_cast<uintptr_t>(c) % 16 == 0) ? 1 : 0;
  p.parts = static_cast<peat::Part64*>(it.parts);
  p.stats = stats;
  p.hist = reinterpret_cast<unsigned long long*>(hist);
  const int nctas = (int)std::max<int64_t>(1, std::min<int64_t>(it.nitems, 2 * (int64_t)h->nsm));
  e = peat::launch_compare64(p, nctas, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "binary64 compare launch");
  return PEAT_OK;
}

// element-wise models of a fused call, already validated
struct InjSpec {
  int n = 0;
  uint64_t seed = 0;
  peat::InjStep step[peat::INJ_MAX];
};

peat_status_t compare_impl(peat_handle_t h, const void* g, const void* c, const int64_t* offsets,
                           int64_t nseg, peat_dtype_t dtype, peat_tol_t tol, peat_stats_t* stats,
                           uint64_t* hist, peat_stream_t stream, const InjSpec* inj = nullptr) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  int B = dtype_bytes(dtype);
  const bool f8 = is_fp8(dtype), f64 = dtype == PEAT_F64;
  if (!B && !f8 && !f64) return fail(h, PEAT_ERR_INVALID_ARG, "dtype must be one of peat_dtype_t");
  if ((f8 || f64) && inj) return fail(h, PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  float rtol, atol;
  if (!round_tol(tol, &rtol, &atol))
    return fail(h, PEAT_ERR_INVALID_ARG, "rtol and atol must be finite and >= 0 after rounding to float32");
  if (nseg < 0) return fail(h, PEAT_ERR_INVALID_ARG, "nseg < 0");
  if (nseg > h->max_segments)
    return fail(h, PEAT_ERR_UNSUPPORTED, "nseg exceeds the handle's max_segments");
  if (!offsets) return fail(h, PEAT_ERR_INVALID_ARG, "offsets is NULL");
  if (offsets[0] != 0) return fail(h, PEAT_ERR_INVALID_ARG, "offsets[0] must be 0");
  for (int64_t s = 0; s < nseg; s++)
    if (offsets[s + 1] < offsets[s]) return fail(h, PEAT_ERR_INVALID_ARG, "offsets must be non-decreasing");
  const int64_t n = offsets[nseg];
  if (n > 0 && (!g || (!c && !inj))) return fail(h, PEAT_ERR_INVALID_ARG, "golden/candidate is NULL");
  if (nseg > 0 && !stats) return fail(h, PEAT_ERR_INVALID_ARG, "stats_out is NULL");
  if (digit_fault_pending()) return fail(h, PEAT_ERR_INTERNAL, DIGIT_FAULT);
  if (h->status_host && *(volatile unsigned int*)h->status_host) {
    *(volatile unsigned int*)h->status_host = 0;
    return fail(h, PEAT_ERR_TIMEOUT,
                "a bounded device-side wait expired in an earlier call on this handle; its outputs are invalid");
  }
  if (nseg == 0) return PEAT_OK;
  DeviceGuard dg(h->device);
  if (!dg.ok) return fail(h, PEAT_ERR_CUDA, "cudaSetDevice failed");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (f8) return compare8_impl(h, g, c, offsets, nseg, dtype, rtol, atol, stats, hist, st);
  if (f64) return compare64_impl(h, g, c, offsets, nseg, rtol, atol, stats, hist, st);

  peat::CompareParams p;
  std::memset(&p, 0, sizeof(p));
  p.g = g;
  p.c = c;
  p.n_total = n;
  p.nseg = nseg;
  if (inj) {  // the candidate is generated from the golden: align on the golden alone
    p.inj_n = inj->n;
    p.inj_k0 = (uint32_t)inj->seed;
    p.inj_k1 = (uint32_t)(inj->seed >> 32);
    for (int m = 0; m < inj->n; m++) p.inj[m] = inj->step[m];
    c = g;
  }
  uintptr_t ag = reinterpret_cast<uintptr_t>(g), ac = reinterpret_cast<uintptr_t>(c);
  if (n > 0 && ag % B == 0 && ac % B == 0 && ag % 16 == ac % 16)
    p.p0 = (int64_t)(((16 - ag % 16) % 16) / B);
  else
    p.p0 = -1;
  // persistent grid; small inputs get about one CTA per 4K elements
  int64_t want = (n + 4095) / 4096;
  p.nctas = (int)std::max<int64_t>(1, std::min<int64_t>(h->max_ctas, want));
  // stage 1 keeps element offsets within a CTA's range in 32 bits
  if (n / p.nctas >= ((int64_t)1 << 31) - 64)
    return fail(h, PEAT_ERR_UNSUPPORTED, "n is too large for one call (more than 2^31 elements per CTA)");

  cudaError_t e;
  if (nseg == 1) {
    // one tensor: offsets and CTA bounds written on the device, no host staging
    // (so back-to-back calls do not wait for each other on the host)
    e = single_bounds(h, dtype, p.nctas, n, p.p0, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "bounds launch");
    p.offsets = h->d_single;
    p.bounds = h->d_single + 2;
  } else {
    peat_status_t ps = wait_staging(h);
    if (ps != PEAT_OK) return ps;
    std::memcpy(h->h_offsets, offsets, sizeof(int64_t) * (size_t)(nseg + 1));
    int64_t* hb = h->h_offsets + nseg + 1;
    const int nsplit = n > 0 ? segment_split(offsets, nseg, n, p.nctas, hb) : 0;
    if (nsplit > 0)
      p.nctas = nsplit;
    else
      for (int b = 0; b <= p.nctas; b++) hb[b] = peat::compare_cta_bound(dtype, b, p.nctas, n, p.p0);
    e = cudaMemcpyAsync(h->d_offsets, h->h_offsets, sizeof(int64_t) * (size_t)(nseg + 2 + p.nctas),
                        cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(offsets)");
    e = cudaEventRecord(h->staged, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventRecord");
    h->staged_pending = true;
    p.offsets = h->d_offsets;
    p.bounds = h->d_offsets + nseg + 1;
  }
  p.acc = h->acc;
  p.partials = h->partials;
  p.glist = h->glist;
  p.has_empty = 0;
  for (int64_t s = 0; s < nseg && !p.has_empty; s++) p.has_empty = offsets[s + 1] == offsets[s];
  p.status = h->status_dev;
  p.stage1_event = h->stage1_event;
  p.wait_limit = h->wait_limit;
  p.rtol = rtol;
  p.atol = atol;
  p.stats = stats;
  p.hist = hist;
  e = peat::launch_compare(dtype, p, st);
  if (e != cudaSuccess) {
    // the accumulators may hold a partial stage 1: clear them for the next call
    cudaMemsetAsync(h->acc, 0, peat::compare_segacc_bytes() * (size_t)nseg, st);
    return cuda_fail(h, e, "compare launch");
  }
  return PEAT_OK;
}

// ---- host Philox4x32-10 for the fixed-count position draws ----
void philox_host(const uint32_t ctr[4], uint64_t seed, uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  for (int r = 0; r < 10; r++) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * c0, p1 = (uint64_t)0xCD9E8D57u * c2;
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0, n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
    c1 = (uint32_t)p1;
    c3 = (uint32_t)p0;
    c0 = n0;
    c2 = n2;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

uint64_t mulhi64(uint64_t w, uint64_t n) { return (uint64_t)(((unsigned __int128)w * n) >> 64); }

peat_status_t grow_inject(peat_handle_t h, size_t need) {
  if (need <= h->inj_cap) return PEAT_OK;
  peat_status_t ps = wait_staging(h);
  if (ps != PEAT_OK) return ps;
  size_t cap = std::max(need, (size_t)4096);
  if (h->d_inj) cudaFree(h->d_inj);
  if (h->h_inj) cudaFreeHost(h->h_inj);
  h->d_inj = nullptr;
  h->h_inj = nullptr;
  h->inj_cap = 0;
  if (cudaMalloc(&h->d_inj, cap * sizeof(int64_t)) != cudaSuccess ||
      cudaMallocHost(&h->h_inj, cap * sizeof(int64_t)) != cudaSuccess) {
    cudaGetLastError();
    return fail(h, PEAT_ERR_ALLOC, "injector staging allocation failed");
  }
  h->inj_cap = cap;
  return PEAT_OK;
}

// ---- scratch of the allocation-free compare ----------------------------------
// One fixed block of device memory per device, reserved when the module
// loads: no call of peat_compare_noalloc allocates.  Its accumulator (acc)
// must be zero when a call starts: static device memory starts at zero, and
// every call that completes leaves it zero (the finalizing CTA clears it).
constexpr int NOALLOC_MAX_CTAS = 320;     // grid cap of the allocation-free compare
constexpr int NOALLOC_MAX_DEVICES = 64;
struct NoallocScratch {
  peat::SegAcc acc;                                  // zero between calls
  unsigned int status;                               // set by an expired device-side wait, cleared per call
  unsigned int pad;
  int64_t offsets[2];                                // {0, n}, written by the bounds kernel
  int64_t bounds[NOALLOC_MAX_CTAS + 1];
  peat::Partial partials[1 + NOALLOC_MAX_CTAS];
  uint32_t glist[(size_t)NOALLOC_MAX_CTAS * peat::GCAP];
};
// testing aid: every bounded wait of the allocation-free compare gives up at once
std::atomic<unsigned int> g_noalloc_wait_limit{1u << 24};

struct NoallocDevice {
  std::atomic<int> ready{0};
  NoallocScratch* scratch = nullptr;
  int nsm = 0;
};
NoallocDevice g_noalloc_dev[NOALLOC_MAX_DEVICES];
std::mutex g_noalloc_setup;

peat_status_t noalloc_fail(peat_status_t st, const char* msg) {
  std::snprintf(g_noalloc_error, sizeof(g_noalloc_error), "%s", msg);
  return st;
}
peat_status_t noalloc_cuda_fail(cudaError_t e, const char* what) {
  cudaGetLastError();
  std::snprintf(g_noalloc_error, sizeof(g_noalloc_error), "%s: %s", what, cudaGetErrorString(e));
  return PEAT_ERR_CUDA;
}

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[sizeof(NoallocScratch)];

extern "C" {

peat_status_t peat_signature_create(peat_handle_t* out, const peat_config_t* cfg) {
  g_null_error_is_noalloc = false;
  g_create_error.clear();
  if (!out) {
    g_create_error = "out is NULL";
    return PEAT_ERR_INVALID_ARG;
  }
  *out = nullptr;
  peat_config_t c;
  std::memset(&c, 0, sizeof(c));
  if (cfg) c = *cfg;
  if ((c.flags & ~PEAT_FLAG_TEST_EXPIRE_WAITS) != 0 || c.max_segments < 0) {
    g_create_error = "bad config (unknown flags, or max_segments < 0)";
    return PEAT_ERR_INVALID_ARG;
  }
  int ndev = 0;
  cudaError_t e = cudaGetDeviceCount(&ndev);
  if (e != cudaSuccess || c.device < 0 || c.device >= ndev) {
    cudaGetLastError();
    g_create_error = std::string("no such CUDA device: ") + (e != cudaSuccess ? cudaGetErrorString(e) : "");
    return e != cudaSuccess ? PEAT_ERR_CUDA : PEAT_ERR_INVALID_ARG;
  }
  peat_handle_t h = new peat_handle_s();
  h->device = c.device;
  h->max_segments = c.max_segments > 0 ? c.max_segments : 4096;
  if (c.flags & PEAT_FLAG_TEST_EXPIRE_WAITS) h->wait_limit = 0;
  DeviceGuard dg(h->device);
  if (!dg.ok) {
    g_create_error = "cudaSetDevice failed";
    delete h;
    return PEAT_ERR_CUDA;
  }
  cudaDeviceGetAttribute(&h->nsm, cudaDevAttrMultiProcessorCount, h->device);
  if (register_digit_status(h->device) != cudaSuccess) {
    cudaGetLastError();
    g_create_error = "could not set up the library's status word";
    delete h;
    return PEAT_ERR_CUDA;
  }
  if (peat::compare_prepare() != cudaSuccess) {
    cudaGetLastError();
    g_create_error = "could not configure the compare kernels";
    delete h;
    return PEAT_ERR_CUDA;
  }
  h->max_ctas = std::max(1, h->nsm * peat::compare_ctas_per_sm());
  // segmented calls may use up to 2 * max_ctas CTAs (see segment_split)
  size_t slots = (size_t)h->max_segments + 2 * (size_t)h->max_ctas;
  size_t staging = (size_t)h->max_segments + 2 + 2 * (size_t)h->max_ctas;
  size_t acc_bytes = (size_t)h->max_segments * peat::compare_segacc_bytes();
  bool ok = cudaMalloc(&h->partials, slots * peat::compare_partial_bytes()) == cudaSuccess &&
            cudaMalloc(&h->acc, acc_bytes) == cudaSuccess &&
            cudaMalloc(&h->glist, sizeof(uint32_t) * (size_t)peat::GCAP * 2 * (size_t)h->max_ctas) == cudaSuccess &&
            cudaHostAlloc((void**)&h->status_host, sizeof(unsigned int), cudaHostAllocMapped) == cudaSuccess &&
            cudaHostGetDevicePointer((void**)&h->status_dev, h->status_host, 0) == cudaSuccess &&
            (*(volatile unsigned int*)h->status_host = 0u, true) &&  // pinned memory starts undefined
            cudaMemset(h->acc, 0, acc_bytes) == cudaSuccess &&
            cudaMalloc(&h->d_offsets, sizeof(int64_t) * staging) == cudaSuccess &&
            cudaMallocHost(&h->h_offsets, sizeof(int64_t) * staging) == cudaSuccess &&
            cudaMalloc(&h->d_single, sizeof(int64_t) * (3 + 2 * (size_t)h->max_ctas)) == cudaSuccess &&
            cudaEventCreateWithFlags(&h->staged, cudaEventDisableTiming) == cudaSuccess &&
            cudaMalloc(&h->topk, sizeof(peat::TopkState)) == cudaSuccess &&
            cudaMemset(h->topk, 0, sizeof(peat::TopkState)) == cudaSuccess &&
            cudaMalloc(&h->topk_list, sizeof(peat::TopkListEntry) * peat::TK_LCAP) == cudaSuccess &&
            cudaMalloc(&h->tsacc, sizeof(peat::TsAcc) * (size_t)h->max_segments) == cudaSuccess &&
            cudaMemset(h->tsacc, 0, sizeof(peat::TsAcc) * (size_t)h->max_segments) == cudaSuccess &&
            cudaDeviceSynchronize() == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    g_create_error = "workspace allocation failed";
    peat_signature_destroy(h);
    return PEAT_ERR_ALLOC;
  }
  *out = h;
  return PEAT_OK;
}

peat_status_t peat_signature_destroy(peat_handle_t h) {
  if (!h) return PEAT_OK;
  {
    DeviceGuard dg(h->device);
    if (h->staged) cudaEventSynchronize(h->staged);
    cudaDeviceSynchronize();
    if (h->partials) cudaFree(h->partials);
    if (h->acc) cudaFree(h->acc);
    if (h->glist) cudaFree(h->glist);
    if (h->status_host) cudaFreeHost(h->status_host);
    if (h->d_offsets) cudaFree(h->d_offsets);
    if (h->h_offsets) cudaFreeHost(h->h_offsets);
    if (h->d_single) cudaFree(h->d_single);
    if (h->d_inj) cudaFree(h->d_inj);
    if (h->h_inj) cudaFreeHost(h->h_inj);
    if (h->d_f8) cudaFree(h->d_f8);
    if (h->h_f8) cudaFreeHost(h->h_f8);
    if (h->topk) cudaFree(h->topk);
    if (h->topk_list) cudaFree(h->topk_list);
    if (h->tsacc) cudaFree(h->tsacc);
    if (h->staged) cudaEventDestroy(h->staged);
    cudaGetLastError();
  }
  delete h;
  return PEAT_OK;
}

peat_status_t peat_compare(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                           peat_dtype_t dtype, peat_tol_t tol, peat_stats_t* stats_out, uint64_t* hist_out,
                           peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  if (n < 0) return fail(h, PEAT_ERR_INVALID_ARG, "n < 0");
  int64_t off[2] = {0, n};
  return compare_impl(h, golden, candidate, off, 1, dtype, tol, stats_out, hist_out, stream);
}

peat_status_t peat_compare_segmented(peat_handle_t h, const void* golden, const void* candidate,
                                     const int64_t* offsets, int64_t nseg, peat_dtype_t dtype,
                                     peat_tol_t tol, peat_stats_t* stats_out, uint64_t* hist_out,
                                     peat_stream_t stream) {
  return compare_impl(h, golden, candidate, offsets, nseg, dtype, tol, stats_out, hist_out, stream);
}

peat_status_t peat_topk_mean(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                             peat_dtype_t dtype, uint64_t num, uint64_t den, peat_topk_t* out,
                             peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  if (own_compare(dtype)) return fail(h, PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  const int B = dtype_bytes(dtype);
  if (!B) return fail(h, PEAT_ERR_INVALID_ARG, "dtype must be PEAT_F32, PEAT_F16 or PEAT_BF16");
  if (n < 0) return fail(h, PEAT_ERR_INVALID_ARG, "n < 0");
  if (n > 0 && (!golden || !candidate)) return fail(h, PEAT_ERR_INVALID_ARG, "golden/candidate is NULL");
  if (num == 0 || num > den) return fail(h, PEAT_ERR_INVALID_ARG, "need 0 < num <= den");
  if (!out) return fail(h, PEAT_ERR_INVALID_ARG, "out is NULL");
  DeviceGuard dg(h->device);
  if (!dg.ok) return fail(h, PEAT_ERR_CUDA, "cudaSetDevice failed");
  if (digit_fault_pending()) return fail(h, PEAT_ERR_INTERNAL, DIGIT_FAULT);
  peat::TopkParams p;
  std::memset(&p, 0, sizeof(p));
  p.g = golden;
  p.c = candidate;
  p.n = n;
  const uintptr_t ag = reinterpret_cast<uintptr_t>(golden), ac = reinterpret_cast<uintptr_t>(candidate);
  const int64_t vec = 16 / B;
  p.p0 = -1;
  if (n > 0 && ag % B == 0 && ac % B == 0 && ag % 16 == ac % 16) {
    const int64_t p0 = (int64_t)(((16 - ag % 16) % 16) / B);
    if (p0 < n) {
      p.p0 = p0;
      p.nvec = (n - p0) / vec;
    }
  }
  p.num = num;
  p.den = den;
  p.st = h->topk;
  p.list = h->topk_list;
  p.out = out;
  // streaming passes: one wave of resident CTAs, about one CTA per 1K elements
  const int64_t want = (n + 1023) / 1024;
  const int nctas = (int)std::max<int64_t>(1, std::min<int64_t>(peat::topk_max_ctas(h->nsm), want));
  // per-thread integer sums in the sum pass stay below 2^64
  if (n / ((int64_t)nctas * 256) >= ((int64_t)1 << 24) - 16)
    return fail(h, PEAT_ERR_UNSUPPORTED, "n is too large for one call (more than 2^24 elements per thread)");
  cudaError_t e = peat::launch_topk(dtype, p, nctas, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    cudaMemsetAsync(h->topk, 0, sizeof(peat::TopkState), reinterpret_cast<cudaStream_t>(stream));
    return cuda_fail(h, e, "top-k launch");
  }
  return PEAT_OK;
}

peat_status_t peat_isclose_grid(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                                peat_dtype_t dtype, const double* rtols, int nr, const double* atols, int na,
                                uint64_t* counts_out, peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  const int B = is_fp8(dtype) ? 1 : (dtype == PEAT_F64 ? 8 : dtype_bytes(dtype));
  if (!B) return fail(h, PEAT_ERR_INVALID_ARG, "dtype must be one of peat_dtype_t");
  if (n < 0) return fail(h, PEAT_ERR_INVALID_ARG, "n < 0");
  if (n > 0 && (!golden || !candidate)) return fail(h, PEAT_ERR_INVALID_ARG, "golden/candidate is NULL");
  if (!rtols || !atols || !counts_out) return fail(h, PEAT_ERR_INVALID_ARG, "rtols/atols/counts_out is NULL");
  if (nr < 1 || na < 1 || nr * na > peat::ISC_MAX)
    return fail(h, PEAT_ERR_INVALID_ARG, "need 1 <= nr, na and nr * na <= 64");
  peat::IscParams p;
  std::memset(&p, 0, sizeof(p));
  for (int i = 0; i < nr; i++) {
    float r, a;
    if (!round_tol(peat_tol_t{rtols[i], 0.0}, &r, &a))
      return fail(h, PEAT_ERR_INVALID_ARG, "rtols must be finite and >= 0 after rounding to float32");
    if (i > 0 && r < p.rtol[i - 1]) return fail(h, PEAT_ERR_INVALID_ARG, "rtols must be non-decreasing");
    p.rtol[i] = r;
  }
  float at[peat::ISC_MAX];
  for (int j = 0; j < na; j++) {
    float r;
    if (!round_tol(peat_tol_t{0.0, atols[j]}, &r, &at[j]))
      return fail(h, PEAT_ERR_INVALID_ARG, "atols must be finite and >= 0 after rounding to float32");
    p.aperm[j] = j;
  }
  // the kernel walks the atols in ascending order (stable: equal atols keep their order)
  std::stable_sort(p.aperm, p.aperm + na, [&](int x, int y) { return at[x] < at[y]; });
  for (int j = 0; j < na; j++) p.atol[j] = at[p.aperm[j]];
  DeviceGuard dg(h->device);
  if (!dg.ok) return fail(h, PEAT_ERR_CUDA, "cudaSetDevice failed");
  if (digit_fault_pending()) return fail(h, PEAT_ERR_INTERNAL, DIGIT_FAULT);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  p.g = golden;
  p.c = candidate;
  p.n = n;
  p.nr = nr;
  p.na = na;
  p.ncells = nr * na;
  p.counts = reinterpret_cast<unsigned long long*>(counts_out);
  const uintptr_t ag = reinterpret_cast<uintptr_t>(golden), ac = reinterpret_cast<uintptr_t>(candidate);
  const int64_t vec = 16 / B;
  p.p0 = -1;
  if (n > 0 && ag % B == 0 && ac % B == 0 && ag % 16 == ac % 16) {
    const int64_t p0 = (int64_t)(((16 - ag % 16) % 16) / B);
    if (p0 < n) {
      p.p0 = p0;
      p.nvec = (n - p0) / vec;
    }
  }
  cudaError_t e = cudaMemsetAsync(counts_out, 0, sizeof(uint64_t) * (size_t)p.ncells, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(counts)");
  if (n == 0) return PEAT_OK;
  const int64_t want = (n + 4095) / 4096;
  const int nctas = (int)std::max<int64_t>(1, std::min<int64_t>((int64_t)h->nsm * 8, want));
  // per-CTA counts are 32-bit
  if (n / nctas >= ((int64_t)1 << 31)) return fail(h, PEAT_ERR_UNSUPPORTED, "more than 2^31 elements per CTA");
  e = dtype == PEAT_F64 ? peat::launch_isclose64(p, nctas, st) : peat::launch_isclose(dtype, p, nctas, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "isclose launch");
  return PEAT_OK;
}

peat_status_t peat_tensor_stats(peat_handle_t h, const void* x, const int64_t* offsets, int64_t nseg,
                                peat_dtype_t dtype, peat_tstats_t* stats_out, peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  if (own_compare(dtype)) return fail(h, PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  const int B = dtype_bytes(dtype);
  if (!B) return fail(h, PEAT_ERR_INVALID_ARG, "dtype must be PEAT_F32, PEAT_F16 or PEAT_BF16");
  if (nseg < 0) return fail(h, PEAT_ERR_INVALID_ARG, "nseg < 0");
  if (nseg > h->max_segments) return fail(h, PEAT_ERR_UNSUPPORTED, "nseg exceeds the handle's max_segments");
  if (!offsets) return fail(h, PEAT_ERR_INVALID_ARG, "offsets is NULL");
  if (offsets[0] != 0) return fail(h, PEAT_ERR_INVALID_ARG, "offsets[0] must be 0");
  for (int64_t s = 0; s < nseg; s++) {
    if (offsets[s + 1] < offsets[s]) return fail(h, PEAT_ERR_INVALID_ARG, "offsets must be non-decreasing");
    if (offsets[s + 1] - offsets[s] >= ((int64_t)1 << 36))
      return fail(h, PEAT_ERR_UNSUPPORTED, "a segment of 2^36 elements or more");
  }
  const int64_t n = offsets[nseg];
  if (n > 0 && !x) return fail(h, PEAT_ERR_INVALID_ARG, "x is NULL");
  if (nseg > 0 && !stats_out) return fail(h, PEAT_ERR_INVALID_ARG, "stats_out is NULL");
  if (nseg == 0) return PEAT_OK;
  DeviceGuard dg(h->device);
  if (!dg.ok) return fail(h, PEAT_ERR_CUDA, "cudaSetDevice failed");
  if (digit_fault_pending()) return fail(h, PEAT_ERR_INTERNAL, DIGIT_FAULT);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  peat::TsParams p;
  std::memset(&p, 0, sizeof(p));
  p.x = x;
  p.n_total = n;
  p.nseg = nseg;
  const uintptr_t ax = reinterpret_cast<uintptr_t>(x);
  p.p0 = (n > 0 && ax % B == 0) ? (int64_t)(((16 - ax % 16) % 16) / B) : -1;
  // one wave of resident CTAs, about one CTA per 8K elements, within the staging area
  const int64_t want = (n + 8191) / 8192;
  const int64_t cap = std::min<int64_t>((int64_t)peat::tstats_ctas_per_sm(dtype) * h->nsm, 2 * (int64_t)h->max_ctas);
  p.nctas = (int)std::max<int64_t>(1, std::min<int64_t>(cap, want));
  cudaError_t e;
  if (nseg == 1) {  // one tensor: no host staging (see compare_impl)
    e = single_bounds(h, dtype, p.nctas, n, p.p0, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "bounds launch");
    p.offsets = h->d_single;
    p.bounds = h->d_single + 2;
  } else {
    peat_status_t ps = wait_staging(h);
    if (ps != PEAT_OK) return ps;
    std::memcpy(h->h_offsets, offsets, sizeof(int64_t) * (size_t)(nseg + 1));
    int64_t* hb = h->h_offsets + nseg + 1;
    for (int b = 0; b <= p.nctas; b++) hb[b] = peat::compare_cta_bound(dtype, b, p.nctas, n, p.p0);
    e = cudaMemcpyAsync(h->d_offsets, h->h_offsets, sizeof(int64_t) * (size_t)(nseg + 2 + p.nctas),
                        cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(offsets)");
    e = cudaEventRecord(h->staged, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventRecord");
    h->staged_pending = true;
    p.offsets = h->d_offsets;
    p.bounds = h->d_offsets + nseg + 1;
  }
  p.acc = h->tsacc;
  p.out = stats_out;
  e = peat::launch_tstats(dtype, p, st);
  if (e != cudaSuccess) {
    cudaMemsetAsync(h->tsacc, 0, sizeof(peat::TsAcc) * (size_t)nseg, st);
    return cuda_fail(h, e, "tensor-stats launch");
  }
  return PEAT_OK;
}

namespace {
peat_status_t host_fail(const char* msg) {
  g_null_error_is_noalloc = false;
  g_create_error = msg;
  return PEAT_ERR_INVALID_ARG;
}
}  // namespace

peat_status_t peat_spearman(const double* x, const double* y, int64_t n, double* rho_out) {
  if (!rho_out || n < 0 || (n > 0 && (!x || !y))) return host_fail("null pointer or n < 0");
  for (int64_t i = 0; i < n; i++)
    if (!std::isfinite(x[i]) || !std::isfinite(y[i])) return host_fail("a value is not finite");
  if (n < 2) {
    *rho_out = std::nan("");
    return PEAT_OK;
  }
  // doubled ranks (integers): a tie group spanning ranks r..r+c-1 takes r + (c - 1) / 2 each
  auto doubled_ranks = [n](const double* v) {
    std::vector<int64_t> idx((size_t)n), r2((size_t)n);
    for (int64_t i = 0; i < n; i++) idx[(size_t)i] = i;
    std::stable_sort(idx.begin(), idx.end(), [v](int64_t a, int64_t b) { return v[a] < v[b]; });
    for (int64_t i = 0; i < n;) {
      int64_t j = i;
      while (j + 1 < n && v[idx[(size_t)(j + 1)]] == v[idx[(size_t)i]]) j++;
      for (int64_t k = i; k <= j; k++) r2[(size_t)idx[(size_t)k]] = (i + 1) + (j + 1);  // 2 * mean rank
      i = j + 1;
    }
    return r2;
  };
  const std::vector<int64_t> rx = doubled_ranks(x), ry = doubled_ranks(y);
  // exact integer moments of the doubled ranks
  __int128 sx = 0, sy = 0, sxx = 0, syy = 0, sxy = 0;
  for (int64_t i = 0; i < n; i++) {
    const __int128 a = rx[(size_t)i], b = ry[(size_t)i];
    sx += a;
    sy += b;
    sxx += a * a;
    syy += b * b;
    sxy += a * b;
  }
  const __int128 N = n;
  const __int128 cxy = N * sxy - sx * sy, cxx = N * sxx - sx * sx, cyy = N * syy - sy * sy;
  if (cxx == 0 || cyy == 0) {
    *rho_out = std::nan("");
    return PEAT_OK;
  }
  const long double num = (long double)cxy, den = sqrtl((long double)cxx) * sqrtl((long double)cyy);
  *rho_out = (double)(num / den);
  return PEAT_OK;
}

peat_status_t peat_mean_std(const double* x, int64_t n, int ddof, double* mean_out, double* std_out) {
  if (!mean_out || !std_out || n < 0 || (n > 0 && !x)) return host_fail("null pointer or n < 0");
  if (ddof != 0 && ddof != 1) return host_fail("ddof must be 0 or 1");
  for (int64_t i = 0; i < n; i++)
    if (!std::isfinite(x[i])) return host_fail("a value is not finite");
  if (n == 0) {
    *mean_out = *std_out = std::nan("");
    return PEAT_OK;
  }
  // two passes with compensated (Neumaier) sums
  auto csum = [n](auto f) {
    double s = 0.0, c = 0.0;
    for (int64_t i = 0; i < n; i++) {
      const double v = f(i), t = s + v;
      c += std::fabs(s) >= std::fabs(v) ? (s - t) + v : (v - t) + s;
      s = t;
    }
    return s + c;
  };
  const double mean = csum([x](int64_t i) { return x[i]; }) / (double)n;
  *mean_out = mean;
  if (n <= ddof) {
    *std_out = std::nan("");
    return PEAT_OK;
  }
  const double ss = csum([x, mean](int64_t i) { return (x[i] - mean) * (x[i] - mean); });
  *std_out = std::sqrt(ss / (double)(n - ddof));
  return PEAT_OK;
}

peat_status_t peat_trend(const double* x, const double* y, int64_t n, double* slope_out, double* intercept_out,
                         double* r2_out, int64_t* used_out) {
  if (!slope_out || !intercept_out || !r2_out || n < 0 || (n > 0 && (!x || !y)))
    return host_fail("null pointer or n < 0");
  std::vector<double> lx, ly;
  for (int64_t i = 0; i < n; i++)
    if (std::isfinite(x[i]) && std::isfinite(y[i]) && x[i] > 0.0 && y[i] > 0.0) {
      lx.push_back(std::log(x[i]));
      ly.push_back(std::log(y[i]));
    }
  const int64_t m = (int64_t)lx.size();
  if (used_out) *used_out = m;
  *slope_out = *intercept_out = *r2_out = std::nan("");
  if (m < 2) return PEAT_OK;
  auto csum = [m](auto f) {  // compensated (Neumaier) sum of f(0..m-1)
    double s = 0.0, c = 0.0;
    for (int64_t i = 0; i < m; i++) {
      const double v = f(i), t = s + v;
      c += std::fabs(s) >= std::fabs(v) ? (s - t) + v : (v - t) + s;
      s = t;
    }
    return s + c;
  };
  const double mx = csum([&](int64_t i) { return lx[i]; }) / (double)m;
  const double my = csum([&](int64_t i) { return ly[i]; }) / (double)m;
  const double sxx = csum([&](int64_t i) { return (lx[i] - mx) * (lx[i] - mx); });
  const double sxy = csum([&](int64_t i) { return (lx[i] - mx) * (ly[i] - my); });
  const double syy = csum([&](int64_t i) { return (ly[i] - my) * (ly[i] - my); });
  if (!(sxx > 0.0)) return PEAT_OK;
  const double b = sxy / sxx, a0 = my - b * mx;
  *slope_out = b;
  *intercept_out = a0;
  if (syy > 0.0) {
    const double sse = csum([&](int64_t i) {
      const double r = ly[i] - (a0 + b * lx[i]);
      return r * r;
    });
    *r2_out = 1.0 - sse / syy;
  }
  return PEAT_OK;
}

peat_status_t peat_inject_compare(peat_handle_t h, const void* golden, int64_t n, peat_dtype_t dtype,
                                  const peat_inject_t* models, int nmodels, uint64_t seed, peat_tol_t tol,
                                  peat_stats_t* stats_out, uint64_t* hist_out, peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  if (own_compare(dtype)) return fail(h, PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  if (!dtype_bytes(dtype)) return fail(h, PEAT_ERR_INVALID_ARG, "bad dtype");
  if (n < 0) return fail(h, PEAT_ERR_INVALID_ARG, "n < 0");
  if (nmodels < 1 || nmodels > peat::INJ_MAX) return fail(h, PEAT_ERR_INVALID_ARG, "nmodels outside [1, 8]");
  if (!models) return fail(h, PEAT_ERR_INVALID_ARG, "models is NULL");
  InjSpec spec;
  spec.n = nmodels;
  spec.seed = seed;
  for (int m = 0; m < nmodels; m++) {
    const peat_inject_t& md = models[m];
    if (md.kind < PEAT_INJ_RZ || md.kind > PEAT_INJ_CAST_BF16_RTZ) return fail(h, PEAT_ERR_INVALID_ARG, "bad model kind");
    if (!peat::inj_elementwise(md.kind))
      return fail(h, PEAT_ERR_UNSUPPORTED, "fixed-count models (RZ, RV, BITFLIP) cannot be fused: inject, then compare");
    if (md.kind <= PEAT_INJ_SIGNFLIP) {
      if (!(md.x >= 0.0 && md.x <= 1.0)) return fail(h, PEAT_ERR_INVALID_ARG, "rate outside [0, 1]");
    } else if (md.kind <= PEAT_INJ_BIAS) {
      if (!std::isfinite(md.x) || !std::isfinite((float)md.x)) return fail(h, PEAT_ERR_INVALID_ARG, "parameter not finite");
    } else if (dtype != PEAT_F32) {
      return fail(h, PEAT_ERR_INVALID_ARG, "cast models apply to float32 tensors only");
    }
    peat::InjStep& st = spec.step[m];
    st.kind = md.kind;
    st.model = (uint32_t)m;
    const double t = std::floor(md.x * 4294967296.0);
    st.threshold = (uint64_t)std::min(std::max(t, 0.0), 4294967296.0);
    st.x = (float)md.x;
  }
  int64_t off[2] = {0, n};
  return compare_impl(h, golden, nullptr, off, 1, dtype, tol, stats_out, hist_out, stream, &spec);
}

peat_status_t peat_pseudo_error_inject(peat_handle_t h, void* dst, const void* src, int64_t n,
                                       peat_dtype_t dtype, const peat_inject_t* models, int nmodels,
                                       uint64_t seed, uint64_t* counts_out, peat_stream_t stream) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  if (own_compare(dtype)) return fail(h, PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  int B = dtype_bytes(dtype);
  if (!B) return fail(h, PEAT_ERR_INVALID_ARG, "bad dtype");
  if (n < 0 || nmodels < 0 || nmodels > 64) return fail(h, PEAT_ERR_INVALID_ARG, "n < 0 or nmodels outside [0, 64]");
  if (nmodels > 0 && (!models || !counts_out)) return fail(h, PEAT_ERR_INVALID_ARG, "models/counts_out is NULL");
  if (n > 0 && (!dst || !src)) return fail(h, PEAT_ERR_INVALID_ARG, "dst/src is NULL");
  if (dst != src && n > 0) {
    uintptr_t a = (uintptr_t)dst, b = (uintptr_t)src, len = (uintptr_t)n * B;
    if (a < b + len && b < a + len) return fail(h, PEAT_ERR_INVALID_ARG, "dst and src overlap partially");
  }
  const int width = B * 8;
  size_t need = 0;
  for (int m = 0; m < nmodels; m++) {
    const peat_inject_t& md = models[m];
    if (md.kind < PEAT_INJ_RZ || md.kind > PEAT_INJ_CAST_BF16_RTZ) return fail(h, PEAT_ERR_INVALID_ARG, "bad model kind");
    if (md.kind <= PEAT_INJ_BITFLIP) {
      if (md.k < 0 || md.k > n || md.k > (1 << 20)) return fail(h, PEAT_ERR_INVALID_ARG, "k outside [0, min(n, 2^20)]");
      if (md.kind == PEAT_INJ_BITFLIP && (md.bit_lo < 0 || md.bit_hi < md.bit_lo || md.bit_hi >= width))
        return fail(h, PEAT_ERR_INVALID_ARG, "bit range outside the element");
      need += 3 * (size_t)md.k;
    } else if (md.kind <= PEAT_INJ_SIGNFLIP) {
      if (!(md.x >= 0.0 && md.x <= 1.0)) return fail(h, PEAT_ERR_INVALID_ARG, "rate outside [0, 1]");
    } else if (md.kind <= PEAT_INJ_BIAS) {
      if (!std::isfinite(md.x) || !std::isfinite((float)md.x)) return fail(h, PEAT_ERR_INVALID_ARG, "parameter not finite");
    } else if (dtype != PEAT_F32) {
      return fail(h, PEAT_ERR_INVALID_ARG, "cast models apply to float32 tensors only");
    }
  }
  DeviceGuard dg(h->device);
  if (!dg.ok) return fail(h, PEAT_ERR_CUDA, "cudaSetDevice failed");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (nmodels > 0) {
    e = cudaMemsetAsync(counts_out, 0, sizeof(uint64_t) * (size_t)nmodels, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(counts)");
  }
  // Draw every fixed-count model's positions up front.  Staging layout per
  // model m: [positions k | aux k | values k] int64, then nmodels counts.
  // aux = RV source index; values = RV source values (filled on the device)
  // or, for BITFLIP, the bit indices as uint32.
  peat_status_t ps = grow_inject(h, need + (size_t)nmodels);
  if (ps != PEAT_OK) return ps;
  ps = wait_staging(h);
  if (ps != PEAT_OK) return ps;
  std::vector<size_t> base(nmodels, 0);
  size_t used = 0;
  for (int m = 0; m < nmodels; m++) {
    const peat_inject_t& md = models[m];
    h->h_inj[need + (size_t)m] = 0;
    if (md.kind > PEAT_INJ_BITFLIP) continue;
    int64_t k = md.k;
    base[m] = used;
    int64_t* pos = h->h_inj + used;
    int64_t* aux = pos + k;
    uint32_t* bits = reinterpret_cast<uint32_t*>(pos + 2 * k);
    std::unordered_set<int64_t> taken;
    taken.reserve((size_t)k * 2 + 1);
    int64_t got = 0;
    for (uint64_t j = 0; got < k; j++) {
      uint32_t ctr[4] = {(uint32_t)j, (uint32_t)(j >> 32), (uint32_t)m, 0x504F5331u}, w[4];
      philox_host(ctr, seed, w);
      int64_t p = (int64_t)mulhi64(((uint64_t)w[1] << 32) | w[0], (uint64_t)n);
      if (!taken.insert(p).second) continue;
      pos[got] = p;
      aux[got] = 0;
      if (md.kind == PEAT_INJ_RV)
        aux[got] = (int64_t)mulhi64(((uint64_t)w[3] << 32) | w[2], (uint64_t)n);
      else if (md.kind == PEAT_INJ_BITFLIP)
        bits[got] = (uint32_t)md.bit_lo + (uint32_t)(((uint64_t)w[2] * (uint64_t)(md.bit_hi - md.bit_lo + 1)) >> 32);
      got++;
    }
    h->h_inj[need + (size_t)m] = k;
    used += 3 * (size_t)k;
  }
  if (nmodels > 0) {
    e = cudaMemcpyAsync(h->d_inj, h->h_inj, (need + (size_t)nmodels) * sizeof(int64_t), cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(positions)");
  }
  // RV source values come from src before any model runs (src may be dst)
  for (int m = 0; m < nmodels; m++)
    if (models[m].kind == PEAT_INJ_RV && models[m].k > 0) {
      int64_t k = models[m].k;
      e = peat::launch_gather(dtype, src, h->d_inj + base[m] + k, h->d_inj + base[m] + 2 * k, k, st);
      if (e != cudaSuccess) return cuda_fail(h, e, "gather launch");
    }
  if (dst != src && n > 0) {
    e = cudaMemcpyAsync(dst, src, (size_t)n * B, cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(dst <- src)");
  }
  for (int m = 0; m < nmodels; m++) {
    const peat_inject_t& md = models[m];
    if (md.kind <= PEAT_INJ_BITFLIP) {
      int64_t k = md.k;
      if (k > 0) {
        peat::InjectScatterParams sp;
        sp.dst = dst;
        sp.src = src;
        sp.n = n;
        sp.kind = md.kind;
        sp.pos = h->d_inj + base[m];
        sp.from = h->d_inj + base[m] + 2 * k;
        sp.bit = reinterpret_cast<const uint32_t*>(h->d_inj + base[m] + 2 * k);
        sp.k = k;
        e = peat::launch_inject_scatter(dtype, sp, st);
        if (e != cudaSuccess) return cuda_fail(h, e, "inject scatter launch");
      }
      e = cudaMemcpyAsync(counts_out + m, h->d_inj + need + m, sizeof(uint64_t), cudaMemcpyDeviceToDevice, st);
      if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemcpyAsync(count)");
    } else {
      peat::InjectElemParams ep;
      ep.dst = dst;
      ep.src = src;
      ep.n = n;
      ep.kind = md.kind;
      ep.model = (uint32_t)m;
      ep.seed = seed;
      double t = std::floor(md.x * 4294967296.0);
      ep.threshold = (uint64_t)std::min(std::max(t, 0.0), 4294967296.0);
      ep.x = (float)md.x;
      ep.count = reinterpret_cast<unsigned long long*>(counts_out + m);
      e = peat::launch_inject_elem(dtype, ep, st);
      if (e != cudaSuccess) return cuda_fail(h, e, "inject launch");
    }
  }
  e = cudaEventRecord(h->staged, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaEventRecord");
  h->staged_pending = true;
  return PEAT_OK;
}

peat_status_t peat_compare_noalloc(const void* golden, const void* candidate, int64_t n, peat_dtype_t dtype,
                                   peat_tol_t tol, peat_stats_t* stats_out, uint64_t* hist_out,
                                   peat_stream_t stream) {
  g_null_error_is_noalloc = true;
  g_noalloc_error[0] = 0;
  if (own_compare(dtype)) return noalloc_fail(PEAT_ERR_UNSUPPORTED, FP8_ONLY);
  const int B = dtype_bytes(dtype);
  if (!B) return noalloc_fail(PEAT_ERR_INVALID_ARG, "dtype must be PEAT_F32, PEAT_F16 or PEAT_BF16");
  float rtol, atol;
  if (!round_tol(tol, &rtol, &atol))
    return noalloc_fail(PEAT_ERR_INVALID_ARG, "rtol and atol must be finite and >= 0 after rounding to float32");
  if (n < 0) return noalloc_fail(PEAT_ERR_INVALID_ARG, "n < 0");
  if (n > 0 && (!golden || !candidate)) return noalloc_fail(PEAT_ERR_INVALID_ARG, "golden/candidate is NULL");
  if (!stats_out) return noalloc_fail(PEAT_ERR_INVALID_ARG, "stats_out is NULL");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return noalloc_cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= NOALLOC_MAX_DEVICES) return noalloc_fail(PEAT_ERR_UNSUPPORTED, "device ordinal above 63");
  NoallocDevice& D = g_noalloc_dev[dev];
  if (!D.ready.load(std::memory_order_acquire)) {
    // first call on this device: find the scratch and configure the kernels
    std::lock_guard<std::mutex> lk(g_noalloc_setup);
    if (!D.ready.load(std::memory_order_relaxed)) {
      void* ptr = nullptr;
      e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
      if (e != cudaSuccess || !ptr) return noalloc_cuda_fail(e, "cudaGetSymbolAddress(scratch)");
      e = peat::compare_prepare();
      if (e != cudaSuccess) return noalloc_cuda_fail(e, "could not configure the compare kernels");
      e = register_digit_status(dev);
      if (e != cudaSuccess) return noalloc_cuda_fail(e, "could not set up the library's status word");
      int nsm = 0;
      e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess || nsm <= 0) return noalloc_cuda_fail(e, "cudaDeviceGetAttribute(SM count)");
      D.scratch = static_cast<NoallocScratch*>(ptr);
      D.nsm = nsm;
      D.ready.store(1, std::memory_order_release);
    }
  }
  if (digit_fault_pending()) return noalloc_fail(PEAT_ERR_INTERNAL, DIGIT_FAULT);
  NoallocScratch* S = D.scratch;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  peat::CompareParams p;
  std::memset(&p, 0, sizeof(p));
  p.g = golden;
  p.c = candidate;
  p.n_total = n;
  p.nseg = 1;
  const uintptr_t ag = reinterpret_cast<uintptr_t>(golden), ac = reinterpret_cast<uintptr_t>(candidate);
  if (n > 0 && ag % B == 0 && ac % B == 0 && ag % 16 == ac % 16)
    p.p0 = (int64_t)(((16 - ag % 16) % 16) / B);
  else
    p.p0 = -1;
  const int max_ctas = std::min(NOALLOC_MAX_CTAS, D.nsm * peat::compare_ctas_per_sm());
  p.nctas = (int)std::max<int64_t>(1, std::min<int64_t>(max_ctas, (n + 4095) / 4096));
  // the per-CTA element offsets of stage 1 are 32-bit
  if (n / p.nctas >= ((int64_t)1 << 31) - 64)
    return noalloc_fail(PEAT_ERR_UNSUPPORTED, "n is too large for one call (2^31 - 64 elements or more per CTA)");
  p.offsets = S->offsets;
  p.bounds = S->bounds;
  p.partials = S->partials;
  p.acc = &S->acc;
  p.glist = S->glist;
  p.has_empty = n == 0;
  p.status = &S->status;
  p.wait_limit = g_noalloc_wait_limit.load(std::memory_order_relaxed);
  p.rtol = rtol;
  p.atol = atol;
  p.stats = stats_out;
  p.hist = hist_out;
  // the bounds kernel also clears the status word: a wait that expired in an
  // earlier call must not mark this call's outputs
  e = peat::launch_bounds_on_device(dtype, S->offsets, S->bounds, p.nctas, n, p.p0, &S->status, st);
  if (e != cudaSuccess) return noalloc_cuda_fail(e, "bounds launch");
  e = peat::launch_compare(dtype, p, st);
  if (e != cudaSuccess) {
    cudaMemsetAsync(&S->acc, 0, sizeof(S->acc), st);  // no partial totals may survive into the next call
    return noalloc_cuda_fail(e, "compare launch");
  }
  return PEAT_OK;
}

peat_status_t peat_set_stage1_event(peat_handle_t h, void* event) {
  if (!h) return PEAT_ERR_INVALID_ARG;
  h->stage1_event = event;
  return PEAT_OK;
}

void peat_test_noalloc_expire_waits(int on) { g_noalloc_wait_limit.store(on ? 0u : (1u << 24)); }

double peat_test_quot_rn(uint64_t w_hi, uint64_t w_lo, int32_t sticky, int32_t e, uint64_t d) {
  if (d == 0 || !(w_hi >> 63)) return std::nan("");
  return peat::test_quot_rn(w_hi, w_lo, sticky, e, d);
}

int32_t peat_test_for_digits(uint64_t m_lo, uint64_t m_hi, int32_t e, int32_t neg, int64_t* digits_out) {
  if (!digits_out) return -1;
  return peat::test_for_digits(m_lo, m_hi, e, neg, digits_out);
}

const char* peat_last_error(peat_handle_t h) {
  if (!h) return g_null_error_is_noalloc ? g_noalloc_error : g_create_error.c_str();
  return h->err.c_str();
}

}  // extern "C"
