// isclose pass counts over a grid of tolerances for binary64 pairs (Section
// III-A; Fig. 5's FP32-FP64 comparison once the float32 side is widened
// exactly): the structure of the float32 grid kernel (a warp queue of the
// differing finite pairs, a binary search per atol bounded by the previous
// atol's result, a shared histogram of first accepting rtols), with the
// binary64 difference as an exact two-term pair and the exact binary64
// tolerance test.
#include <cstdint>

#include "exact64.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

using namespace x64;

constexpr int TB = 256, NW = TB / 32;
constexpr int QCAP = 64;
constexpr int NBIN = 2 * ISC_MAX;

struct QE64 {
  Mag a;
  double ag;
};

struct Isc64Smem {
  double R[ISC_MAX], A[ISC_MAX];
  unsigned H[NBIN];
  QE64 q[NW][QCAP];
};

// kind 0 accepted by every tolerance (EXACT), 1 by none, 2 finite and different
__device__ __forceinline__ int classify64(uint64_t G, uint64_t C, Mag& a, double& ag) {
  if (G == C) return 0;
  const uint64_t INF = 0x7FF0000000000000ull;
  const uint64_t mg = G & 0x7FFFFFFFFFFFFFFFull, mc = C & 0x7FFFFFFFFFFFFFFFull;
  if (mg >= INF || mc >= INF) return (mg > INF && mc > INF) ? 0 : 1;
  if ((mg | mc) == 0) return 0;  // +0 and -0 (the bit patterns differ)
  const double gd = from_bits64(G), cd = from_bits64(C);
  bool dneg;
  a = diff64(gd, cd, dneg);
  ag = from_bits64(mg);
  return 2;
}

__device__ __forceinline__ void run_batch64(const IscParams& p, Isc64Smem& sm, const QE64& e, bool valid) {
  const int nb = p.nr + 1;
  int prev = valid ? p.nr : 0;
  for (int j = 0; j < p.na; j++) {
    const unsigned vmask = __ballot_sync(0xFFFFFFFFu, valid && prev > 0);
    if (vmask == 0u) {
      const int nvalid = __popc(__ballot_sync(0xFFFFFFFFu, valid));
      if ((threadIdx.x & 31) == 0)
        for (int jj = j; jj < p.na; jj++) atomicAdd(&sm.H[jj * nb], (unsigned)nvalid);
      return;
    }
    int f = prev;
    if (valid && prev > 0) {
      int lo = 0, hi = prev;
      const double at = sm.A[j];
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (within64(e.a, e.ag, sm.R[mid], at)) hi = mid;
        else lo = mid + 1;
      }
      f = lo;
    }
    prev = f;
    const int key = valid ? f : -1;
    const unsigned grp = __match_any_sync(0xFFFFFFFFu, key);
    if (valid && (threadIdx.x & 31) == __ffs(grp) - 1) atomicAdd(&sm.H[j * nb + f], (unsigned)__popc(grp));
  }
}

__device__ __forceinline__ void pair_slot64(const IscParams& p, Isc64Smem& sm, uint64_t G, uint64_t C, bool ok,
                                            int& qn, uint32_t& nexact) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  Mag a{0.0, 0.0, 0};
  double ag = 0.0;
  const int kind = ok ? classify64(G, C, a, ag) : 1;
  nexact += kind == 0;
  const unsigned m = __ballot_sync(0xFFFFFFFFu, kind == 2);
  if (m == 0u) return;
  if (kind == 2) sm.q[warp][qn + __popc(m & ((1u << lane) - 1u))] = QE64{a, ag};
  qn += __popc(m);
  if (qn < 32) return;
  __syncwarp();
  const QE64 e = sm.q[warp][lane];
  __syncwarp();
  if (lane < qn - 32) sm.q[warp][lane] = sm.q[warp][32 + lane];
  qn -= 32;
  __syncwarp();
  run_batch64(p, sm, e, true);
}

__global__ void __launch_bounds__(TB) isclose_grid64(IscParams p) {
  __shared__ Isc64Smem sm;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < ISC_MAX; i += TB) {
    sm.R[i] = i < p.nr ? (double)p.rtol[i] : 0.0;
    sm.A[i] = i < p.na ? (double)p.atol[i] : 0.0;
  }
  for (int i = threadIdx.x; i < NBIN; i += TB) sm.H[i] = 0u;
  __syncthreads();
  const int64_t stride = (int64_t)gridDim.x * TB;
  const int64_t gt = (int64_t)blockIdx.x * TB + threadIdx.x;
  int qn = 0;
  uint32_t nexact = 0;
  // rounds of one 16-byte vector (two pairs) per thread, whole warps in every round
  for (int64_t v = gt; __any_sync(0xFFFFFFFFu, v < p.nvec); v += stride) {
    const bool ok = v < p.nvec;
    ulonglong2 gv = make_ulonglong2(0, 0), cv = gv;
    if (ok) {
      gv = __ldg(reinterpret_cast<const ulonglong2*>(reinterpret_cast<const char*>(p.g) + (p.p0 + v * 2) * 8));
      cv = __ldg(reinterpret_cast<const ulonglong2*>(reinterpret_cast<const char*>(p.c) + (p.p0 + v * 2) * 8));
    }
    if (__all_sync(0xFFFFFFFFu, !ok || (gv.x == cv.x && gv.y == cv.y))) {
      nexact += ok ? 2 : 0;
      continue;
    }
    pair_slot64(p, sm, gv.x, cv.x, ok, qn, nexact);
    pair_slot64(p, sm, gv.y, cv.y, ok, qn, nexact);
  }
  // elements outside the vector grid
  const int64_t head = p.p0 >= 0 ? p.p0 : p.n, tail = p.p0 >= 0 ? p.p0 + p.nvec * 2 : p.n;
  const int64_t ns = head + (p.n - tail);
  for (int64_t r = gt - lane; r < ns; r += stride) {
    const int64_t idx = r + lane;
    const bool ok = idx < ns;
    uint64_t G = 0, C = 0;
    if (ok) {
      const int64_t i = idx < head ? idx : tail + (idx - head);
      G = __ldg(reinterpret_cast<const unsigned long long*>(p.g) + i);
      C = __ldg(reinterpret_cast<const unsigned long long*>(p.c) + i);
    }
    pair_slot64(p, sm, G, C, ok, qn, nexact);
  }
  if (qn > 0) {
    __syncwarp();
    const QE64 e = sm.q[warp][lane < qn ? lane : 0];
    run_batch64(p, sm, e, lane < qn);
  }
  const uint32_t ne = __reduce_add_sync(0xFFFFFFFFu, nexact);
  if (lane == 0 && ne)
    for (int j = 0; j < p.na; j++) atomicAdd(&sm.H[j * (p.nr + 1)], ne);
  __syncthreads();
  for (int c = threadIdx.x; c < p.ncells; c += TB) {
    const int i = c / p.na, j = c - i * p.na;
    unsigned long long cnt = 0;
    for (int f = 0; f <= i; f++) cnt += sm.H[j * (p.nr + 1) + f];
    if (cnt) atomicAdd(p.counts + i * p.na + p.aperm[j], cnt);
  }
}

}  // namespace

cudaError_t launch_isclose64(const IscParams& p, int nctas, cudaStream_t s) {
  isclose_grid64<<<nctas, TB, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace peat
