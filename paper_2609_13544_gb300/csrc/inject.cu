// Seeded pseudo-error injection on sm_103a (the Inject step of Alg. 1 and
// Alg. 2; error models of Section IV-A -- FP16 cast, random value, random
// zero -- and Section II-B -- random bit flip, random NaN -- plus Gaussian
// noise, bias and sign flips).
//
// Element-wise models run one grid-stride pass each; fixed-count models
// (RZ, RV, BITFLIP) scatter at positions drawn on the host.  Randomness is
// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, SC'11), counter-based, so
// element i of model m always sees the same four words.  Gaussian variates
// use Box-Muller with a natural log (atanh series after reduction to
// [sqrt(1/2), sqrt(2)]) and cos(2 pi u) (quadrant reduction on u, Taylor
// series on [-pi/4, pi/4]), every float32 operation written as an explicit
// correctly rounded intrinsic so the sequence of roundings is fixed.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>

#include "inject_models.cuh"
#include "peat_internal.h"

namespace peat {
namespace {

using namespace inj;

template <int DT>
__global__ void __launch_bounds__(256) inject_elem(InjectElemParams p) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const uint32_t k0 = (uint32_t)p.seed, k1 = (uint32_t)(p.seed >> 32);
  uint32_t fired = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < p.n; i += stride) {
    const uint32_t b = ld_bits<DT>(p.dst, i);
    bool f;
    const uint32_t nb = apply_model<DT>(b, i, p.kind, p.model, p.threshold, p.x, k0, k1, f);
    if (!f) continue;
    fired++;
    st_bits<DT>(p.dst, i, nb);
  }
  fired = __reduce_add_sync(0xFFFFFFFFu, fired);
  if ((threadIdx.x & 31) == 0 && fired) atomicAdd(p.count, (unsigned long long)fired);
}

template <int DT>
__global__ void __launch_bounds__(256) inject_scatter(InjectScatterParams p) {
  int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= p.k) return;
  int64_t i = p.pos[j];
  if (p.kind == PEAT_INJ_RZ) {
    st_bits<DT>(p.dst, i, 0u);
  } else if (p.kind == PEAT_INJ_RV) {
    st_bits<DT>(p.dst, i, (uint32_t)p.from[j]);  // the source value, gathered before any model ran
  } else {
    st_bits<DT>(p.dst, i, ld_bits<DT>(p.dst, i) ^ (1u << p.bit[j]));
  }
}

template <int DT>
__global__ void gather_values(const void* src, const int64_t* from, int64_t* out, int64_t k) {
  int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (j < k) out[j] = (int64_t)ld_bits<DT>(src, from[j]);
}

template <int DT>
cudaError_t elem_t(const InjectElemParams& p, cudaStream_t s) {
  if (p.n <= 0) return cudaSuccess;
  int64_t blocks = (p.n + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  inject_elem<DT><<<(unsigned)blocks, 256, 0, s>>>(p);
  return cudaGetLastError();
}
template <int DT>
cudaError_t scatter_t(const InjectScatterParams& p, cudaStream_t s) {
  if (p.k <= 0) return cudaSuccess;
  inject_scatter<DT><<<(unsigned)((p.k + 255) / 256), 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_inject_elem(int dtype, const InjectElemParams& p, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return elem_t<PEAT_F32>(p, s);
    case PEAT_F16: return elem_t<PEAT_F16>(p, s);
    case PEAT_BF16: return elem_t<PEAT_BF16>(p, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_inject_scatter(int dtype, const InjectScatterParams& p, cudaStream_t s) {
  switch (dtype) {
    case PEAT_F32: return scatter_t<PEAT_F32>(p, s);
    case PEAT_F16: return scatter_t<PEAT_F16>(p, s);
    case PEAT_BF16: return scatter_t<PEAT_BF16>(p, s);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gather(int dtype, const void* src, const int64_t* from, int64_t* out, int64_t k,
                          cudaStream_t s) {
  if (k <= 0) return cudaSuccess;
  unsigned blocks = (unsigned)((k + 255) / 256);
  switch (dtype) {
    case PEAT_F32: gather_values<PEAT_F32><<<blocks, 256, 0, s>>>(src, from, out, k); break;
    case PEAT_F16: gather_values<PEAT_F16><<<blocks, 256, 0, s>>>(src, from, out, k); break;
    case PEAT_BF16: gather_values<PEAT_BF16><<<blocks, 256, 0, s>>>(src, from, out, k); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace peat
