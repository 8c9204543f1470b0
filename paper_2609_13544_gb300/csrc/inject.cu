// Seeded pseudo-error injection on sm_103a (the Inject step of Alg. 1 and
// Alg. 2; error models of Section IV-A -- FP16 cast, random value, random
// zero -- and Section II-B -- random bit flip, random NaN -- plus Gaussian
// noise, bias and sign flips).
//
// Element-wise models run one grid-stride pass each, a thread per block of
// four elements (one Philox4x32-10 draw, see inject_models.cuh); fixed-count
// models (RZ, RV, BITFLIP) scatter at positions drawn on the host.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>

#include "inject_models.cuh"
#include <nvtx3/nvToolsExt.h>
#include "peat_internal.h"

namespace peat {
namespace {

using namespace inj;

template <int DT, int K>
__global__ void __launch_bounds__(256) inject_elem(InjectElemParams p) {
  constexpr int B = DT == PEAT_F32 ? 4 : 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const uint32_t k0 = (uint32_t)p.seed, k1 = (uint32_t)(p.seed >> 32);
  const int64_t nfull = p.n >> 2;  // whole blocks of four
  const bool vec = (reinterpret_cast<uintptr_t>(p.dst) % (4 * B)) == 0;
  uint32_t fired = 0;
  for (int64_t d = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; d < nfull; d += stride) {
    const int64_t i0 = d << 2;
    uint32_t e[4];
    if (vec) {
      if constexpr (B == 4) {
        const uint4 v = reinterpret_cast<const uint4*>(p.dst)[d];
        e[0] = v.x, e[1] = v.y, e[2] = v.z, e[3] = v.w;
      } else {
        const uint2 v = reinterpret_cast<const uint2*>(p.dst)[d];
        e[0] = v.x & 0xFFFFu, e[1] = v.x >> 16, e[2] = v.y & 0xFFFFu, e[3] = v.y >> 16;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 4; j++) e[j] = ld_bits<DT>(p.dst, i0 + j);
    }
    uint32_t mask;
    fired += apply_blocks<DT, K, 1>(e, i0, p.model, p.threshold, p.x, k0, k1, &mask);
    if (!mask) continue;
    if (vec) {
      if constexpr (B == 4) reinterpret_cast<uint4*>(p.dst)[d] = make_uint4(e[0], e[1], e[2], e[3]);
      else reinterpret_cast<uint2*>(p.dst)[d] = make_uint2(e[0] | (e[1] << 16), e[2] | (e[3] << 16));
    } else {
#pragma unroll
      for (int j = 0; j < 4; j++)
        if (mask >> j & 1u) st_bits<DT>(p.dst, i0 + j, e[j]);
    }
  }
  // the last n mod 4 elements, one thread each
  const int64_t gt = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (gt < (p.n & 3)) {
    const int64_t i = (nfull << 2) + gt;
    bool f;
    const uint32_t nb = apply_one<DT, K>(ld_bits<DT>(p.dst, i), i, p.model, p.threshold, p.x, k0, k1, f);
    if (f) {
      fired++;
      st_bits<DT>(p.dst, i, nb);
    }
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
  int64_t blocks = ((p.n + 3) / 4 + 255) / 256;
  if (blocks > 152 * 16) blocks = 152 * 16;
  nvtxRangePushA("peat pseudo-error inject");
  struct Pop {
    ~Pop() { nvtxRangePop(); }
  } pop;
  switch (p.kind) {
    case PEAT_INJ_NAN_INF: inject_elem<DT, PEAT_INJ_NAN_INF><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_SIGNFLIP: inject_elem<DT, PEAT_INJ_SIGNFLIP><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_REL_GAUSS: inject_elem<DT, PEAT_INJ_REL_GAUSS><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_ADD_GAUSS: inject_elem<DT, PEAT_INJ_ADD_GAUSS><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_BIAS: inject_elem<DT, PEAT_INJ_BIAS><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_CAST_F16_RNE: inject_elem<DT, PEAT_INJ_CAST_F16_RNE><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_CAST_F16_RTZ: inject_elem<DT, PEAT_INJ_CAST_F16_RTZ><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_CAST_BF16_RNE: inject_elem<DT, PEAT_INJ_CAST_BF16_RNE><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case PEAT_INJ_CAST_BF16_RTZ: inject_elem<DT, PEAT_INJ_CAST_BF16_RTZ><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}
template <int DT>
cudaError_t scatter_t(const InjectScatterParams& p, cudaStream_t s) {
  if (p.k <= 0) return cudaSuccess;
  nvtxRangePushA("peat pseudo-error inject (fixed-count scatter)");
  inject_scatter<DT><<<(unsigned)((p.k + 255) / 256), 256, 0, s>>>(p);
  nvtxRangePop();
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
