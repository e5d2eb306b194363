// Launch helpers shared by the per-N translation units.
#pragma once

#include "kd_kernels.cuh"
#include "kd_ops.h"

namespace kd {

// Opt the kernel in to its dynamic shared memory (> 48 KB for large N).  Done on
// every launch: the attribute is per function and per device, and the call
// costs about a microsecond next to millisecond-scale kernels.
template <class K>
inline cudaError_t prepare(K kernel, size_t smem) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

template <class K>
inline int occupancy(K kernel, int threads, size_t smem) {
  if (prepare(kernel, smem) != cudaSuccess) return 0;
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, threads, smem) != cudaSuccess) return 0;
  return nb;
}

template <class PL>
struct Ops {
  static cudaError_t decompose(const DecParams& p, const BatchParams* bp, int grid, cudaStream_t s) {
    auto k = p.trace ? decompose_kernel<PL, true> : decompose_kernel<PL, false>;
    cudaError_t e = prepare(k, PL::SMEM);
    if (e != cudaSuccess) return e;
    if (bp) {
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, *bp);
    } else {
      BatchParams none{};
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, none);
    }
    return cudaGetLastError();
  }
  static cudaError_t reconstruct(const RecParams& p, const RecBatch* rb, int grid, cudaStream_t s) {
    auto k = reconstruct_kernel<PL>;
    cudaError_t e = prepare(k, PL::SMEM);
    if (e != cudaSuccess) return e;
    if (rb) {
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, *rb);
    } else {
      RecBatch none{};
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, none);
    }
    return cudaGetLastError();
  }
  static cudaError_t apply(const ApplyParams& p, const ApplyBatch* ab, int grid, cudaStream_t s) {
    auto k = apply_p_kernel<PL>;
    cudaError_t e = prepare(k, PL::SMEM);
    if (e != cudaSuccess) return e;
    if (ab) {
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, *ab);
    } else {
      ApplyBatch none{};
      k<<<grid, PL::THREADS, PL::SMEM, s>>>(p, none);
    }
    return cudaGetLastError();
  }
  static cudaError_t setup(float2* twt, uint32_t* eps, uint32_t* status, uint64_t seed, int64_t, cudaStream_t s) {
    constexpr int threads = 256;
    constexpr int work = PL::TWN > (PL::N + 31) / 32 ? PL::TWN : (PL::N + 31) / 32;
    constexpr int blocks = (work + threads - 1) / threads;
    setup_kernel<PL><<<blocks, threads, 0, s>>>(twt, eps, status, seed);
    return cudaGetLastError();
  }
  static int ctas_per_sm(int which, int64_t) {
    if (which == 0) return occupancy(decompose_kernel<PL, false>, PL::THREADS, PL::SMEM);
    if (which == 1) return occupancy(apply_p_kernel<PL>, PL::THREADS, PL::SMEM);
    return occupancy(reconstruct_kernel<PL>, PL::THREADS, PL::SMEM);
  }
  static const PlanOps* ops() {
    static const PlanOps o{PL::N, PL::THREADS, PL::Q, PL::SMEM, PL::UMODE == UGMEM, PL::BATCH, PL::TWN,
                           &Ops::ctas_per_sm, &Ops::decompose, &Ops::apply, &Ops::reconstruct, &Ops::setup};
    return &o;
  }
};

}  // namespace kd
