// Measured FP32 throughput of this GPU, for the ALU roofline of the transform
// kernels: independent chains of packed FFMA2 in every thread of a full grid,
// timed with CUDA events on the caller's stream.  A fixed amount of work (no
// waits); a few milliseconds.
#include <cuda_runtime.h>

#include "kashin.h"

namespace kd {
namespace {

constexpr int kChains = 8;

__device__ float g_sink[256];  // written only if a chain ends on an impossible value

__global__ void __launch_bounds__(256) ffma2_chains(float* sink, int iters, float b, float c) {
  float2 a[kChains];
#pragma unroll
  for (int i = 0; i < kChains; ++i) a[i] = make_float2(threadIdx.x * 1e-3f + i, i * 0.5f);
  const float2 bb = make_float2(b, b), cc = make_float2(c, c);
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int i = 0; i < kChains; ++i) a[i] = __ffma2_rn(a[i], bb, cc);
  }
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < kChains; ++i) s += a[i].x + a[i].y;
  if (s == 12345.f) sink[threadIdx.x] = s;  // keeps the chains live; never true in practice
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_measure_fp32_peak(double* tflops, void* stream) {
  if (!tflops) return KD_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KD_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return KD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* sink = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void**>(&sink), kd::g_sink) != cudaSuccess) return KD_ERR_CUDA;
  cudaEvent_t e0, e1;
  if (cudaEventCreate(&e0) != cudaSuccess) return KD_ERR_CUDA;
  if (cudaEventCreate(&e1) != cudaSuccess) {
    cudaEventDestroy(e0);
    return KD_ERR_CUDA;
  }
  const int grid = sms * 8, block = 256, iters = 8192;
  kd::ffma2_chains<<<grid, block, 0, s>>>(sink, iters / 8, 1.0001f, 1e-7f);  // warm-up
  float best = 0.f;
  kd_status st = KD_OK;
  for (int rep = 0; rep < 3 && st == KD_OK; ++rep) {
    cudaEventRecord(e0, s);
    kd::ffma2_chains<<<grid, block, 0, s>>>(sink, iters, 1.0001f, 1e-7f);
    cudaEventRecord(e1, s);
    float ms = 0.f;
    if (cudaEventSynchronize(e1) != cudaSuccess || cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess) {
      st = KD_ERR_CUDA;
    } else if (best == 0.f || ms < best) {
      best = ms;
    }
  }
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (st != KD_OK || best <= 0.f) return KD_ERR_CUDA;
  // per thread per iteration: kChains FFMA2 = 2 kChains FMAs = 4 kChains flops
  const double flops = (double)grid * block * iters * kd::kChains * 4.0;
  *tflops = flops / (best * 1e-3) / 1e12;
  return KD_OK;
}
