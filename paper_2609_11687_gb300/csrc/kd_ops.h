// Host-side interface between the C ABI (kd_api.cu) and the per-N translation
// units (kd_plan_<N>.cu), each of which instantiates the kernels of one plan, and
// the run-time-length path (kd_generic.cu).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace kd {
struct DecParams;
struct BatchParams;
struct ApplyParams;
struct ApplyBatch;
struct RecParams;
struct RecBatch;

struct PlanOps {
  int n;
  int threads;      // threads per CTA
  int q;            // vector pairs per CTA per iteration
  size_t smem;      // dynamic shared memory per CTA
  bool u_in_gmem;   // u lives in per-team workspace slots
  bool batch;       // the decompose kernel takes several matrices per launch
  int twn;          // entries of the access-ordered twiddle table
  // CTAs of vector length n that fit on one SM (occupancy), 0 on error
  int (*ctas_per_sm)(int which, int64_t n);  // which: 0 decompose, 1 apply, 2 reconstruct
  // bp: the matrices of a batched launch, or nullptr for DecParams' single matrix
  cudaError_t (*decompose)(const DecParams&, const BatchParams* bp, int grid, cudaStream_t);
  // ab: the matrices of a batched launch (plans with batch only), or nullptr
  cudaError_t (*apply)(const ApplyParams&, const ApplyBatch* ab, int grid, cudaStream_t);
  // rb: the matrices of a batched launch, or nullptr for RecParams' single matrix
  cudaError_t (*reconstruct)(const RecParams&, const RecBatch* rb, int grid, cudaStream_t);
  // tables for one call of vector length n: twiddles (float2[twn]), sign bits, cleared status word
  cudaError_t (*setup)(float2* twt, uint32_t* eps, uint32_t* status, uint64_t seed, int64_t n, cudaStream_t);
};

// Argument checks of kd_decompose, in its order and with its status codes (a kd_status
// value): sizes, counts and enums, the plan for n, ld, required pointers, alignment.
// The workspace is not checked here.
int check_decompose_args(const void* w, int dtype, int layout, int64_t n, int64_t m, int64_t ld, int iters,
                         int kmeans_iters, const void* codes_u, const void* codes_v, const void* centres_u,
                         const void* centres_v, const void* coeffs, const void* u, const void* vhat,
                         const void* resid);

// The compiled plan of length n, else the run-time-length path (kd_generic.cu), else nullptr.
const PlanOps* plan_ops(int64_t n);
// The compiled plan of length n, or nullptr.
const PlanOps* tuned_plan_ops(int64_t n);
// The run-time-length path for n (any 1 <= n <= 16384 whose prime factors are in
// {2, 3, 5, 7, 11, 13, 43}), or nullptr.
const PlanOps* generic_plan_ops(int64_t n);
}  // namespace kd
