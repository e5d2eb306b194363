// kd_decompose_static: kd_decompose for callers that cannot allocate device memory.
//
// Some callers have no way to hand the library a workspace: a plugin loaded into a
// host application that owns every device allocation through its own pool (and
// forbids direct cudaMalloc), or a latency-critical loop where cudaMalloc's implicit
// device synchronisation is not acceptable.  This entry point runs the same
// decomposition kernels with their scratch (the per-call sign mask, the transform
// twiddles and the device status word) in a file-scope static device array instead
// of a caller workspace, so it allocates nothing.
//
// Limits and sharing:
//  - the array holds the tables of one vector length up to 8192; after the same
//    argument checks as kd_decompose, longer vectors (and lengths whose tables do
//    not fit) are rejected with KD_ERR_WORKSPACE before anything is enqueued;
//  - every GPU that loads the library holds the array until the process exits;
//  - all calls share it and it keeps the last call's contents; each call rewrites
//    the tables and clears the status word on its own stream before its kernel
//    runs, so calls that overlap on the GPU (different streams, or a second call
//    enqueued on another stream before the first finished) race;
//  - the first call on a device resolves the array's device address with
//    cudaGetSymbolAddress (once per device, with that device current); make that
//    first call before any stream capture;
//  - a non-finite input sets the status word at the start of the array, which
//    kd_read_status_static copies back (after synchronising the caller's stream).
#include <mutex>

#include "kashin.h"
#include "kd_kernels.cuh"
#include "kd_ops.h"

namespace kd {
namespace {

constexpr int64_t kStaticMaxN = 8192;
constexpr size_t kStaticBytes = 160 * 1024;  // >= kd_workspace_size(n) for every n <= 8192 (checked per call)
constexpr int kMaxDevices = 64;

// Host code must not pass `kd_static_scratch` itself to a kernel: on the host that
// name is only a stand-in for the symbol, not a device address.
static __device__ __align__(256) unsigned char kd_static_scratch[kStaticBytes];

std::mutex g_mu;
void* g_scratch[kMaxDevices] = {};

// Device address of the static scratch on the current device (resolved once).
cudaError_t scratch_on_current_device(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, kd_static_scratch);
    if (e != cudaSuccess) return e;
    g_scratch[dev] = p;
  }
  *out = g_scratch[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_decompose_static(const void* w, kd_dtype dtype, kd_layout layout, int64_t n, int64_t m,
                                         int64_t ld, uint64_t sign_seed, int iters, int kmeans_iters,
                                         uint32_t* codes_u, uint32_t* codes_v, float* centres_u, float* centres_v,
                                         float* coeffs, float* u, float* vhat, float* resid, int8_t* trace,
                                         void* stream) {
  // the caller's arguments first, exactly as kd_decompose checks them
  const kd_status chk = (kd_status)kd::check_decompose_args(w, dtype, layout, n, m, ld, iters, kmeans_iters, codes_u,
                                                            codes_v, centres_u, centres_v, coeffs, u, vhat, resid);
  if (chk != KD_OK) return chk;
  // then the array's limits
  if (n > kd::kStaticMaxN) return KD_ERR_WORKSPACE;
  const size_t need = kd_workspace_size(n);
  if (need == 0) return KD_ERR_CUDA;
  if (need > kd::kStaticBytes) return KD_ERR_WORKSPACE;
  // and only then the device address (loads the module on first use)
  void* scratch = nullptr;
  if (kd::scratch_on_current_device(&scratch) != cudaSuccess) return KD_ERR_CUDA;
  return kd_decompose(w, dtype, layout, n, m, ld, sign_seed, iters, kmeans_iters, codes_u, codes_v, centres_u,
                      centres_v, coeffs, u, vhat, resid, trace, scratch, kd::kStaticBytes, stream);
}

// The status word sits at the start of the array (offset 0 of the workspace layout,
// which kd_decompose's set-up clears before every kernel).
extern "C" kd_status kd_read_status_static(void* stream) {
  void* scratch = nullptr;
  if (kd::scratch_on_current_device(&scratch) != cudaSuccess) return KD_ERR_CUDA;
  return kd_read_status(scratch, stream);
}
