// C ABI of libkashin (declared in include/kashin.h): argument validation, the
// per-call workspace layout, table set-up and kernel dispatch by vector length.
#include <cstring>

#include "kashin.h"
#include "kd_kernels.cuh"
#include "kd_ops.h"

namespace kd {
#define KD_PLAN(n) const PlanOps* plan_ops_##n();
KD_PLAN(16) KD_PLAN(32) KD_PLAN(64) KD_PLAN(128) KD_PLAN(256) KD_PLAN(512) KD_PLAN(768)
KD_PLAN(1024) KD_PLAN(1536) KD_PLAN(2048) KD_PLAN(3072) KD_PLAN(4096) KD_PLAN(8192)
KD_PLAN(11008) KD_PLAN(14336) KD_PLAN(16384)
#undef KD_PLAN

const PlanOps* tuned_plan_ops(int64_t n) {
  switch (n) {
    case 16: return plan_ops_16();
    case 32: return plan_ops_32();
    case 64: return plan_ops_64();
    case 128: return plan_ops_128();
    case 256: return plan_ops_256();
    case 512: return plan_ops_512();
    case 768: return plan_ops_768();
    case 1024: return plan_ops_1024();
    case 1536: return plan_ops_1536();
    case 2048: return plan_ops_2048();
    case 3072: return plan_ops_3072();
    case 4096: return plan_ops_4096();
    case 8192: return plan_ops_8192();
    case 11008: return plan_ops_11008();
    case 14336: return plan_ops_14336();
    case 16384: return plan_ops_16384();
    default: return nullptr;
  }
}

const PlanOps* plan_ops(int64_t n) {
  const PlanOps* ops = tuned_plan_ops(n);
  return ops ? ops : generic_plan_ops(n);
}

namespace {

constexpr size_t kAlign = 256;
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// A workspace must be non-null and 16-byte aligned (its tables are read with
// 128-bit loads); cudaMalloc and the caching allocators return 256-byte alignment.
inline bool ws_ok(const void* ws) { return ws && reinterpret_cast<uintptr_t>(ws) % 16 == 0; }

// Workspace layout: [status word | pad][sign bits, one set per matrix][access-ordered twiddles][u slots]
struct WsLayout {
  size_t status, eps, tw, uslots, total;
};

// sign bits of several matrices: set i at eps + i * words (batched launches)
struct SeedList {
  int count, words;
  int64_t n;
  uint64_t seed[kMaxBatch];
};

__global__ void eps_batch_kernel(uint32_t* eps, SeedList sl) {
  const int total = sl.count * sl.words;
  for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < total; g += gridDim.x * blockDim.x) {
    const int i = g / sl.words, wd = g - i * sl.words;
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; ++bb) {
      const int64_t j = (int64_t)wd * 32 + bb;
      if (j >= sl.n) break;
      bits |= (uint32_t)(splitmix64_mix(sl.seed[i] + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull) >> 63) << bb;
    }
    eps[g] = bits;
  }
}

int sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

// Most CTAs a decompose launch of this plan ever uses on the current device.
int max_decompose_ctas(const PlanOps* ops) {
  const int per = ops->ctas_per_sm(0, ops->n);
  const int sms = sm_count();
  if (per <= 0 || sms <= 0) return 0;
  return per * sms;
}

bool layout_of(const PlanOps* ops, WsLayout* L, int nsets = 1) {
  const size_t n = (size_t)ops->n;
  L->status = 0;
  L->eps = kAlign;
  L->tw = L->eps + align_up((size_t)nsets * ((n + 31) / 32) * sizeof(uint32_t));
  L->uslots = L->tw + align_up((size_t)ops->twn * sizeof(float2));
  size_t us = 0;
  if (ops->u_in_gmem) {
    const int ctas = max_decompose_ctas(ops);
    if (ctas <= 0) return false;
    us = align_up((size_t)ctas * ops->q * n * sizeof(float2));
  }
  L->total = L->uslots + us;
  return true;
}

kd_status setup(const PlanOps* ops, const WsLayout& L, void* ws, uint64_t seed, cudaStream_t s) {
  char* b = static_cast<char*>(ws);
  cudaError_t e = ops->setup(reinterpret_cast<float2*>(b + L.tw), reinterpret_cast<uint32_t*>(b + L.eps),
                             reinterpret_cast<uint32_t*>(b + L.status), seed, ops->n, s);
  return e == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

// Tables of a batched call: twiddles, status and sign set 0 from the first seed, then
// sign sets 1 .. count-1 (set i at eps + i * ceil(n / 32)).
kd_status setup_batch(const PlanOps* ops, const WsLayout& L, void* ws, const uint64_t* seeds, int count, int64_t n,
                      cudaStream_t s) {
  kd_status st = setup(ops, L, ws, seeds[0], s);
  if (st != KD_OK || count == 1) return st;
  SeedList sl;
  sl.count = count;
  sl.words = (int)((n + 31) / 32);
  sl.n = n;
  for (int i = 0; i < count; ++i) sl.seed[i] = seeds[i];
  const int total = count * sl.words;
  eps_batch_kernel<<<(total + 255) / 256, 256, 0, s>>>(reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + L.eps),
                                                       sl);
  return cudaGetLastError() == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

int grid_for(int64_t npairs, int q, int ctas_max) {
  const int64_t want = (npairs + q - 1) / q;
  return (int)(want < ctas_max ? want : ctas_max);
}

bool valid_dtype(int d) { return d == KD_F32 || d == KD_F16 || d == KD_BF16; }

// Blocks k and refinement iterations a call may ask for (keeps every step and trace
// row count far inside int range).
constexpr int kMaxIters = 1 << 16;

// Every pointer a decomposition reads or writes element-wise must be aligned to its
// element: the input to its dtype, the code words and fp32 outputs to 4 bytes.
bool aligned_to(const void* ptr, size_t a) { return reinterpret_cast<uintptr_t>(ptr) % a == 0; }
bool outputs_aligned(const void* w, int dtype, const void* codes_u, const void* codes_v, const void* centres_u,
                     const void* centres_v, const void* coeffs, const void* u, const void* vhat, const void* resid) {
  const size_t esz = dtype == KD_F32 ? 4 : 2;
  return aligned_to(w, esz) && aligned_to(codes_u, 4) && aligned_to(codes_v, 4) && aligned_to(centres_u, 4) &&
         aligned_to(centres_v, 4) && aligned_to(coeffs, 4) && aligned_to(u, 4) && aligned_to(vhat, 4) &&
         aligned_to(resid, 4);
}
bool valid_layout(int l) { return l == KD_VEC_ROWS || l == KD_VEC_COLUMNS; }

// Output rows that can be written in 16-byte stores (W_hat of kd_reconstruct).
bool rows_vec_ok(const void* out, int dtype, int layout, int64_t n, int64_t ld) {
  const int64_t esz = dtype == KD_F32 ? 4 : 2;
  return layout == KD_VEC_ROWS && aligned_to(out, 16) && (ld * esz) % 16 == 0 && (n * esz) % 16 == 0;
}

// A matrix whose vectors are contiguous rows starting on 16-byte boundaries: the
// decomposition stages each pair's rows into shared memory with bulk copies.
bool rows_bulk_ok(const void* w, int dtype, int layout, int64_t n, int64_t ld) {
  const int64_t esz = dtype == KD_F32 ? 4 : 2;
  return layout == KD_VEC_ROWS && aligned_to(w, 16) && (ld * esz) % 16 == 0 && (n * esz) % 16 == 0;
}

}  // namespace

int check_decompose_args(const void* w, int dtype, int layout, int64_t n, int64_t m, int64_t ld, int iters,
                         int kmeans_iters, const void* codes_u, const void* codes_v, const void* centres_u,
                         const void* centres_v, const void* coeffs, const void* u, const void* vhat,
                         const void* resid) {
  if (n <= 0 || m < 0 || iters < 0 || iters > kMaxIters || kmeans_iters < 0 || kmeans_iters > 64 ||
      !valid_dtype(dtype) || !valid_layout(layout))
    return KD_ERR_INVALID_ARG;
  if (!plan_ops(n)) return KD_ERR_UNSUPPORTED_N;
  if (layout == KD_VEC_ROWS ? ld < n : ld < m) return KD_ERR_INVALID_ARG;
  if (m > 0 && (!w || !codes_u || !codes_v || !centres_u || !centres_v)) return KD_ERR_INVALID_ARG;
  if (!outputs_aligned(w, dtype, codes_u, codes_v, centres_u, centres_v, coeffs, u, vhat, resid))
    return KD_ERR_INVALID_ARG;
  return KD_OK;
}
}  // namespace kd

using namespace kd;

extern "C" {

const char* kd_status_string(kd_status s) {
  switch (s) {
    case KD_OK: return "KD_OK";
    case KD_ERR_INVALID_ARG: return "KD_ERR_INVALID_ARG";
    case KD_ERR_UNSUPPORTED_N: return "KD_ERR_UNSUPPORTED_N";
    case KD_ERR_CUDA: return "KD_ERR_CUDA";
    case KD_ERR_NONFINITE: return "KD_ERR_NONFINITE";
    case KD_ERR_WORKSPACE: return "KD_ERR_WORKSPACE";
    case KD_ERR_TIMEOUT: return "KD_ERR_TIMEOUT";
    default: return "KD_ERR_UNKNOWN";
  }
}

const char* kd_version(void) { return "libkashin 0.1.0 (sm_103a)"; }

kd_status kd_supported(int64_t n) { return plan_ops(n) ? KD_OK : KD_ERR_UNSUPPORTED_N; }

int kd_tuned(int64_t n) { return tuned_plan_ops(n) ? 1 : 0; }

size_t kd_workspace_size(int64_t n) {
  const PlanOps* ops = plan_ops(n);
  if (!ops) return 0;
  WsLayout L;
  if (!layout_of(ops, &L)) return 0;
  return L.total;
}

kd_status kd_signs(uint64_t sign_seed, int64_t n, int8_t* eps_host) {
  if (n <= 0 || !eps_host) return KD_ERR_INVALID_ARG;
  for (int64_t j = 0; j < n; ++j) {
    uint64_t z = sign_seed + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    z = z ^ (z >> 31);
    eps_host[j] = (z >> 63) ? (int8_t)-1 : (int8_t)1;
  }
  return KD_OK;
}

kd_status kd_decompose(const void* w, kd_dtype dtype, kd_layout layout, int64_t n, int64_t m, int64_t ld,
                       uint64_t sign_seed, int iters, int kmeans_iters, uint32_t* codes_u, uint32_t* codes_v,
                       float* centres_u, float* centres_v, float* coeffs, float* u, float* vhat,
                       float* resid, int8_t* trace, void* workspace, size_t ws_bytes, void* stream) {
  const kd_status chk = (kd_status)check_decompose_args(w, dtype, layout, n, m, ld, iters, kmeans_iters, codes_u, codes_v,
                                             centres_u, centres_v, coeffs, u, vhat, resid);
  if (chk != KD_OK) return chk;
  const PlanOps* ops = plan_ops(n);
  WsLayout L;
  if (!layout_of(ops, &L)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kd_status st = setup(ops, L, workspace, sign_seed, s);
  if (st != KD_OK || m == 0) return st;
  char* b = static_cast<char*>(workspace);
  DecParams p;
  p.w = w;
  p.dtype = (int)dtype;
  p.layout = (int)layout;
  p.n = n;
  p.m = m;
  p.ld = ld;
  p.iters = iters;
  p.kmeans_iters = kmeans_iters;
  p.codes_u = codes_u;
  p.codes_v = codes_v;
  p.centres_u = centres_u;
  p.centres_v = centres_v;
  p.coeffs = coeffs;
  p.u = u;
  p.vhat = vhat;
  p.resid = resid;
  p.trace = trace;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.status = reinterpret_cast<uint32_t*>(b + L.status);
  p.uslots = ops->u_in_gmem ? reinterpret_cast<float2*>(b + L.uslots) : nullptr;
  p.npairs = (m + 1) / 2;
  p.bulk = rows_bulk_ok(w, dtype, layout, n, ld) ? 1 : 0;
  const int ctas = max_decompose_ctas(ops);
  if (ctas <= 0) return KD_ERR_CUDA;
  const int grid = grid_for(p.npairs, ops->q, ctas);
  return ops->decompose(p, nullptr, grid, s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

size_t kd_workspace_size_batch(int64_t n, int count) {
  const PlanOps* ops = plan_ops(n);
  if (!ops || count < 1 || count > KD_MAX_BATCH) return 0;
  WsLayout L;
  if (!layout_of(ops, &L, count)) return 0;
  return L.total;
}

kd_status kd_decompose_batch(const kd_matrix* mats, int count, kd_dtype dtype, kd_layout layout, int64_t n,
                             int iters, int kmeans_iters, void* workspace, size_t ws_bytes, void* stream) {
  static_assert(KD_MAX_BATCH == kMaxBatch, "batch limit of the header and the kernel");
  if (!mats || count < 1 || count > KD_MAX_BATCH || n <= 0 || iters < 0 || iters > kMaxIters ||
      kmeans_iters < 0 || kmeans_iters > 64 || !valid_dtype(dtype) || !valid_layout(layout))
    return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  BatchParams bp;
  bp.count = count;
  int64_t npairs = 0;
  for (int i = 0; i < count; ++i) {
    const kd_matrix& a = mats[i];
    if (a.m < 0 || (layout == KD_VEC_ROWS ? a.ld < n : a.ld < a.m)) return KD_ERR_INVALID_ARG;
    if (a.m > 0 && (!a.w || !a.codes_u || !a.codes_v || !a.centres_u || !a.centres_v)) return KD_ERR_INVALID_ARG;
    if (!outputs_aligned(a.w, dtype, a.codes_u, a.codes_v, a.centres_u, a.centres_v, a.coeffs, nullptr, nullptr,
                         nullptr))
      return KD_ERR_INVALID_ARG;
    BatchMat& b = bp.mat[i];
    b.w = a.w;
    b.m = a.m;
    b.ld = a.ld;
    b.pair0 = npairs;
    b.codes_u = a.codes_u;
    b.codes_v = a.codes_v;
    b.centres_u = a.centres_u;
    b.centres_v = a.centres_v;
    b.coeffs = a.coeffs;
    npairs += (a.m + 1) / 2;
  }
  WsLayout L;
  if (!layout_of(ops, &L, count)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!ops->batch) {
    // long vectors: one launch per matrix on the same workspace, in stream order
    for (int i = 0; i < count; ++i) {
      const kd_matrix& a = mats[i];
      const kd_status sti = kd_decompose(a.w, dtype, layout, n, a.m, a.ld, a.sign_seed, iters, kmeans_iters,
                                         a.codes_u, a.codes_v, a.centres_u, a.centres_v, a.coeffs, nullptr,
                                         nullptr, nullptr, nullptr, workspace, ws_bytes, stream);
      if (sti != KD_OK) return sti;
    }
    return KD_OK;
  }
  uint64_t seeds[KD_MAX_BATCH];
  for (int i = 0; i < count; ++i) seeds[i] = mats[i].sign_seed;
  kd_status st = setup_batch(ops, L, workspace, seeds, count, n, s);
  if (st != KD_OK) return st;
  char* b = static_cast<char*>(workspace);
  if (npairs == 0) return KD_OK;
  DecParams p;
  std::memset(&p, 0, sizeof(p));
  p.w = mats[0].w;
  p.dtype = (int)dtype;
  p.layout = (int)layout;
  p.n = n;
  p.m = mats[0].m;
  p.ld = mats[0].ld;
  p.iters = iters;
  p.kmeans_iters = kmeans_iters;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.status = reinterpret_cast<uint32_t*>(b + L.status);
  p.uslots = ops->u_in_gmem ? reinterpret_cast<float2*>(b + L.uslots) : nullptr;
  p.npairs = npairs;
  p.bulk = 1;
  for (int i = 0; i < count; ++i)
    if (mats[i].m > 0 && !rows_bulk_ok(mats[i].w, dtype, layout, n, mats[i].ld)) p.bulk = 0;
  const int ctas = max_decompose_ctas(ops);
  if (ctas <= 0) return KD_ERR_CUDA;
  const int grid = grid_for(p.npairs, ops->q, ctas);
  return ops->decompose(p, &bp, grid, s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

kd_status kd_apply_p(const float* x, float* y, int64_t n, int64_t m, uint64_t sign_seed, void* workspace,
                     size_t ws_bytes, void* stream) {
  if (n <= 0 || m < 0) return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  if (m > 0 && (!x || !y)) return KD_ERR_INVALID_ARG;
  if (!aligned_to(x, 4) || !aligned_to(y, 4)) return KD_ERR_INVALID_ARG;
  WsLayout L;
  if (!layout_of(ops, &L)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kd_status st = setup(ops, L, workspace, sign_seed, s);
  if (st != KD_OK || m == 0) return st;
  char* b = static_cast<char*>(workspace);
  ApplyParams p;
  p.x = x;
  p.y = y;
  p.n = n;
  p.m = m;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.npairs = (m + 1) / 2;
  const int per = ops->ctas_per_sm(1, n);
  const int sms = sm_count();
  if (per <= 0 || sms <= 0) return KD_ERR_CUDA;
  const int grid = grid_for(p.npairs, ops->q, per * sms);
  return ops->apply(p, nullptr, grid, s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

}  // extern "C"

namespace kd {
namespace {

// kd_apply_p_batch and kd_apply_p_prepared: with `prepared` the workspace already holds
// the twiddle table and sign set i of matrix i (kd_prepare_p); otherwise they are derived
// here from the matrices' seeds first.
kd_status apply_p_many(const kd_pmat* mats, int count, int64_t n, void* workspace, size_t ws_bytes, void* stream,
                       bool prepared) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || n <= 0) return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  ApplyBatch ab;
  ab.count = count;
  int64_t npairs = 0;
  for (int i = 0; i < count; ++i) {
    const kd_pmat& a = mats[i];
    if (a.m < 0) return KD_ERR_INVALID_ARG;
    if (a.m > 0 && (!a.x || !a.y)) return KD_ERR_INVALID_ARG;
    if (!aligned_to(a.x, 4) || !aligned_to(a.y, 4)) return KD_ERR_INVALID_ARG;
    ab.mat[i].x = a.x;
    ab.mat[i].y = a.y;
    ab.mat[i].m = a.m;
    ab.mat[i].pair0 = npairs;
    npairs += (a.m + 1) / 2;
  }
  WsLayout L;
  if (!layout_of(ops, &L, count)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!ops->batch && !prepared) {
    // long vectors and the run-time-length path: one launch per matrix, in stream order
    for (int i = 0; i < count; ++i) {
      const kd_status sti = kd_apply_p(mats[i].x, mats[i].y, n, mats[i].m, mats[i].sign_seed, workspace, ws_bytes,
                                       stream);
      if (sti != KD_OK) return sti;
    }
    return KD_OK;
  }
  if (!prepared) {
    uint64_t seeds[KD_MAX_BATCH];
    for (int i = 0; i < count; ++i) seeds[i] = mats[i].sign_seed;
    const kd_status st = setup_batch(ops, L, workspace, seeds, count, n, s);
    if (st != KD_OK) return st;
  }
  if (npairs == 0) return KD_OK;
  char* b = static_cast<char*>(workspace);
  const int per = ops->ctas_per_sm(1, n);
  const int sms = sm_count();
  if (per <= 0 || sms <= 0) return KD_ERR_CUDA;
  ApplyParams p;
  std::memset(&p, 0, sizeof(p));
  p.n = n;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  if (!ops->batch) {
    // one launch per matrix, each on its own prepared sign set
    const size_t words = (size_t)((n + 31) / 32);
    for (int i = 0; i < count; ++i) {
      if (mats[i].m == 0) continue;
      p.m = mats[i].m;
      p.x = mats[i].x;
      p.y = mats[i].y;
      p.eps = reinterpret_cast<const uint32_t*>(b + L.eps) + (size_t)i * words;
      p.npairs = (mats[i].m + 1) / 2;
      if (ops->apply(p, nullptr, grid_for(p.npairs, ops->q, per * sms), s) != cudaSuccess) return KD_ERR_CUDA;
    }
    return KD_OK;
  }
  p.m = mats[0].m;
  p.x = mats[0].x;
  p.y = mats[0].y;
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.npairs = npairs;
  return ops->apply(p, &ab, grid_for(p.npairs, ops->q, per * sms), s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

}  // namespace
}  // namespace kd

extern "C" {

kd_status kd_apply_p_batch(const kd_pmat* mats, int count, int64_t n, void* workspace, size_t ws_bytes,
                           void* stream) {
  return kd::apply_p_many(mats, count, n, workspace, ws_bytes, stream, false);
}

kd_status kd_prepare_p(const uint64_t* seeds, int count, int64_t n, void* workspace, size_t ws_bytes,
                       void* stream) {
  if (!seeds || count < 1 || count > KD_MAX_BATCH || n <= 0) return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  WsLayout L;
  if (!layout_of(ops, &L, count)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  return setup_batch(ops, L, workspace, seeds, count, n, static_cast<cudaStream_t>(stream));
}

kd_status kd_apply_p_prepared(const kd_pmat* mats, int count, int64_t n, void* workspace, size_t ws_bytes,
                              void* stream) {
  return kd::apply_p_many(mats, count, n, workspace, ws_bytes, stream, true);
}

kd_status kd_reconstruct(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                         const float* centres_v, int64_t n, int64_t m, uint64_t sign_seed, kd_dtype out_dtype,
                         kd_layout layout, void* w_hat, int64_t ld, void* workspace, size_t ws_bytes,
                         void* stream) {
  if (n <= 0 || m < 0 || !valid_dtype(out_dtype) || !valid_layout(layout)) return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  if (layout == KD_VEC_ROWS ? ld < n : ld < m) return KD_ERR_INVALID_ARG;
  if (m > 0 && (!codes_u || !codes_v || !centres_u || !centres_v || !w_hat)) return KD_ERR_INVALID_ARG;
  if (m > 0 && ((reinterpret_cast<uintptr_t>(centres_u) | reinterpret_cast<uintptr_t>(centres_v)) % 16 != 0))
    return KD_ERR_INVALID_ARG;
  if (!aligned_to(codes_u, 4) || !aligned_to(codes_v, 4) || !aligned_to(w_hat, out_dtype == KD_F32 ? 4 : 2))
    return KD_ERR_INVALID_ARG;
  WsLayout L;
  if (!layout_of(ops, &L)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kd_status st = setup(ops, L, workspace, sign_seed, s);
  if (st != KD_OK || m == 0) return st;
  char* b = static_cast<char*>(workspace);
  RecParams p;
  p.dtype = (int)out_dtype;
  p.layout = (int)layout;
  p.codes_u = codes_u;
  p.codes_v = codes_v;
  p.centres_u = centres_u;
  p.centres_v = centres_v;
  p.n = n;
  p.m = m;
  p.ld = ld;
  p.out = w_hat;
  p.vec = rows_vec_ok(w_hat, out_dtype, layout, n, ld) ? 1 : 0;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.npairs = (m + 1) / 2;
  const int per = ops->ctas_per_sm(2, n);
  const int sms = sm_count();
  if (per <= 0 || sms <= 0) return KD_ERR_CUDA;
  const int grid = grid_for(p.npairs, ops->q, per * sms);
  return ops->reconstruct(p, nullptr, grid, s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

kd_status kd_reconstruct_batch(const kd_recmat* mats, int count, int64_t n, kd_dtype out_dtype, kd_layout layout,
                               void* workspace, size_t ws_bytes, void* stream) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || n <= 0 || !valid_dtype(out_dtype) || !valid_layout(layout))
    return KD_ERR_INVALID_ARG;
  const PlanOps* ops = plan_ops(n);
  if (!ops) return KD_ERR_UNSUPPORTED_N;
  RecBatch rb;
  rb.count = count;
  int64_t npairs = 0;
  for (int i = 0; i < count; ++i) {
    const kd_recmat& a = mats[i];
    if (a.m < 0 || (layout == KD_VEC_ROWS ? a.ld < n : a.ld < a.m)) return KD_ERR_INVALID_ARG;
    if (a.m > 0 && (!a.codes_u || !a.codes_v || !a.centres_u || !a.centres_v || !a.w_hat)) return KD_ERR_INVALID_ARG;
    if (!aligned_to(a.centres_u, 16) || !aligned_to(a.centres_v, 16) || !aligned_to(a.codes_u, 4) ||
        !aligned_to(a.codes_v, 4) || !aligned_to(a.w_hat, out_dtype == KD_F32 ? 4 : 2))
      return KD_ERR_INVALID_ARG;
    RecMat& r = rb.mat[i];
    r.codes_u = a.codes_u;
    r.codes_v = a.codes_v;
    r.centres_u = a.centres_u;
    r.centres_v = a.centres_v;
    r.out = a.w_hat;
    r.m = a.m;
    r.ld = a.ld;
    r.pair0 = npairs;
    npairs += (a.m + 1) / 2;
  }
  WsLayout L;
  if (!layout_of(ops, &L, count)) return KD_ERR_CUDA;
  if (!ws_ok(workspace) || ws_bytes < L.total) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!ops->batch) {
    // long vectors: one launch per matrix on the same workspace, in stream order
    for (int i = 0; i < count; ++i) {
      const kd_recmat& a = mats[i];
      const kd_status sti = kd_reconstruct(a.codes_u, a.codes_v, a.centres_u, a.centres_v, n, a.m, a.sign_seed,
                                           out_dtype, layout, a.w_hat, a.ld, workspace, ws_bytes, stream);
      if (sti != KD_OK) return sti;
    }
    return KD_OK;
  }
  uint64_t seeds[KD_MAX_BATCH];
  for (int i = 0; i < count; ++i) seeds[i] = mats[i].sign_seed;
  kd_status st = setup_batch(ops, L, workspace, seeds, count, n, s);
  if (st != KD_OK || npairs == 0) return st;
  char* b = static_cast<char*>(workspace);
  RecParams p;
  std::memset(&p, 0, sizeof(p));
  p.dtype = (int)out_dtype;
  p.layout = (int)layout;
  p.n = n;
  p.m = mats[0].m;
  p.ld = mats[0].ld;
  p.twt = reinterpret_cast<const float2*>(b + L.tw);
  p.eps = reinterpret_cast<const uint32_t*>(b + L.eps);
  p.npairs = npairs;
  p.vec = 1;
  for (int i = 0; i < count; ++i)
    if (mats[i].m > 0 && !rows_vec_ok(mats[i].w_hat, out_dtype, layout, n, mats[i].ld)) p.vec = 0;
  const int per = ops->ctas_per_sm(2, n);
  const int sms = sm_count();
  if (per <= 0 || sms <= 0) return KD_ERR_CUDA;
  const int grid = grid_for(p.npairs, ops->q, per * sms);
  return ops->reconstruct(p, &rb, grid, s) == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

kd_status kd_read_status(const void* workspace, void* stream) {
  if (!ws_ok(workspace)) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t word = 0;
  if (cudaMemcpyAsync(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost, s) != cudaSuccess) return KD_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return KD_ERR_CUDA;
  // bit 1: a staged-input wait expired; bit 0: a non-finite input
  if (word & 2u) return KD_ERR_TIMEOUT;
  return (word & 1u) ? KD_ERR_NONFINITE : KD_OK;
}

}  // extern "C"
