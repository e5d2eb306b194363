// kd_decompose_batch_host: the batched decomposition from host memory to host memory.
//
// A caller holding the weights on the host gets one call that enqueues, on its
// stream, the upload of every matrix into a caller-provided device staging buffer,
// the batched decomposition (kd_decompose_batch on the staged copies) and the
// download of the codes, centres and coefficients.  The library allocates nothing:
// the staging buffer and the workspace come from the caller, and each copy is one
// cudaMemcpyAsync.
#include <cstring>

#include "kashin.h"

namespace {

constexpr size_t kAlign = 256;
inline size_t up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Device staging of one matrix: [input][codes_u][codes_v][centres_u][centres_v][coeffs]
struct Stage {
  size_t in, cu, cv, eu, ev, co, end;
  size_t in_bytes, code_bytes, cent_bytes;
};

bool plan_stage(const kd_matrix_host& a, size_t base, int dtype, int layout, int64_t n, Stage* st) {
  if (a.m < 0 || a.ld < 0) return false;
  const size_t esz = dtype == KD_F32 ? 4 : 2;
  const size_t rows = layout == KD_VEC_ROWS ? (size_t)a.m : (size_t)n;
  st->in_bytes = rows * (size_t)a.ld * esz;
  st->code_bytes = (size_t)a.m * (size_t)((n + 15) / 16) * sizeof(uint32_t);
  st->cent_bytes = (size_t)a.m * 4 * sizeof(float);
  st->in = base;
  st->cu = up(st->in + st->in_bytes);
  st->cv = up(st->cu + st->code_bytes);
  st->eu = up(st->cv + st->code_bytes);
  st->ev = up(st->eu + st->cent_bytes);
  st->co = up(st->ev + st->cent_bytes);
  st->end = up(st->co + (a.coeffs ? st->cent_bytes : 0));
  return true;
}

bool valid_enums(int dtype, int layout) {
  return (dtype == KD_F32 || dtype == KD_F16 || dtype == KD_BF16) &&
         (layout == KD_VEC_ROWS || layout == KD_VEC_COLUMNS);
}

}  // namespace

extern "C" size_t kd_staging_size_host(const kd_matrix_host* mats, int count, kd_dtype dtype, kd_layout layout,
                                       int64_t n) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || n <= 0 || !valid_enums(dtype, layout)) return 0;
  size_t off = 0;
  for (int i = 0; i < count; ++i) {
    Stage st;
    if (!plan_stage(mats[i], off, dtype, layout, n, &st)) return 0;
    off = st.end;
  }
  return off;
}

extern "C" kd_status kd_decompose_batch_host(const kd_matrix_host* mats, int count, kd_dtype dtype,
                                             kd_layout layout, int64_t n, int iters, int kmeans_iters, void* staging,
                                             size_t staging_bytes, void* workspace, size_t ws_bytes, void* stream) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || n <= 0 || iters < 0 || iters > (1 << 16) || kmeans_iters < 0 ||
      kmeans_iters > 64 || !valid_enums(dtype, layout))
    return KD_ERR_INVALID_ARG;
  if (kd_supported(n) != KD_OK) return KD_ERR_UNSUPPORTED_N;
  for (int i = 0; i < count; ++i) {
    const kd_matrix_host& a = mats[i];
    if (a.m < 0 || (layout == KD_VEC_ROWS ? a.ld < n : a.ld < a.m)) return KD_ERR_INVALID_ARG;
    if (a.m > 0 && (!a.w || !a.codes_u || !a.codes_v || !a.centres_u || !a.centres_v)) return KD_ERR_INVALID_ARG;
  }
  const size_t need = kd_staging_size_host(mats, count, dtype, layout, n);
  if (!staging || reinterpret_cast<uintptr_t>(staging) % kAlign != 0 || staging_bytes < need)
    return KD_ERR_WORKSPACE;
  const size_t ws_need = kd_workspace_size_batch(n, count);
  if (ws_need == 0) return KD_ERR_CUDA;
  if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 16 != 0 || ws_bytes < ws_need) return KD_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* dev = static_cast<char*>(staging);
  kd_matrix dm[KD_MAX_BATCH];
  Stage st[KD_MAX_BATCH];
  size_t off = 0;
  for (int i = 0; i < count; ++i) {
    const kd_matrix_host& a = mats[i];
    plan_stage(a, off, dtype, layout, n, &st[i]);
    off = st[i].end;
    kd_matrix& d = dm[i];
    std::memset(&d, 0, sizeof(d));
    d.w = dev + st[i].in;
    d.m = a.m;
    d.ld = a.ld;
    d.sign_seed = a.sign_seed;
    d.codes_u = reinterpret_cast<uint32_t*>(dev + st[i].cu);
    d.codes_v = reinterpret_cast<uint32_t*>(dev + st[i].cv);
    d.centres_u = reinterpret_cast<float*>(dev + st[i].eu);
    d.centres_v = reinterpret_cast<float*>(dev + st[i].ev);
    d.coeffs = a.coeffs ? reinterpret_cast<float*>(dev + st[i].co) : nullptr;
  }
  // every argument the batched call checks has been checked above (the staged
  // pointers are 256-byte aligned), so nothing is enqueued on an argument error
  for (int i = 0; i < count; ++i) {
    if (mats[i].m == 0) continue;
    if (cudaMemcpyAsync(dev + st[i].in, mats[i].w, st[i].in_bytes, cudaMemcpyHostToDevice, s) != cudaSuccess)
      return KD_ERR_CUDA;
  }
  const kd_status r = kd_decompose_batch(dm, count, dtype, layout, n, iters, kmeans_iters, workspace, ws_bytes,
                                         stream);
  if (r != KD_OK) return r;
  for (int i = 0; i < count; ++i) {
    const kd_matrix_host& a = mats[i];
    if (a.m == 0) continue;
    const kd_matrix& d = dm[i];
    if (cudaMemcpyAsync(a.codes_u, d.codes_u, st[i].code_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemcpyAsync(a.codes_v, d.codes_v, st[i].code_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemcpyAsync(a.centres_u, d.centres_u, st[i].cent_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemcpyAsync(a.centres_v, d.centres_v, st[i].cent_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess)
      return KD_ERR_CUDA;
    if (a.coeffs &&
        cudaMemcpyAsync(a.coeffs, d.coeffs, st[i].cent_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess)
      return KD_ERR_CUDA;
  }
  return KD_OK;
}
