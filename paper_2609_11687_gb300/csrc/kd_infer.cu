// Dequantisation of one 2-bit factor plane (App. C, inference): the dense factor
// matrix U_q (or V_q) with entry i of vector j equal to centres[j][code_j(i)].
//
// App. C folds the layer product as  X W = X U_q + (X P) V_q = [X | XP] [U_q; V_q]:
// on hardware without 2-bit matrix units the factors are expanded once at load
// time and the product runs as an ordinary GEMM; kd_apply_p gives XP and
// kd_reconstruct gives W_hat = U_q + P V_q directly.
//
// Bound by HBM: per entry 1/4 byte of codes is read and 2 or 4 bytes are written.
// Row layout: one warp per vector, consecutive lanes writing consecutive 16-byte
// chunks (two per code word for 16-bit output, four for fp32), each lane with the
// code loads of four chunks in flight.  Column layout: consecutive threads take
// consecutive vectors of the same word, so every store instruction of a warp writes
// consecutive addresses.  One launch serves one plane (kd_dequantise) or up to
// KD_MAX_BATCH planes of one length (kd_dequantise_batch).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "kashin.h"

namespace kd {
namespace {

struct DeqParams {
  const uint32_t* codes;
  const float* centres;
  void* out;
  int64_t n, m, ld, words;  // words = ceil(n / 16) per vector
  int dtype, layout;
  int vec;                  // row layout: 16-byte stores are aligned
};

__device__ __forceinline__ void put(void* out, int dtype, int64_t idx, float v) {
  if (dtype == KD_F32) {
    static_cast<float*>(out)[idx] = v;
  } else if (dtype == KD_F16) {
    static_cast<__half*>(out)[idx] = __float2half_rn(v);
  } else {
    static_cast<__nv_bfloat16*>(out)[idx] = __float2bfloat16_rn(v);
  }
}

// Column layout, one CTA step b: code word w = b % words of vectors 256 (b / words) +
// threadIdx.x (consecutive threads store to consecutive addresses).
__device__ __forceinline__ void dequant_col_step(const DeqParams& p, int64_t b) {
  const int64_t jb = b / p.words;
  const int64_t w = b - jb * p.words;
  const int64_t j = jb * 256 + threadIdx.x;
  if (j >= p.m) return;
  const uint32_t code = __ldg(p.codes + j * p.words + w);
  const float4 c = __ldg(reinterpret_cast<const float4*>(p.centres) + j);
  const int64_t i0 = 16 * w;
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    if (i0 + e < p.n) {
      const uint32_t q = (code >> (2 * e)) & 3u;
      const float lo = (q & 1u) ? c.y : c.x;
      const float hi = (q & 1u) ? c.w : c.z;
      put(p.out, p.dtype, (i0 + e) * p.ld + j, (q & 2u) ? hi : lo);
    }
  }
}

int64_t col_steps(const DeqParams& p) { return p.words * ((p.m + 255) / 256); }

// Several planes of one vector length in one launch: plane i owns the work units
// [first[i], first[i + 1]) (its vectors, one warp each, in the row layout; its
// column steps, one CTA each, in the column layout); the grid strides over all of
// them.
struct DeqBatch {
  int count;
  int64_t first[KD_MAX_BATCH + 1];
  DeqParams p[KD_MAX_BATCH];
};

__device__ __forceinline__ int plane_of(const DeqBatch& bt, int64_t b) {
  int i = 0;
  while (i + 1 < bt.count && b >= bt.first[i + 1]) ++i;
  return i;
}

// Output chunk `part` (EPT = 16 / TPW entries, 16 bytes when vectorised) of code word
// w of vector j, from the word cw and the centres c.
template <int TPW>
__device__ __forceinline__ void dequant_chunk(const DeqParams& p, int64_t j, int w, int part, uint32_t cw,
                                              float4 c) {
  constexpr int EPT = 16 / TPW;
  cw >>= 2 * EPT * part;
  float v[EPT];
#pragma unroll
  for (int e = 0; e < EPT; ++e) {
    const uint32_t q = (cw >> (2 * e)) & 3u;
    const float lo = (q & 1u) ? c.y : c.x;
    const float hi = (q & 1u) ? c.w : c.z;
    v[e] = (q & 2u) ? hi : lo;
  }
  const int64_t i0 = 16 * (int64_t)w + EPT * part;
  const int64_t at = j * p.ld + i0;
  if (p.vec && i0 + EPT <= p.n) {
    if constexpr (EPT == 4) {
      *reinterpret_cast<float4*>(static_cast<float*>(p.out) + at) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
      uint32_t h[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (p.dtype == KD_F16) {
          const __half2 t2 = __floats2half2_rn(v[2 * k], v[2 * k + 1]);
          h[k] = *reinterpret_cast<const uint32_t*>(&t2);
        } else {
          const __nv_bfloat162 t2 = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
          h[k] = *reinterpret_cast<const uint32_t*>(&t2);
        }
      }
      *reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.out) + at) = make_uint4(h[0], h[1], h[2], h[3]);
    }
  } else {
#pragma unroll
    for (int e = 0; e < EPT; ++e)
      if (i0 + e < p.n) put(p.out, p.dtype, at + e, v[e]);
  }
}

// Row layout over all planes of a launch: one warp per vector (the vectors of all
// planes numbered one after another).  The vector's output is cut into chunks of
// EPT = 16 / TPW entries (TPW chunks per code word); consecutive lanes write
// consecutive chunks, so every store instruction of the warp is contiguous.  A lane
// loads the code words of U chunks before its first store.
template <int TPW, int U>
__global__ void __launch_bounds__(256) dequant_rows_batch_kernel(const __grid_constant__ DeqBatch bt) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t rows = bt.first[bt.count];
  for (int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += nwarps) {
    const int i = plane_of(bt, r);
    const DeqParams& p = bt.p[i];
    const int64_t j = r - bt.first[i];
    const float4 c = __ldg(reinterpret_cast<const float4*>(p.centres) + j);
    const uint32_t* cj = p.codes + j * p.words;
    const int chunks = (int)p.words * TPW;
    for (int c0 = lane; c0 < chunks; c0 += 32 * U) {
      uint32_t cw[U];
#pragma unroll
      for (int k = 0; k < U; ++k) cw[k] = (c0 + 32 * k < chunks) ? __ldg(cj + (c0 + 32 * k) / TPW) : 0u;
#pragma unroll
      for (int k = 0; k < U; ++k) {
        const int ch = c0 + 32 * k;
        if (ch < chunks) dequant_chunk<TPW>(p, j, ch / TPW, ch % TPW, cw[k], c);
      }
    }
  }
}

__global__ void __launch_bounds__(256) dequant_cols_batch_kernel(const __grid_constant__ DeqBatch bt) {
  for (int64_t b = blockIdx.x; b < bt.first[bt.count]; b += gridDim.x) {
    const int i = plane_of(bt, b);
    dequant_col_step(bt.p[i], b - bt.first[i]);
  }
}

}  // namespace
}  // namespace kd

namespace kd {
namespace {

// Validated parameters of one plane (KD_OK) or the argument error.
kd_status deq_params(const uint32_t* codes, const float* centres, int64_t n, int64_t m, kd_dtype out_dtype,
                     kd_layout layout, void* out, int64_t ld, DeqParams* p) {
  if (n <= 0 || m < 0 || (out_dtype != KD_F32 && out_dtype != KD_F16 && out_dtype != KD_BF16) ||
      (layout != KD_VEC_ROWS && layout != KD_VEC_COLUMNS))
    return KD_ERR_INVALID_ARG;
  if (layout == KD_VEC_ROWS ? ld < n : ld < m) return KD_ERR_INVALID_ARG;
  if (m > 0 && (!codes || !centres || !out)) return KD_ERR_INVALID_ARG;
  if (m > 0 && reinterpret_cast<uintptr_t>(centres) % 16 != 0) return KD_ERR_INVALID_ARG;
  p->codes = codes;
  p->centres = centres;
  p->out = out;
  p->n = n;
  p->m = m;
  p->ld = ld;
  p->words = (n + 15) / 16;
  p->dtype = (int)out_dtype;
  p->layout = (int)layout;
  const int esz = out_dtype == KD_F32 ? 4 : 2;
  p->vec = (reinterpret_cast<uintptr_t>(out) % 16 == 0) && ((ld * esz) % 16 == 0) && (layout == KD_VEC_ROWS);
  return KD_OK;
}

kd_status grid_cap(int64_t want, int* grid) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KD_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return KD_ERR_CUDA;
  const int64_t cap = (int64_t)sms * 8;
  *grid = (int)(want < cap ? want : cap);
  return KD_OK;
}

}  // namespace
}  // namespace kd

namespace kd {
namespace {

constexpr int kDeqU = 4;  // chunks whose code words a lane of the row kernel loads ahead

// Work units of plane p: vectors for the row layout (one warp each), column steps for
// the column layout (one CTA each).
int64_t plane_units(const DeqParams& p) { return p.layout == KD_VEC_ROWS ? p.m : col_steps(p); }

kd_status launch_batch(const DeqBatch& bt, cudaStream_t s) {
  const int64_t units = bt.first[bt.count];
  if (units == 0) return KD_OK;
  const DeqParams& p0 = bt.p[0];
  int grid = 0;
  if (p0.layout == KD_VEC_ROWS) {
    if (grid_cap((units + 7) / 8, &grid) != KD_OK) return KD_ERR_CUDA;  // 8 warps (vectors) per CTA
    if (p0.dtype == KD_F32) {
      dequant_rows_batch_kernel<4, kDeqU><<<grid, 256, 0, s>>>(bt);
    } else {
      dequant_rows_batch_kernel<2, kDeqU><<<grid, 256, 0, s>>>(bt);
    }
  } else {
    if (grid_cap(units, &grid) != KD_OK) return KD_ERR_CUDA;
    dequant_cols_batch_kernel<<<grid, 256, 0, s>>>(bt);
  }
  return cudaGetLastError() == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_dequantise(const uint32_t* codes, const float* centres, int64_t n, int64_t m,
                                   kd_dtype out_dtype, kd_layout layout, void* out, int64_t ld, void* stream) {
  kd::DeqBatch bt;
  const kd_status st = kd::deq_params(codes, centres, n, m, out_dtype, layout, out, ld, &bt.p[0]);
  if (st != KD_OK) return st;
  bt.count = 1;
  bt.first[0] = 0;
  bt.first[1] = kd::plane_units(bt.p[0]);
  return kd::launch_batch(bt, static_cast<cudaStream_t>(stream));
}

extern "C" kd_status kd_dequantise_batch(const kd_plane* planes, int count, int64_t n, kd_dtype out_dtype,
                                         kd_layout layout, void* stream) {
  if (count < 1 || count > KD_MAX_BATCH || !planes) return KD_ERR_INVALID_ARG;
  kd::DeqBatch bt;
  bt.count = count;
  bt.first[0] = 0;
  for (int i = 0; i < count; ++i) {
    const kd_plane& q = planes[i];
    const kd_status st = kd::deq_params(q.codes, q.centres, n, q.m, out_dtype, layout, q.out, q.ld, &bt.p[i]);
    if (st != KD_OK) return st;
    bt.first[i + 1] = bt.first[i] + kd::plane_units(bt.p[i]);
  }
  return kd::launch_batch(bt, static_cast<cudaStream_t>(stream));
}
