// Dequantisation of one 2-bit factor plane (App. C, inference): the dense factor
// matrix U_q (or V_q) with entry i of vector j equal to centres[j][code_j(i)].
//
// App. C folds the layer product as  X W = X U_q + (X P) V_q = [X | XP] [U_q; V_q]:
// on hardware without 2-bit matrix units the factors are expanded once at load
// time and the product runs as an ordinary GEMM; kd_apply_p gives XP and
// kd_reconstruct gives W_hat = U_q + P V_q directly.
//
// Bound by HBM: per entry 1/4 byte of codes is read and 2 or 4 bytes are written.
// Row layout: one vector per CTA step, two (16-bit output) or four (fp32) threads
// per code word, each with one 16-byte centre load and one 16-byte store.  Column
// layout: consecutive threads take consecutive vectors of the same word, so every
// store instruction of a warp writes consecutive addresses.
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

// TPW threads per code word, each writing 16 contiguous bytes (4 fp32 or 8 16-bit
// entries): consecutive lanes write consecutive 16-byte pieces
template <int TPW>
__global__ void __launch_bounds__(256) dequant_rows_kernel(DeqParams p) {
  constexpr int EPT = 16 / TPW;
  const int per_row = (int)p.words * TPW;
  for (int64_t j = blockIdx.x; j < p.m; j += gridDim.x)
  for (int g = threadIdx.x; g < per_row; g += blockDim.x) {
    const int w = g / TPW;
    const int part = g - w * TPW;
    const int64_t word = j * p.words + w;
    const uint32_t code = __ldg(p.codes + word) >> (2 * EPT * part);
    const float4 c = __ldg(reinterpret_cast<const float4*>(p.centres) + j);
    float v[EPT];
#pragma unroll
    for (int e = 0; e < EPT; ++e) {
      const uint32_t q = (code >> (2 * e)) & 3u;
      const float lo = (q & 1u) ? c.y : c.x;
      const float hi = (q & 1u) ? c.w : c.z;
      v[e] = (q & 2u) ? hi : lo;
    }
    const int64_t i0 = 16 * w + EPT * part;
    const int64_t base = j * p.ld + i0;
    if (p.vec && i0 + EPT <= p.n) {
      if constexpr (EPT == 4) {
        *reinterpret_cast<float4*>(static_cast<float*>(p.out) + base) = make_float4(v[0], v[1], v[2], v[3]);
      } else {
        uint32_t h[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (p.dtype == KD_F16) {
            const __half2 t = __floats2half2_rn(v[2 * k], v[2 * k + 1]);
            h[k] = *reinterpret_cast<const uint32_t*>(&t);
          } else {
            const __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
            h[k] = *reinterpret_cast<const uint32_t*>(&t);
          }
        }
        *reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.out) + base) = make_uint4(h[0], h[1], h[2], h[3]);
      }
    } else {
#pragma unroll
      for (int e = 0; e < EPT; ++e)
        if (i0 + e < p.n) put(p.out, p.dtype, base + e, v[e]);
    }
  }
}

__global__ void __launch_bounds__(256) dequant_cols_kernel(DeqParams p) {
  // CTA step b covers code word w = b % words of vectors 256 (b / words) + threadIdx.x
  const int64_t jblocks = (p.m + 255) / 256;
  for (int64_t b = blockIdx.x; b < p.words * jblocks; b += gridDim.x) {
    const int64_t jb = b / p.words;
    const int64_t w = b - jb * p.words;
    const int64_t j = jb * 256 + threadIdx.x;
    if (j >= p.m) continue;
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
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_dequantise(const uint32_t* codes, const float* centres, int64_t n, int64_t m,
                                   kd_dtype out_dtype, kd_layout layout, void* out, int64_t ld, void* stream) {
  if (n <= 0 || m < 0 || (out_dtype != KD_F32 && out_dtype != KD_F16 && out_dtype != KD_BF16) ||
      (layout != KD_VEC_ROWS && layout != KD_VEC_COLUMNS))
    return KD_ERR_INVALID_ARG;
  if (layout == KD_VEC_ROWS ? ld < n : ld < m) return KD_ERR_INVALID_ARG;
  if (m == 0) return KD_OK;
  if (!codes || !centres || !out) return KD_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(centres) % 16 != 0) return KD_ERR_INVALID_ARG;
  kd::DeqParams p;
  p.codes = codes;
  p.centres = centres;
  p.out = out;
  p.n = n;
  p.m = m;
  p.ld = ld;
  p.words = (n + 15) / 16;
  p.dtype = (int)out_dtype;
  p.layout = (int)layout;
  const int esz = out_dtype == KD_F32 ? 4 : 2;
  p.vec = (reinterpret_cast<uintptr_t>(out) % 16 == 0) && ((ld * esz) % 16 == 0) && (layout == KD_VEC_ROWS);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KD_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return KD_ERR_CUDA;
  const int tpw = out_dtype == KD_F32 ? 4 : 2;
  const int64_t want = layout == KD_VEC_ROWS ? m : p.words * ((m + 255) / 256);  // CTA steps
  const int64_t cap = (int64_t)sms * 8;
  const int grid = (int)(want < cap ? want : cap);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (layout == KD_VEC_ROWS) {
    if (tpw == 4) {
      kd::dequant_rows_kernel<4><<<grid, 256, 0, s>>>(p);
    } else {
      kd::dequant_rows_kernel<2><<<grid, 256, 0, s>>>(p);
    }
  } else {
    kd::dequant_cols_kernel<<<grid, 256, 0, s>>>(p);
  }
  return cudaGetLastError() == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}
