// The folded 2-bit layer product of App. C, straight from the code planes:
//
//     Y = X W_hat^T,   W_hat = U_q + P V_q   (vector j of W_hat = output channel j)
//       = X U_q^T + (X P) V_q^T               (P symmetric)
//     y[r][j] = sum_i cu_j[code_u(j, i)] x[r][i] + sum_i cv_j[code_v(j, i)] xp[r][i]
//
// with xp = X P from kd_apply_p.  Neither U_q nor V_q is expanded: every weight costs
// its 2-bit code in each plane (0.5 byte per weight in all), read once from HBM.
//
// Mapping.  A CTA owns RT consecutive output channels; each of its warps owns slices
// of 32 consecutive code words (512 inputs) and holds its lane's 16 inputs of x and xp
// in registers, then walks the CTA's channels: per channel one coalesced code word
// per plane and lane.  Two codes at a time (4 bits) index a per-channel table of the
// 16 centre pairs (c[q0], c[q1]) in shared memory: one 64-bit shared load and one
// packed FP32x2 FMA per two weights, plane and batch row.  The lanes' and warps'
// partial sums are added in a fixed order (deterministic results).
#include <cuda_runtime.h>

#include "kashin.h"

namespace kd {
namespace {

constexpr int kFoldWarps = 8;
constexpr int kFoldThreads = 32 * kFoldWarps;

struct FoldParams {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  const float* x;
  const float* xp;
  float* y;
  int64_t n, m, words, ldx, ldy;
  int rows;  // batch rows of this launch (<= B)
};

// output channels per CTA: RT x B = 8 partial sums per lane, so that two CTAs of
// 256 threads fit on an SM for one or two batch rows (enough loads in flight to keep
// HBM busy); four rows hold 128 inputs per lane and run one CTA per SM
template <int B>
struct FoldTile {
  static constexpr int RT = 8 / B;
};

template <int B>
__global__ void __launch_bounds__(kFoldThreads, B == 4 ? 1 : 2) fold_kernel(const FoldParams p) {
  constexpr int RT = FoldTile<B>::RT;
  constexpr int K = RT * B;  // partial sums per lane
  static_assert(K >= 1 && K <= 16 && (K & (K - 1)) == 0, "the reduction scatters a power of two <= 16 values");
  __shared__ float2 tab[2][RT][16];
  __shared__ float red[kFoldWarps][K];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int64_t j0 = (int64_t)blockIdx.x * RT;

  // pair tables: entry q0 | q1 << 2 = (c[q0], c[q1]) for the elements 2k, 2k + 1 of a word
  for (int t = threadIdx.x; t < 2 * RT * 16; t += kFoldThreads) {
    const int plane = t / (RT * 16);
    const int r = (t / 16) % RT;
    const int e = t % 16;
    float2 v = make_float2(0.f, 0.f);
    if (j0 + r < p.m) {
      const float4 c = __ldg(reinterpret_cast<const float4*>(plane ? p.centres_v : p.centres_u) + j0 + r);
      const float cc[4] = {c.x, c.y, c.z, c.w};
      v = make_float2(cc[e & 3], cc[e >> 2]);
    }
    tab[plane][r][e] = v;
  }
  __syncthreads();

  float2 acc[RT][B];
#pragma unroll
  for (int r = 0; r < RT; ++r)
#pragma unroll
    for (int b = 0; b < B; ++b) acc[r][b] = make_float2(0.f, 0.f);

  const int64_t nslices = (p.words + 31) / 32;
  for (int64_t s = warp; s < nslices; s += kFoldWarps) {
    const int64_t wi = s * 32 + lane;
    const bool valid = wi < p.words;
    // this lane's 16 inputs of x and xp for every batch row (zero past n)
    float2 xv[B][8], pv[B][8];
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const bool live = b < p.rows;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t i = 16 * wi + 2 * k;
        const int64_t o = (int64_t)b * p.ldx + i;
        const bool i0 = live && valid && i < p.n, i1 = live && valid && i + 1 < p.n;
        xv[b][k] = make_float2(i0 ? __ldg(p.x + o) : 0.f, i1 ? __ldg(p.x + o + 1) : 0.f);
        pv[b][k] = make_float2(i0 ? __ldg(p.xp + o) : 0.f, i1 ? __ldg(p.xp + o + 1) : 0.f);
      }
    }
    uint32_t cu[RT], cv[RT];
#pragma unroll
    for (int r = 0; r < RT; ++r) {
      const bool ok = valid && j0 + r < p.m;
      cu[r] = ok ? __ldg(p.codes_u + (j0 + r) * p.words + wi) : 0u;
      cv[r] = ok ? __ldg(p.codes_v + (j0 + r) * p.words + wi) : 0u;
    }
#pragma unroll
    for (int r = 0; r < RT; ++r) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float2 tu = tab[0][r][(cu[r] >> (4 * k)) & 15u];
        const float2 tv = tab[1][r][(cv[r] >> (4 * k)) & 15u];
#pragma unroll
        for (int b = 0; b < B; ++b) {
          acc[r][b] = __ffma2_rn(tu, xv[b][k], acc[r][b]);
          acc[r][b] = __ffma2_rn(tv, pv[b][k], acc[r][b]);
        }
      }
    }
  }

  // lane sums, then a butterfly reduce-scatter: lane l ends with its warp's total of
  // value l % K (value index r * B + b)
  float v[K];
#pragma unroll
  for (int r = 0; r < RT; ++r)
#pragma unroll
    for (int b = 0; b < B; ++b) v[r * B + b] = __fadd_rn(acc[r][b].x, acc[r][b].y);
#pragma unroll
  for (int k = K / 2; k >= 1; k >>= 1) {
#pragma unroll
    for (int i = 0; i < k; ++i) {
      const bool hi = (lane & k) != 0;
      const float send = hi ? v[i] : v[i + k];
      const float keep = hi ? v[i + k] : v[i];
      v[i] = __fadd_rn(keep, __shfl_xor_sync(0xffffffffu, send, k));
    }
  }
#pragma unroll
  for (int off = K; off < 32; off <<= 1) v[0] = __fadd_rn(v[0], __shfl_xor_sync(0xffffffffu, v[0], off));
  if (lane < K) red[warp][lane] = v[0];
  __syncthreads();
  if (threadIdx.x < K) {
    float t = red[0][threadIdx.x];
#pragma unroll
    for (int w = 1; w < kFoldWarps; ++w) t = __fadd_rn(t, red[w][threadIdx.x]);
    const int r = threadIdx.x / B, b = threadIdx.x % B;
    if (j0 + r < p.m && b < p.rows) p.y[(int64_t)b * p.ldy + j0 + r] = t;
  }
}

template <int B>
cudaError_t launch_fold(FoldParams p, cudaStream_t s) {
  constexpr int RT = FoldTile<B>::RT;
  const int64_t grid = (p.m + RT - 1) / RT;
  fold_kernel<B><<<(unsigned)grid, kFoldThreads, 0, s>>>(p);
  return cudaGetLastError();
}

bool aligned(const void* ptr, size_t a) { return reinterpret_cast<uintptr_t>(ptr) % a == 0; }

}  // namespace
}  // namespace kd

extern "C" kd_status kd_matmul_2bit(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                                    const float* centres_v, int64_t n, int64_t m, const float* x, const float* xp,
                                    int64_t batch, int64_t ldx, float* y, int64_t ldy, void* stream) {
  if (n <= 0 || m < 0 || batch < 0 || ldx < n || ldy < m) return KD_ERR_INVALID_ARG;
  if (m == 0 || batch == 0) return KD_OK;
  if (!codes_u || !codes_v || !centres_u || !centres_v || !x || !xp || !y) return KD_ERR_INVALID_ARG;
  if (!kd::aligned(centres_u, 16) || !kd::aligned(centres_v, 16) || !kd::aligned(codes_u, 4) ||
      !kd::aligned(codes_v, 4) || !kd::aligned(x, 4) || !kd::aligned(xp, 4) || !kd::aligned(y, 4))
    return KD_ERR_INVALID_ARG;
  if ((m + 1) / 2 > 0x7fffffffll) return KD_ERR_INVALID_ARG;  // grid size
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kd::FoldParams p{codes_u, codes_v, centres_u, centres_v, x, xp, y, n, m, (n + 15) / 16, ldx, ldy, 0};
  // batch rows four, two or one at a time (each launch reads the code planes once)
  for (int64_t b0 = 0; b0 < batch;) {
    const int64_t left = batch - b0;
    const int rows = left >= 4 ? 4 : (left >= 2 ? 2 : 1);
    p.x = x + b0 * ldx;
    p.xp = xp + b0 * ldx;
    p.y = y + b0 * ldy;
    p.rows = rows;
    const cudaError_t e = rows == 4 ? kd::launch_fold<4>(p, s) : rows == 2 ? kd::launch_fold<2>(p, s)
                                                                            : kd::launch_fold<1>(p, s);
    if (e != cudaSuccess) return KD_ERR_CUDA;
    b0 += rows;
  }
  return KD_OK;
}
