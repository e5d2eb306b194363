// The folded 2-bit layer product of App. C, straight from the code planes:
//
//     Y = X W_hat^T,   W_hat = U_q + P V_q   (vector j of W_hat = output channel j)
//       = X U_q^T + (X P) V_q^T               (P symmetric)
//     y[r][j] = sum_i cu_j[code_u(j, i)] x[r][i] + sum_i cv_j[code_v(j, i)] xp[r][i]
//
// with xp = X P from kd_apply_p.  Neither U_q nor V_q is expanded: every weight costs
// its 2-bit code in each plane (0.5 byte per weight in all), read once from HBM.
//
// Mapping.  One launch serves up to KD_MAX_BATCH matrices (a layer): persistent CTAs
// of eight warps walk the work items (matrix, tile of RT = 16 / B output channels).
// Per item each warp takes slices of 32 consecutive code words (512 inputs): it loads
// its lane's 16 inputs of x and xp (L2-resident, shared by every item of the matrix)
// into registers, then the code words of all RT channels of the tile (one coalesced
// word per channel, plane and lane, all in flight together).  Two codes at a time (4
// bits) index a per-channel table of the 16 centre pairs (c[q0], c[q1]) in shared
// memory: one 64-bit shared load and one packed FP32x2 FMA per two weights, plane
// and batch row.  The lanes' and warps' partial sums are added in a fixed order
// (deterministic results).
#include <cuda_runtime.h>

#include "kashin.h"

namespace kd {
namespace {

constexpr int kFoldWarps = 8;
constexpr int kFoldThreads = 32 * kFoldWarps;

struct FoldMat {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  const float* x;
  const float* xp;
  float* y;
  int64_t n, m, words, ldx, ldy;
  int64_t tile0;  // first work item of this matrix
  int vec;        // x and xp 16-byte aligned with ldx a multiple of 4: 128-bit input loads
};

struct FoldParams {
  int count;
  int rows;        // batch rows of this launch (<= B)
  int64_t items;   // work items of all matrices
  FoldMat mat[KD_MAX_BATCH];
};

// RT x B = 16 partial sums per lane
template <int B>
struct FoldTile {
  static constexpr int RT = 16 / B;
};

template <int B>
__global__ void __launch_bounds__(kFoldThreads, 2) fold_kernel(const __grid_constant__ FoldParams p) {
  constexpr int RT = FoldTile<B>::RT;
  constexpr int K = RT * B;  // partial sums per lane
  static_assert(K == 16, "the reduction scatters 16 values per lane");
  __shared__ float2 tab[2 * RT * 16];
  __shared__ float red[kFoldWarps * 16];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;

  int mi = 0;
  for (int64_t item = blockIdx.x; item < p.items; item += gridDim.x) {
    while (mi + 1 < p.count && item >= p.mat[mi + 1].tile0) ++mi;
    const FoldMat& a = p.mat[mi];
    const int64_t j0 = (item - a.tile0) * RT;
    __syncthreads();  // the previous item's readers of the tables are done
    // pair tables: entry q0 | q1 << 2 = (c[q0], c[q1]) for the elements 2k, 2k + 1 of a word
    for (int t = threadIdx.x; t < 2 * RT * 16; t += kFoldThreads) {
      const int plane = t / (RT * 16);
      const int r = (t / 16) % RT;
      const int e = t % 16;
      float2 v = make_float2(0.f, 0.f);
      if (j0 + r < a.m) {
        const float4 c = __ldg(reinterpret_cast<const float4*>(plane ? a.centres_v : a.centres_u) + j0 + r);
        const float cc[4] = {c.x, c.y, c.z, c.w};
        v = make_float2(cc[e & 3], cc[e >> 2]);
      }
      tab[t] = v;
    }
    __syncthreads();

    float2 acc[RT][B];
#pragma unroll
    for (int r = 0; r < RT; ++r)
#pragma unroll
      for (int b = 0; b < B; ++b) acc[r][b] = make_float2(0.f, 0.f);

    const int64_t nslices = (a.words + 31) / 32;
    for (int64_t s = warp; s < nslices; s += kFoldWarps) {
      const int64_t wi = s * 32 + lane;
      const bool valid = wi < a.words;
      uint32_t cu[RT], cv[RT];
#pragma unroll
      for (int r = 0; r < RT; ++r) {
        const bool ok = valid && j0 + r < a.m;
        cu[r] = ok ? __ldg(a.codes_u + (j0 + r) * a.words + wi) : 0u;
        cv[r] = ok ? __ldg(a.codes_v + (j0 + r) * a.words + wi) : 0u;
      }
      // this lane's 16 inputs of x and xp per batch row (zero past n and past the rows):
      // four 128-bit loads each when the whole word lies inside aligned rows
      float2 xv[B][8], pv[B][8];
      {
        const bool vec = a.vec && 16 * wi + 16 <= a.n;
#pragma unroll
        for (int b = 0; b < B; ++b) {
          const bool live = valid && b < p.rows;
          const int64_t o0 = (int64_t)b * a.ldx + 16 * wi;
          if (vec && live) {
#pragma unroll
            for (int k = 0; k < 8; k += 2) {
              const float4 u = __ldg(reinterpret_cast<const float4*>(a.x + o0 + 2 * k));
              const float4 w = __ldg(reinterpret_cast<const float4*>(a.xp + o0 + 2 * k));
              xv[b][k] = make_float2(u.x, u.y);
              xv[b][k + 1] = make_float2(u.z, u.w);
              pv[b][k] = make_float2(w.x, w.y);
              pv[b][k + 1] = make_float2(w.z, w.w);
            }
          } else {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const int64_t i = 16 * wi + 2 * k;
              const bool i0 = live && i < a.n, i1 = live && i + 1 < a.n;
              xv[b][k] = make_float2(i0 ? __ldg(a.x + o0 + 2 * k) : 0.f, i1 ? __ldg(a.x + o0 + 2 * k + 1) : 0.f);
              pv[b][k] = make_float2(i0 ? __ldg(a.xp + o0 + 2 * k) : 0.f, i1 ? __ldg(a.xp + o0 + 2 * k + 1) : 0.f);
            }
          }
        }
      }
#pragma unroll
      for (int r = 0; r < RT; ++r) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float2 tu = tab[r * 16 + ((cu[r] >> (4 * k)) & 15u)];
          const float2 tv = tab[(RT + r) * 16 + ((cv[r] >> (4 * k)) & 15u)];
#pragma unroll
          for (int b = 0; b < B; ++b) {
            acc[r][b] = __ffma2_rn(tu, xv[b][k], acc[r][b]);
            acc[r][b] = __ffma2_rn(tv, pv[b][k], acc[r][b]);
          }
        }
      }
    }

    // lane sums, then a butterfly reduce-scatter: lane l ends with its warp's total of
    // value l % 16 (value index r * B + b)
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
    v[0] = __fadd_rn(v[0], __shfl_xor_sync(0xffffffffu, v[0], 16));
    if (lane < K) red[warp * 16 + lane] = v[0];
    __syncthreads();
    if (threadIdx.x < K) {
      float t = red[threadIdx.x];
#pragma unroll
      for (int w = 1; w < kFoldWarps; ++w) t = __fadd_rn(t, red[w * 16 + threadIdx.x]);
      const int r = threadIdx.x / B, b = threadIdx.x % B;
      if (j0 + r < a.m && b < p.rows) a.y[(int64_t)b * a.ldy + j0 + r] = t;
    }
  }
}

template <int B>
cudaError_t launch_fold(const FoldParams& p, cudaStream_t s) {
  int dev = 0, sms = 0, per = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, fold_kernel<B>, kFoldThreads, 0)) != cudaSuccess)
    return e;
  if (per < 1) return cudaErrorInvalidConfiguration;
  const int64_t grid = p.items < (int64_t)per * sms ? p.items : (int64_t)per * sms;
  fold_kernel<B><<<(unsigned)grid, kFoldThreads, 0, s>>>(p);
  return cudaGetLastError();
}

bool aligned(const void* ptr, size_t a) { return reinterpret_cast<uintptr_t>(ptr) % a == 0; }

}  // namespace
}  // namespace kd

namespace kd {
namespace {

kd_status check_fold(const kd_fold_mat& a, int64_t batch) {
  if (a.n <= 0 || a.m < 0 || a.ldx < a.n || a.ldy < a.m) return KD_ERR_INVALID_ARG;
  if (a.m == 0 || batch == 0) return KD_OK;
  if (!a.codes_u || !a.codes_v || !a.centres_u || !a.centres_v || !a.x || !a.xp || !a.y) return KD_ERR_INVALID_ARG;
  if (!aligned(a.centres_u, 16) || !aligned(a.centres_v, 16) || !aligned(a.codes_u, 4) ||
      !aligned(a.codes_v, 4) || !aligned(a.x, 4) || !aligned(a.xp, 4) || !aligned(a.y, 4))
    return KD_ERR_INVALID_ARG;
  return KD_OK;
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_matmul_2bit_batch(const kd_fold_mat* mats, int count, int64_t batch, void* stream) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || batch < 0) return KD_ERR_INVALID_ARG;
  for (int i = 0; i < count; ++i) {
    const kd_status st = kd::check_fold(mats[i], batch);
    if (st != KD_OK) return st;
  }
  if (batch == 0) return KD_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // batch rows two (or one) at a time: each launch reads the code planes once
  for (int64_t b0 = 0; b0 < batch;) {
    const int rows = batch - b0 >= 2 ? 2 : 1;
    const int rt = rows == 2 ? kd::FoldTile<2>::RT : kd::FoldTile<1>::RT;
    kd::FoldParams p;
    p.count = count;
    p.rows = rows;
    int64_t items = 0;
    for (int i = 0; i < count; ++i) {
      const kd_fold_mat& a = mats[i];
      kd::FoldMat& f = p.mat[i];
      f.codes_u = a.codes_u;
      f.codes_v = a.codes_v;
      f.centres_u = a.centres_u;
      f.centres_v = a.centres_v;
      f.x = a.x + b0 * a.ldx;
      f.xp = a.xp + b0 * a.ldx;
      f.y = a.y + b0 * a.ldy;
      f.n = a.n;
      f.m = a.m;
      f.words = (a.n + 15) / 16;
      f.ldx = a.ldx;
      f.ldy = a.ldy;
      f.tile0 = items;
      f.vec = kd::aligned(f.x, 16) && kd::aligned(f.xp, 16) && a.ldx % 4 == 0;
      items += (a.m + rt - 1) / rt;
    }
    p.items = items;
    if (items > 0) {
      const cudaError_t e = rows == 2 ? kd::launch_fold<2>(p, s) : kd::launch_fold<1>(p, s);
      if (e != cudaSuccess) return KD_ERR_CUDA;
    }
    b0 += rows;
  }
  return KD_OK;
}

extern "C" kd_status kd_matmul_2bit(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                                    const float* centres_v, int64_t n, int64_t m, const float* x, const float* xp,
                                    int64_t batch, int64_t ldx, float* y, int64_t ldy, void* stream) {
  const kd_fold_mat a{codes_u, codes_v, centres_u, centres_v, x, xp, y, n, m, ldx, ldy};
  return kd_matmul_2bit_batch(&a, 1, batch, stream);
}
