// The folded 2-bit layer product of App. C for 16-bit activations (fp16 or bf16), on the
// tensor cores:
//
//     y[r][j] = sum_i h(cu_j[code_u(j, i)]) x[r][i] + sum_i h(cv_j[code_v(j, i)]) xp[r][i]
//
// with x, xp in the 16-bit type (xp = X P from kd_apply_p, rounded by the caller), h()
// the rounding of a centre to that type, fp32 accumulation.  Neither plane is expanded
// in memory: each code becomes its 16-bit centre in registers and feeds an mma.sync B
// fragment directly.
//
// Mapping.  mma.m16n8k16 with M = the batch rows (up to 16 per launch), N = 8 output
// channels, K = 16 inputs.  A work item is a tile of 32 channels (four n-tiles) of one
// matrix and one CTA; its four warps split the inputs into groups of 64 (four k-steps)
// round-robin, each loading the next group's code words and inputs while it computes
// the current one, then add their partial tiles in a fixed order (deterministic
// results).  Items are numbered longest vectors first, so the hardware starts the long
// ones first.  Launches of at most 8 batch rows skip the rows g + 8 of the A fragments
// (fewer registers, more warps per SM).
//
// K order inside a group of 64 inputs.  The product is a sum over inputs, so A and B
// may enumerate them in any common order.  In k-step j the lanes with t = lane % 4
// take inputs 16 t + 4 j + {0, 1} for k-slots 2t, 2t+1 and 16 t + 4 j + {2, 3} for
// k-slots 2t+8, 2t+9.  A lane's A fragments for the whole group are then its 16
// consecutive inputs of rows g and g + 8 (g = lane / 4: two 16-byte loads per row), and
// its B fragments are code word t of the group (inputs 16 t .. 16 t + 15) of its
// channel: byte j of that word holds the four codes of k-step j.
//
// Decoding.  The four 16-bit centres of a channel are kept as two words, L (their low
// bytes) and H (their high bytes).  For two codes q0, q1 one byte permute with the
// selector nibbles (q0, q0 + 4, q1, q1 + 4) yields the pair (c[q0], c[q1]); the
// selectors of two k-steps are formed together from one shifted code word.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "kashin.h"

namespace kd {
namespace {

constexpr int kF16Warps = 4;
constexpr int kF16Threads = 32 * kF16Warps;
constexpr int kF16Rows = 16;  // batch rows per launch (the mma's M)
constexpr int kF16Tile = 32;  // output channels per work item (four n-tiles)
constexpr int kRedStride = kF16Tile + 1;

struct Fold16Mat {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  const unsigned short* x;
  const unsigned short* xp;
  float* y;
  int64_t n, m, words, ldx, ldy;
  int64_t item0;  // first work item of this matrix
  int vec;        // x and xp 16-byte aligned with ldx a multiple of 8: 128-bit input loads
};

struct Fold16Params {
  int count;
  int rows;  // batch rows of this launch (<= 16)
  int64_t items;
  Fold16Mat mat[KD_MAX_BATCH];
};

// D += A B for one m16n8k16 tile; BF: the 16-bit operands are bf16 instead of fp16
template <bool BF>
__device__ __forceinline__ void mma_16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                       uint32_t b0, uint32_t b1) {
  if constexpr (BF) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  } else {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
}

// a centre rounded (nearest, ties to even) to the activations' 16-bit type, as bits
template <bool BF>
__device__ __forceinline__ uint32_t bits16(float c) {
  if constexpr (BF) return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(c));
  else return (uint32_t)__half_as_ushort(__float2half_rn(c));
}

// Byte selectors for the code nibbles at bits 0..3 (low half) and 16..19 (high half) of
// t: nibble v = q0 | q1 << 2 gives the selector nibbles (q0, q0 + 4, q1, q1 + 4).
__device__ __forceinline__ uint32_t selectors(uint32_t t) {
  // q0 to bits 0-1, q1 to bits 8-9 (and 16-17, 24-25): one mask, one shift, one multiplex
  const uint32_t u = t & 0x000F000Fu;
  const uint32_t x = (u & 0x00C300C3u) | ((u << 6) & ~0x00C300C3u);
  return x * 0x11u + 0x40404040u;
}

// The 16-bit centres of one channel as (low bytes, high bytes), zero past m.
template <bool BF>
__device__ __forceinline__ uint2 centre_bytes(const float* centres, int64_t j, bool ok) {
  if (!ok) return make_uint2(0u, 0u);
  const float4 c = __ldg(reinterpret_cast<const float4*>(centres) + j);
  const uint32_t p01 = bits16<BF>(c.x) | (bits16<BF>(c.y) << 16);
  const uint32_t p23 = bits16<BF>(c.z) | (bits16<BF>(c.w) << 16);
  return make_uint2(__byte_perm(p01, p23, 0x6420u), __byte_perm(p01, p23, 0x7531u));
}

// A lane's 16 fp16 inputs of one row at i0 .. i0 + 15 as 8 pairs, zero past n or for a
// row outside the batch.
__device__ __forceinline__ void load_row16(uint32_t (&r)[8], const unsigned short* row, int64_t i0, int64_t n,
                                           bool live, bool vec) {
  if (!live) {
#pragma unroll
    for (int k = 0; k < 8; ++k) r[k] = 0u;
  } else if (vec && i0 + 16 <= n) {
    const uint4 a = __ldg(reinterpret_cast<const uint4*>(row + i0));
    const uint4 b = __ldg(reinterpret_cast<const uint4*>(row + i0 + 8));
    r[0] = a.x; r[1] = a.y; r[2] = a.z; r[3] = a.w;
    r[4] = b.x; r[5] = b.y; r[6] = b.z; r[7] = b.w;
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int64_t i = i0 + 2 * k;
      const uint32_t lo = i < n ? (uint32_t)__ldg(row + i) : 0u;
      const uint32_t hi = i + 1 < n ? (uint32_t)__ldg(row + i + 1) : 0u;
      r[k] = lo | (hi << 16);
    }
  }
}

template <bool HI, bool BF>
__global__ void __launch_bounds__(kF16Threads, HI ? 3 : 4) fold16_kernel(const __grid_constant__ Fold16Params p) {
  __shared__ float red[kF16Warps][kF16Rows][kRedStride];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;

  int mi = 0;
  for (int64_t item = blockIdx.x; item < p.items; item += gridDim.x) {
    while (mi + 1 < p.count && item >= p.mat[mi + 1].item0) ++mi;
    const Fold16Mat& a = p.mat[mi];
    const int64_t c0 = (item - a.item0) * kF16Tile;

    // this lane's channel of each n-tile: centres as byte words, code rows
    uint2 cu[4], cv[4];
    const uint32_t* ru[4];
    const uint32_t* rv[4];
    bool live[4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
      const int64_t j = c0 + 8 * nt + g;
      live[nt] = j < a.m;
      cu[nt] = centre_bytes<BF>(a.centres_u, j, live[nt]);
      cv[nt] = centre_bytes<BF>(a.centres_v, j, live[nt]);
      ru[nt] = a.codes_u + (live[nt] ? j : 0) * a.words;
      rv[nt] = a.codes_v + (live[nt] ? j : 0) * a.words;
    }
    float acc[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;

    const bool lo_live = g < p.rows, hi_live = g + 8 < p.rows;
    const unsigned short* xg = a.x + (int64_t)g * a.ldx;
    const unsigned short* xh = a.x + (int64_t)(g + 8) * a.ldx;
    const unsigned short* pg = a.xp + (int64_t)g * a.ldx;
    const unsigned short* ph = a.xp + (int64_t)(g + 8) * a.ldx;
    const int64_t groups = (a.words + 3) / 4;
    // software pipeline: the next group's code words and inputs load while this one computes
    uint32_t wu[4], wv[4], ax[8], axh[8], ap[8], aph[8];
    auto fetch = [&](int64_t gi) {
      const int64_t wi = 4 * gi + t;  // this lane's code word of the group
      const int64_t i0 = 64 * gi + 16 * t;
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
        const bool ok = live[nt] && wi < a.words;
        wu[nt] = ok ? __ldg(ru[nt] + wi) : 0u;
        wv[nt] = ok ? __ldg(rv[nt] + wi) : 0u;
      }
      load_row16(ax, xg, i0, a.n, lo_live, a.vec);
      load_row16(ap, pg, i0, a.n, lo_live, a.vec);
      if constexpr (HI) {
        load_row16(axh, xh, i0, a.n, hi_live, a.vec);
        load_row16(aph, ph, i0, a.n, hi_live, a.vec);
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) axh[k] = aph[k] = 0u;
      }
    };
    if (warp < groups) fetch(warp);
    for (int64_t gi = warp; gi < groups; gi += kF16Warps) {
      uint32_t cwu[4], cwv[4], cax[8], caxh[8], cap[8], caph[8];
#pragma unroll
      for (int k = 0; k < 4; ++k) { cwu[k] = wu[k]; cwv[k] = wv[k]; }
#pragma unroll
      for (int k = 0; k < 8; ++k) { cax[k] = ax[k]; caxh[k] = axh[k]; cap[k] = ap[k]; caph[k] = aph[k]; }
      if (gi + kF16Warps < groups) fetch(gi + kF16Warps);
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
        // k-steps (0, 2) from nibbles at bits (0, 16) and (4, 20); (1, 3) from (8, 24), (12, 28)
        const uint32_t su0 = selectors(cwu[nt]), su1 = selectors(cwu[nt] >> 4);
        const uint32_t su2 = selectors(cwu[nt] >> 8), su3 = selectors(cwu[nt] >> 12);
        const uint32_t sv0 = selectors(cwv[nt]), sv1 = selectors(cwv[nt] >> 4);
        const uint32_t sv2 = selectors(cwv[nt] >> 8), sv3 = selectors(cwv[nt] >> 12);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t s0u = (j & 1) ? su2 : su0, s1u = (j & 1) ? su3 : su1;
          const uint32_t s0v = (j & 1) ? sv2 : sv0, s1v = (j & 1) ? sv3 : sv1;
          const int sh = (j & 2) ? 16 : 0;
          const uint32_t bu0 = __byte_perm(cu[nt].x, cu[nt].y, s0u >> sh);
          const uint32_t bu1 = __byte_perm(cu[nt].x, cu[nt].y, s1u >> sh);
          const uint32_t bv0 = __byte_perm(cv[nt].x, cv[nt].y, s0v >> sh);
          const uint32_t bv1 = __byte_perm(cv[nt].x, cv[nt].y, s1v >> sh);
          mma_16<BF>(acc[nt], cax[2 * j], caxh[2 * j], cax[2 * j + 1], caxh[2 * j + 1], bu0, bu1);
          mma_16<BF>(acc[nt], cap[2 * j], caph[2 * j], cap[2 * j + 1], caph[2 * j + 1], bv0, bv1);
        }
      }
    }

    // partial tiles of the four warps, added in warp order
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
      red[warp][g][8 * nt + 2 * t] = acc[nt][0];
      red[warp][g][8 * nt + 2 * t + 1] = acc[nt][1];
      red[warp][g + 8][8 * nt + 2 * t] = acc[nt][2];
      red[warp][g + 8][8 * nt + 2 * t + 1] = acc[nt][3];
    }
    __syncthreads();
    for (int o = threadIdx.x; o < kF16Rows * kF16Tile; o += kF16Threads) {
      const int r = o / kF16Tile, c = o % kF16Tile;
      if (r < p.rows && c0 + c < a.m) {
        float s = red[0][r][c];
#pragma unroll
        for (int w = 1; w < kF16Warps; ++w) s = __fadd_rn(s, red[w][r][c]);
        a.y[(int64_t)r * a.ldy + c0 + c] = s;
      }
    }
    __syncthreads();  // red is reused by the next item
  }
}

bool aligned16(const void* ptr, size_t a) { return reinterpret_cast<uintptr_t>(ptr) % a == 0; }

kd_status check_fold16(const kd_fold_mat_f16& a, int64_t batch) {
  if (a.n <= 0 || a.m < 0 || a.ldx < a.n || a.ldy < a.m) return KD_ERR_INVALID_ARG;
  if (a.m == 0 || batch == 0) return KD_OK;
  if (!a.codes_u || !a.codes_v || !a.centres_u || !a.centres_v || !a.x || !a.xp || !a.y) return KD_ERR_INVALID_ARG;
  if (!aligned16(a.centres_u, 16) || !aligned16(a.centres_v, 16) || !aligned16(a.codes_u, 4) ||
      !aligned16(a.codes_v, 4) || !aligned16(a.x, 2) || !aligned16(a.xp, 2) || !aligned16(a.y, 4))
    return KD_ERR_INVALID_ARG;
  return KD_OK;
}

}  // namespace
}  // namespace kd

namespace kd {
namespace {

kd_status fold16_run(const kd_fold_mat_f16* mats, int count, int64_t batch, void* stream, bool bf) {
  if (!mats || count < 1 || count > KD_MAX_BATCH || batch < 0) return KD_ERR_INVALID_ARG;
  for (int i = 0; i < count; ++i) {
    const kd_status st = check_fold16(mats[i], batch);
    if (st != KD_OK) return st;
  }
  int64_t work = 0;
  for (int i = 0; i < count; ++i) work += mats[i].m;
  if (batch == 0 || work == 0) return KD_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // batch rows sixteen at a time (the mma's M): each launch reads the code planes once
  for (int64_t b0 = 0; b0 < batch; b0 += kF16Rows) {
    Fold16Params p;
    p.count = count;
    p.rows = (int)(batch - b0 < kF16Rows ? batch - b0 : kF16Rows);
    // work items numbered longest vectors first, so that the long items of a layer are
    // not the last ones started
    int order[KD_MAX_BATCH];
    for (int i = 0; i < count; ++i) order[i] = i;
    for (int i = 1; i < count; ++i)
      for (int k = i; k > 0 && mats[order[k]].n > mats[order[k - 1]].n; --k) {
        const int tmp = order[k];
        order[k] = order[k - 1];
        order[k - 1] = tmp;
      }
    int64_t items = 0;
    for (int i = 0; i < count; ++i) {
      const kd_fold_mat_f16& a = mats[order[i]];
      Fold16Mat& f = p.mat[i];
      f.codes_u = a.codes_u;
      f.codes_v = a.codes_v;
      f.centres_u = a.centres_u;
      f.centres_v = a.centres_v;
      f.x = static_cast<const unsigned short*>(a.x) + b0 * a.ldx;
      f.xp = static_cast<const unsigned short*>(a.xp) + b0 * a.ldx;
      f.y = a.y + b0 * a.ldy;
      f.n = a.n;
      f.m = a.m;
      f.words = (a.n + 15) / 16;
      f.ldx = a.ldx;
      f.ldy = a.ldy;
      f.item0 = items;
      f.vec = aligned16(f.x, 16) && aligned16(f.xp, 16) && a.ldx % 8 == 0;
      items += (a.m + kF16Tile - 1) / kF16Tile;
    }
    p.items = items;
    if (items == 0) continue;
    // one CTA per work item (the grid-stride loop covers grids past 2^30 items)
    const int64_t grid = items < (int64_t)1 << 30 ? items : (int64_t)1 << 30;
    const unsigned gr = (unsigned)grid;
    if (bf) {
      if (p.rows > 8) fold16_kernel<true, true><<<gr, kF16Threads, 0, s>>>(p);
      else fold16_kernel<false, true><<<gr, kF16Threads, 0, s>>>(p);
    } else {
      if (p.rows > 8) fold16_kernel<true, false><<<gr, kF16Threads, 0, s>>>(p);
      else fold16_kernel<false, false><<<gr, kF16Threads, 0, s>>>(p);
    }
    if (cudaGetLastError() != cudaSuccess) return KD_ERR_CUDA;
  }
  return KD_OK;
}

}  // namespace
}  // namespace kd

extern "C" kd_status kd_matmul_2bit_f16_batch(const kd_fold_mat_f16* mats, int count, int64_t batch,
                                              void* stream) {
  return kd::fold16_run(mats, count, batch, stream, false);
}

extern "C" kd_status kd_matmul_2bit_bf16_batch(const kd_fold_mat_f16* mats, int count, int64_t batch,
                                               void* stream) {
  return kd::fold16_run(mats, count, batch, stream, true);
}

extern "C" kd_status kd_matmul_2bit_f16(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                                        const float* centres_v, int64_t n, int64_t m, const void* x,
                                        const void* xp, int64_t batch, int64_t ldx, float* y, int64_t ldy,
                                        void* stream) {
  const kd_fold_mat_f16 a{codes_u, codes_v, centres_u, centres_v, x, xp, y, n, m, ldx, ldy};
  return kd_matmul_2bit_f16_batch(&a, 1, batch, stream);
}

extern "C" kd_status kd_matmul_2bit_bf16(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                                         const float* centres_v, int64_t n, int64_t m, const void* x,
                                         const void* xp, int64_t batch, int64_t ldx, float* y, int64_t ldy,
                                         void* stream) {
  const kd_fold_mat_f16 a{codes_u, codes_v, centres_u, centres_v, x, xp, y, n, m, ldx, ldy};
  return kd_matmul_2bit_bf16_batch(&a, 1, batch, stream);
}
