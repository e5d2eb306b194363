// Randomized-Hadamard incoherence rotation (Sec. 4: the "+H" of Kashin-DCT+H is a
// randomized Hadamard transform applied to the weights before the decomposition).
//
// Per vector of length n:  forward  y = (I_{n/b} (x) H_b / sqrt b) diag(s) x,
//                          inverse  x = diag(s) (I_{n/b} (x) H_b / sqrt b) y,
// with the Sylvester Hadamard matrix H_b on each contiguous block of b entries,
// b = the largest power of two dividing n (at most 16384), and the signs s drawn
// like the decomposition's eps (SplitMix64 of seed + (j + 1) * gamma, bit 63 set
// means -1).
//
// The rotation is bound by HBM: it reads every entry once (2 or 4 B) and writes
// it once as fp32, with log2(b) additions per entry in between.  A team of b/16
// threads transforms one block: each thread keeps 16 entries in registers and
// applies four butterfly levels (16 = 2^4 index values) per pass; between passes
// the block goes through shared memory so that the next four index bits land
// inside each thread.  The butterfly levels of different index bits commute, so
// the forward rotation takes the low bits first (its load is 16 contiguous
// entries per thread, where the sign flip is one shared-memory word) and the
// inverse takes them last (its store is the contiguous one, after its sign flip).
#include <atomic>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "kashin.h"
#include "kd_math.cuh"

namespace kd {
namespace {

constexpr int kRhtMinLogB = 4;
constexpr int kRhtMaxLogB = 14;
constexpr int64_t kRhtMaxN = int64_t(1) << 16;  // the sign bits of one vector stay in shared memory (8 KB)

struct RhtParams {
  const void* x;
  float* y;
  int64_t n, ldx, ldy, units;
  uint64_t seed;
  float scale;
  int dtype;
  int vec_in;   // the contiguous (forward) load may use 16-byte accesses
  int vec_out;  // the contiguous (inverse) store may use 16-byte accesses
};

KD_HD constexpr int rht_threads(int log_b) { return ((1 << log_b) / 16) > 256 ? ((1 << log_b) / 16) : 256; }

// shared-memory slot of block index i: one pad word per 16 entries keeps the
// 16-strided accesses of the first pass conflict-free
__device__ __forceinline__ int rpad(int i) { return i + (i >> 4); }

// radix of pass K: four index bits, fewer in the last pass when log2 b % 4 != 0
template <int LOG_B, int K>
KD_HD constexpr int rht_radix() {
  return (LOG_B - 4 * K) >= 4 ? 16 : (1 << (LOG_B - 4 * K));
}

// Block index held in register e of thread t during pass K (bits 4K .. 4K+3 of
// the index vary with e).  Pass 0: 16 contiguous entries.  Full passes: stride
// S = 16^K inside a run of 16 S.  A short last pass (radix R < 16): 16/R groups
// of R entries at stride S, consecutive threads on consecutive groups.
template <int LOG_B, int K>
__device__ __forceinline__ int rht_index(int t, int e) {
  constexpr int B = 1 << LOG_B;
  constexpr int TB = B / 16;
  constexpr int S = 1 << (4 * K);
  constexpr int R = rht_radix<LOG_B, K>();
  if constexpr (K == 0) {
    return 16 * t + e;
  } else if constexpr (R == 16) {
    return (t & (S - 1)) + S * e + 16 * S * (t / S);
  } else {
    return t + TB * (e / R) + S * (e % R);
  }
}

// Walsh-Hadamard butterflies on each group of R consecutive registers
template <int R>
__device__ __forceinline__ void fwht_groups(float (&r)[16]) {
#pragma unroll
  for (int h = 1; h < R; h <<= 1) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if ((i & h) == 0) {
        const float a = r[i], b = r[i + h];
        r[i] = __fadd_rn(a, b);
        r[i + h] = __fsub_rn(a, b);
      }
    }
  }
}

__device__ __forceinline__ float flip(float v, uint32_t bit) {
  return __int_as_float(__float_as_int(v) ^ (int)(bit << 31));
}

__device__ __forceinline__ float load_one(const void* x, int dtype, int64_t o) {
  if (dtype == KD_F32) return __ldg(static_cast<const float*>(x) + o);
  if (dtype == KD_F16) return __half2float(__ldg(static_cast<const __half*>(x) + o));
  return __bfloat162float(__ldg(static_cast<const __nv_bfloat16*>(x) + o));
}

// 16 contiguous entries starting at element offset o
__device__ __forceinline__ void load16(const RhtParams& p, int64_t o, float (&r)[16]) {
  if (p.vec_in) {
    if (p.dtype == KD_F32) {
      const float4* q = reinterpret_cast<const float4*>(static_cast<const float*>(p.x) + o);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const float4 a = __ldg(q + v);
        r[4 * v] = a.x; r[4 * v + 1] = a.y; r[4 * v + 2] = a.z; r[4 * v + 3] = a.w;
      }
    } else {
      const uint4* q = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p.x) + o);
#pragma unroll
      for (int v = 0; v < 2; ++v) {
        const uint4 a = __ldg(q + v);
        const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          float2 f;
          if (p.dtype == KD_F16) {
            f = __half22float2(*reinterpret_cast<const __half2*>(&w[h]));
          } else {
            f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[h]));
          }
          r[8 * v + 2 * h] = f.x;
          r[8 * v + 2 * h + 1] = f.y;
        }
      }
    }
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e) r[e] = load_one(p.x, p.dtype, o + e);
  }
}

template <int LOG_B, bool INV>
__global__ void __launch_bounds__(rht_threads(LOG_B)) rht_kernel(RhtParams p) {
  constexpr int B = 1 << LOG_B;
  constexpr int TB = B / 16;
  constexpr int THREADS = rht_threads(LOG_B);
  constexpr int TEAMS = THREADS / TB;
  constexpr int NPASS = (LOG_B + 3) / 4;
  constexpr int SLOTS = B + B / 16;  // rpad(B - 1) < SLOTS
  extern __shared__ __align__(16) float smem[];
  const int words = (int)((p.n + 31) / 32);
  uint32_t* sbits = reinterpret_cast<uint32_t*>(smem);
  const int team = threadIdx.x / TB;
  const int t = threadIdx.x % TB;
  float* buf = smem + ((words + 3) & ~3) + team * SLOTS;

  // the vector's sign bits, once per CTA
  for (int wd = threadIdx.x; wd < words; wd += THREADS) {
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; ++bb) {
      const int64_t j = (int64_t)wd * 32 + bb;
      if (j >= p.n) break;
      bits |= (uint32_t)(splitmix64_mix(p.seed + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull) >> 63) << bb;
    }
    sbits[wd] = bits;
  }
  __syncthreads();

  const int64_t nblk = p.n / B;
  for (int64_t base = (int64_t)blockIdx.x * TEAMS; base < p.units; base += (int64_t)gridDim.x * TEAMS) {
    const int64_t unit = base + team;
    const bool active = unit < p.units;
    const int64_t j = active ? unit / nblk : 0;
    const int64_t off = active ? (unit - j * nblk) * B : 0;  // block start inside the vector
    float r[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) r[e] = 0.f;
    // contiguous run of this thread in pass 0: entries off + 16 t .. + 15 (one sign half-word)
    const int64_t run = off + 16 * t;
    const uint32_t run_bits = (sbits[run >> 5] >> (run & 16)) & 0xFFFFu;

    if (active) {
      if constexpr (!INV) {
        load16(p, j * p.ldx + run, r);
#pragma unroll
        for (int e = 0; e < 16; ++e) r[e] = flip(r[e], (run_bits >> e) & 1u);
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e)
          r[e] = load_one(p.x, p.dtype, j * p.ldx + off + rht_index<LOG_B, NPASS - 1>(t, e));
      }
    }

    static_for<0, NPASS>([&](auto kk) {
      constexpr int KI = decltype(kk)::value;
      constexpr int K = INV ? NPASS - 1 - KI : KI;
      if constexpr (KI > 0) {
        constexpr int KP = INV ? K + 1 : K - 1;
        __syncthreads();  // the previous unit's reads of buf are done
#pragma unroll
        for (int e = 0; e < 16; ++e) buf[rpad(rht_index<LOG_B, KP>(t, e))] = r[e];
        __syncthreads();
#pragma unroll
        for (int e = 0; e < 16; ++e) r[e] = buf[rpad(rht_index<LOG_B, K>(t, e))];
      }
      fwht_groups<rht_radix<LOG_B, K>()>(r);
    });

#pragma unroll
    for (int e = 0; e < 16; ++e) r[e] = __fmul_rn(r[e], p.scale);
    if (active) {
      if constexpr (!INV) {
        float* yo = p.y + j * p.ldy + off;
#pragma unroll
        for (int e = 0; e < 16; ++e) yo[rht_index<LOG_B, NPASS - 1>(t, e)] = r[e];
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) r[e] = flip(r[e], (run_bits >> e) & 1u);
        float* yo = p.y + j * p.ldy + run;
        if (p.vec_out) {
          float4* q = reinterpret_cast<float4*>(yo);
#pragma unroll
          for (int v = 0; v < 4; ++v) q[v] = make_float4(r[4 * v], r[4 * v + 1], r[4 * v + 2], r[4 * v + 3]);
        } else {
#pragma unroll
          for (int e = 0; e < 16; ++e) yo[e] = r[e];
        }
      }
    }
  }
}

size_t rht_smem_bytes(int log_b, int64_t n) {
  const int B = 1 << log_b;
  const int teams = rht_threads(log_b) / (B / 16);
  const size_t words = (size_t)((n + 31) / 32);
  return ((words + 3) & ~size_t(3)) * 4 + (size_t)teams * (B + B / 16) * 4;
}

template <int LOG_B, bool INV>
cudaError_t launch_rht(const RhtParams& p, cudaStream_t s) {
  constexpr int THREADS = rht_threads(LOG_B);
  constexpr int TEAMS = THREADS / ((1 << LOG_B) / 16);
  const size_t smem = rht_smem_bytes(LOG_B, p.n);
  cudaError_t e = cudaFuncSetAttribute(rht_kernel<LOG_B, INV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, rht_kernel<LOG_B, INV>, THREADS, smem)) !=
      cudaSuccess)
    return e;
  if (per < 1) return cudaErrorInvalidConfiguration;
  const int64_t want = (p.units + TEAMS - 1) / TEAMS;
  const int64_t cap = (int64_t)per * sms;
  const int grid = (int)(want < cap ? want : cap);
  rht_kernel<LOG_B, INV><<<grid, THREADS, smem, s>>>(p);
  return cudaGetLastError();
}

template <bool INV>
cudaError_t dispatch_rht(int log_b, const RhtParams& p, cudaStream_t s) {
  switch (log_b) {
    case 4: return launch_rht<4, INV>(p, s);
    case 5: return launch_rht<5, INV>(p, s);
    case 6: return launch_rht<6, INV>(p, s);
    case 7: return launch_rht<7, INV>(p, s);
    case 8: return launch_rht<8, INV>(p, s);
    case 9: return launch_rht<9, INV>(p, s);
    case 10: return launch_rht<10, INV>(p, s);
    case 11: return launch_rht<11, INV>(p, s);
    case 12: return launch_rht<12, INV>(p, s);
    case 13: return launch_rht<13, INV>(p, s);
    case 14: return launch_rht<14, INV>(p, s);
    default: return cudaErrorInvalidValue;
  }
}

int log2_block(int64_t n) {
  int64_t b = n & -n;
  if (b > (int64_t(1) << kRhtMaxLogB)) b = int64_t(1) << kRhtMaxLogB;
  int l = 0;
  while ((int64_t(1) << l) < b) ++l;
  return l;
}

}  // namespace
}  // namespace kd

extern "C" int64_t kd_rht_block(int64_t n) {
  if (n < 16 || n % 16 != 0 || n > kd::kRhtMaxN) return 0;
  return int64_t(1) << kd::log2_block(n);
}

extern "C" kd_status kd_rht(const void* x, kd_dtype dtype, int64_t n, int64_t m, int64_t ldx, uint64_t seed,
                            int inverse, float* y, int64_t ldy, void* stream) {
  if (kd_rht_block(n) == 0) return KD_ERR_UNSUPPORTED_N;
  if (m < 0 || ldx < n || ldy < n || (dtype != KD_F32 && dtype != KD_F16 && dtype != KD_BF16) ||
      (inverse != 0 && inverse != 1))
    return KD_ERR_INVALID_ARG;
  if (m == 0) return KD_OK;
  if (!x || !y) return KD_ERR_INVALID_ARG;
  // in place only over the same fp32 array with the same stride
  if (static_cast<const void*>(y) == x && (dtype != KD_F32 || ldx != ldy)) return KD_ERR_INVALID_ARG;
  const int log_b = kd::log2_block(n);
  kd::RhtParams p;
  p.x = x;
  p.y = y;
  p.n = n;
  p.ldx = ldx;
  p.ldy = ldy;
  p.units = m * (n >> log_b);
  p.seed = seed;
  p.scale = (float)(1.0 / __builtin_sqrt((double)(int64_t(1) << log_b)));
  p.dtype = (int)dtype;
  const int esz = dtype == KD_F32 ? 4 : 2;
  p.vec_in = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && ((ldx * esz) % 16 == 0);
  p.vec_out = (reinterpret_cast<uintptr_t>(y) % 16 == 0) && ((ldy * 4) % 16 == 0);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const cudaError_t e = inverse ? kd::dispatch_rht<true>(log_b, p, s) : kd::dispatch_rht<false>(log_b, p, s);
  return e == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}
