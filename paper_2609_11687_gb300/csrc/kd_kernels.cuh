// Kashin-DCT decomposition kernels (sm_103a).
//
// One team of T threads owns a PAIR of vectors (2j, 2j+1) for the whole of
// Algorithm 1: the two real vectors are the real and imaginary parts of one
// complex vector held on-chip, so one complex FFT of length N transforms both.
//
// Transform (Sec. 3.1, Alg. 1: P z = IDCT(eps * DCT(z))).  With the vector held
// in Makhoul's even/odd order v[p] = x[2p], v[N-1-p] = x[2p+1] (J. Makhoul, IEEE
// TASSP 1980) the orthonormal DCT-II is Re(exp(-i pi k / 2N) DFT(v)_k) up to a
// per-k scale that cancels in IDCT o T_eps o DCT, and P becomes
//     P' z = IDFT( M( DFT(z) ) ),
//     M: Z'_k = e+_k Z_k + e-_k exp(i pi k/N) Z_{N-k},  e+-_k = (eps_k +- eps_{N-k})/2,
//        Z'_0 = eps_0 Z_0,  Z'_{N/2} = eps_{N/2} Z_{N/2},
// which is complex-linear, so it acts on both packed vectors at once.
//
// The greedy steps (sign, l1 norm, update) are permutation-invariant, so the
// vectors stay in Makhoul order in the "spatial" domain for all k blocks: the
// forward FFT runs decimation-in-frequency (natural in, digit-reversed out), M
// pairs digit-reversed slots, and the inverse runs the mirror passes back to
// natural order -- no reordering pass exists anywhere.
//
// Data layout per team: the spatial vector lives in registers, E = R0 complex
// values per thread at positions t + j*T (which is exactly the first radix
// pass's group), and a padded shared-memory buffer of N float2 carries the
// exchanges between radix passes.  The factor u lives in registers (the smallest
// plans), in shared memory after the team's buffer (up to n = 11008), or in a
// per-team slot of the workspace (n = 14336, 16384); the last two are updated in
// place by each u-step.  vhat is not stored during the loop: after the last block
// it is recovered as P(x - u - r) (P^2 = I).
#pragma once

#include <cstdint>
#include <type_traits>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "kd_bulk.cuh"
#include "kd_math.cuh"
#include "kd_xform.cuh"

namespace kd {

enum { DT_F32 = 0, DT_F16 = 1, DT_BF16 = 2 };
enum { LAY_ROWS = 0, LAY_COLS = 1 };

// Natural index of Makhoul position p (N even).
template <int N>
__device__ __forceinline__ int nat_of(int p) {
  return (p < N / 2) ? 2 * p : 2 * N - 1 - 2 * p;
}

// Sum of v over the team; every thread receives the identical result.
template <class PL>
__device__ __forceinline__ float2 team_sum(float2 v, float2* red, int lt, int& parity) {
  constexpr int W = PL::T < 32 ? PL::T : 32;
#pragma unroll
  for (int off = W / 2; off > 0; off >>= 1) {
    v.x = __fadd_rn(v.x, __shfl_xor_sync(0xffffffffu, v.x, off));
    v.y = __fadd_rn(v.y, __shfl_xor_sync(0xffffffffu, v.y, off));
  }
  if constexpr (PL::NW == 1) {
    return v;
  } else {
    float2* r = red + parity * PL::NW;
    parity ^= 1;
    if ((lt & 31) == 0) r[lt >> 5] = v;
    team_sync<PL>();
    float2 s = r[0];
#pragma unroll
    for (int w = 1; w < PL::NW; ++w) s = cadd(s, r[w]);
    return s;
  }
}

// Sum of K (a power of two <= 32) per-thread values over the team; every thread
// receives all K totals in `tot` (fixed summation order: deterministic).
// Whole-warp teams: butterfly reduce-scatter (K - 1 shuffles, then one shuffle per
// remaining lane bit) leaves lane l with its warp's total of value l % K, then a
// fixed-order sum over warps through `scratch` (K (NW + 1) floats of shared
// memory).  Narrower teams: butterfly all-reduce over the team's lanes.
template <class PL, int K>
__device__ __forceinline__ void team_sum_k(float (&v)[K], float (&tot)[K], float* scratch, int lt) {
  static_assert(K >= 1 && K <= 32 && (K & (K - 1)) == 0, "K must be a power of two <= 32");
  if constexpr (PL::T < 32) {
#pragma unroll
    for (int off = PL::T / 2; off > 0; off >>= 1) {
#pragma unroll
      for (int i = 0; i < K; ++i) v[i] = __fadd_rn(v[i], __shfl_xor_sync(0xffffffffu, v[i], off));
    }
#pragma unroll
    for (int i = 0; i < K; ++i) tot[i] = v[i];
  } else {
    const int lane = lt & 31;
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
    // lane l now holds its warp's total of value l % K
    float* wpart = scratch;             // [NW][K]
    float* fin = scratch + K * PL::NW;  // [K]
    if (lane < K) wpart[(lt >> 5) * K + lane] = v[0];
    team_sync<PL>();
    if (lt < K) {
      float t = wpart[lt];
#pragma unroll
      for (int w = 1; w < PL::NW; ++w) t = __fadd_rn(t, wpart[w * K + lt]);
      fin[lt] = t;
    }
    team_sync<PL>();
#pragma unroll
    for (int i = 0; i < K; ++i) tot[i] = fin[i];
    team_sync<PL>();
  }
}

// Shared memory of a CTA: [twiddle table (if staged)][team 0 buffer | red][team 1 ...].
// Copies the table in and returns this team's buffer.
template <class PL>
__device__ __forceinline__ float2* cta_setup(float2* smem, const float2* __restrict__ twg, const float2*& tw,
                                             int team) {
  if constexpr (PL::TW_SMEM) {
    for (int i = threadIdx.x; i < PL::TWN; i += blockDim.x) smem[i] = __ldg(&twg[i]);
    __syncthreads();
    tw = smem;
  } else {
    tw = twg;
  }
  return smem + PL::SMEM_TW / sizeof(float2) + team * PL::TEAM;
}

// ---------------------------------------------------------------------------
// Element loads / stores
// ---------------------------------------------------------------------------
// dtype and layout are uniform per launch: branching on them costs nothing
// measurable next to the transform and keeps one kernel per plan.
__device__ __forceinline__ float load_elem(const void* __restrict__ w, int dt, int64_t idx) {
  if (dt == DT_F32) return __ldg(reinterpret_cast<const float*>(w) + idx);
  if (dt == DT_F16) return __half2float(__ldg(reinterpret_cast<const __half*>(w) + idx));
  return __bfloat162float(__ldg(reinterpret_cast<const __nv_bfloat16*>(w) + idx));
}

__device__ __forceinline__ void store_elem(void* __restrict__ w, int dt, int64_t idx, float x) {
  if (dt == DT_F32) {
    reinterpret_cast<float*>(w)[idx] = x;
  } else if (dt == DT_F16) {
    reinterpret_cast<__half*>(w)[idx] = __float2half_rn(x);
  } else {
    reinterpret_cast<__nv_bfloat16*>(w)[idx] = __float2bfloat16_rn(x);
  }
}

__device__ __forceinline__ int64_t elem_index(int lay, int64_t vec, int i, int64_t ld) {
  return (lay == LAY_ROWS) ? vec * ld + i : (int64_t)i * ld + vec;
}

// 2^e as float for -126 <= e <= 127 (exact)
__device__ __forceinline__ float pow2f(int e) { return __int_as_float((127 + e) << 23); }

// ---------------------------------------------------------------------------
// Kernel parameters
// ---------------------------------------------------------------------------
struct DecParams {
  const void* w;
  int dtype, layout;
  int64_t n, m, ld;
  int iters;
  int kmeans_iters;
  uint32_t* codes_u;
  uint32_t* codes_v;
  float* centres_u;
  float* centres_v;
  float* coeffs;
  float* u;
  float* vhat;
  float* resid;
  int8_t* trace;
  const float2* twt;      // access-ordered twiddle table (global)
  const uint32_t* eps;
  uint32_t* status;
  float2* uslots;
  int64_t npairs;
  // 1: every vector of the launch is a contiguous, 16-byte aligned row (KD_VEC_ROWS,
  // w and ld * element size multiples of 16 bytes): pairs are staged by bulk copies
  int bulk;
};

// Several matrices of one vector length in one launch (kd_decompose_batch): their
// pairs are numbered one after another; matrix i owns global pairs
// [pair0, pair0 + ceil(m / 2)) and the sign bits at eps + i * ceil(n / 32).
constexpr int kMaxBatch = 32;
struct BatchMat {
  const void* w;
  int64_t m, ld, pair0;
  uint32_t* codes_u;
  uint32_t* codes_v;
  float* centres_u;
  float* centres_v;
  float* coeffs;
};
struct BatchParams {
  int count;  // 0: the single matrix of DecParams
  BatchMat mat[kMaxBatch];
};

// sign(r) * c with sign(0) = 0
__device__ __forceinline__ float signed_step(float r, float c) {
  return (r == 0.f) ? 0.f : copysignf(c, r);
}

// ---------------------------------------------------------------------------
// kd_decompose kernel
// ---------------------------------------------------------------------------
template <class PL, bool TRACE>
__global__ void __launch_bounds__(PL::THREADS, PL::MINB) decompose_kernel(DecParams p, const __grid_constant__ BatchParams bp) {
  constexpr int N = PL::N;
  constexpr int T = PL::T;
  constexpr int E = PL::E;
  extern __shared__ __align__(16) float2 smem[];
  const int team = threadIdx.x / T;
  const int lt = threadIdx.x - team * T;
  const float2* tw;
  float2* buf = cta_setup<PL>(smem, p.twt, tw, team);
  float2* red = buf + PL::BUF;
  Xform<PL> xf;
  xf.init(buf, tw, p.eps, lt);
  int parity = 0;
  const int nsteps = 4 * p.iters + 2 * p.kmeans_iters;  // trace rows per vector

  float2 uu_reg[PL::UMODE == UREG ? E : 1];
  // u outside registers: per-team workspace slot (global) or shared memory after red
  float2* uslot = nullptr;
  if constexpr (PL::UMODE == UGMEM) uslot = p.uslots + ((int64_t)blockIdx.x * PL::Q + team) * N;
  if constexpr (PL::UMODE == USMEM) uslot = red + PL::RED;

  static_assert(PL::SMEM_TW % 16 == 0 && PL::TEAM % 2 == 0, "team buffers must start 16-byte aligned");
  // Staged input (p.bulk): the pair's two rows land in the team's exchange buffer by
  // bulk copy (16-byte aligned rows, completion on the team's mbarrier), and every
  // thread reads its elements in Makhoul order from there; the same staging re-reads
  // x after the last block.  Otherwise the elements are gathered from global memory.
  uint64_t* mbar = reinterpret_cast<uint64_t*>(buf + PL::BUF + PL::RED + PL::USL);
  uint32_t mphase = 0;
  if (p.bulk) {
    if (lt == 0) {
      mbar_init(mbar, 1);
      mbar_init_fence();
    }
    __syncthreads();
  }
  const int esz = p.dtype == DT_F32 ? 4 : 2;

  int cur_mat = 0;  // matrix whose sign set the transform holds (batch launches)
  for (int64_t base = (int64_t)blockIdx.x * PL::Q; base < p.npairs; base += (int64_t)gridDim.x * PL::Q) {
    const int64_t pair = base + team;
    const bool active = pair < p.npairs;
    int64_t pr = active ? pair : base;
    // this pair's matrix: index mi into bp (batched launch) or DecParams' matrix;
    // its fields are re-read from the parameter space where used (no registers held)
    int mi = 0;
    if (PL::BATCH && bp.count > 0) {
      while (mi + 1 < bp.count && pr >= bp.mat[mi + 1].pair0) ++mi;
      pr -= bp.mat[mi].pair0;
      if (mi != cur_mat) {  // uniform per team: Q == 1 whenever T > 32
        xf.set_eps(p.eps + (int64_t)mi * ((N + 31) / 32));
        cur_mat = mi;
      }
    }
    const bool batched = PL::BATCH && bp.count > 0;
    auto w_in = [&]() -> const void* { return batched ? bp.mat[mi].w : p.w; };
    auto ld_in = [&]() -> int64_t { return batched ? bp.mat[mi].ld : p.ld; };
    const int64_t m_in = batched ? bp.mat[mi].m : p.m;
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < m_in;
    const int64_t colB = hasB ? colA + 1 : colA;

    // Bulk-copy both rows of the pair into buf (free: every reader of the previous
    // use passed a team barrier); false if the copy did not land in time, decided for
    // the whole CTA so that its barriers stay uniform.
    auto stage_rows = [&](bool prefetch_next) -> bool {
      const uint32_t rb = (uint32_t)(N * esz);
      if (lt == 0) {
        const char* w0 = static_cast<const char*>(w_in());
        fence_proxy_async_smem();  // earlier generic accesses to buf before the copy's writes
        mbar_arrive_expect_tx(mbar, hasB ? 2 * rb : rb);
        bulk_copy_g2s(buf, w0 + colA * ld_in() * esz, rb, mbar);
        if (hasB) bulk_copy_g2s(reinterpret_cast<char*>(buf) + rb, w0 + colB * ld_in() * esz, rb, mbar);
        // the rows this team takes next, into L2 while this pair is decomposed
        const int64_t nxt = pair + (int64_t)gridDim.x * PL::Q;
        if (prefetch_next && nxt < p.npairs) {
          int mn = 0;
          int64_t pn = nxt;
          if (batched) {
            while (mn + 1 < bp.count && pn >= bp.mat[mn + 1].pair0) ++mn;
            pn -= bp.mat[mn].pair0;
          }
          const char* wn = static_cast<const char*>(batched ? bp.mat[mn].w : p.w);
          const int64_t ldn = batched ? bp.mat[mn].ld : p.ld;
          const int64_t mm = batched ? bp.mat[mn].m : p.m;
          bulk_prefetch_l2(wn + 2 * pn * ldn * esz, rb);
          if (2 * pn + 1 < mm) bulk_prefetch_l2(wn + (2 * pn + 1) * ldn * esz, rb);
        }
      }
      const bool ok = mbar_wait_bounded(mbar, mphase);
      mphase ^= 1u;
      if (__syncthreads_or(!ok)) {
        if (lt == 0) {
          atomicOr(p.status, 2u);
          mbar_wait_bounded(mbar, mphase ^ 1u);  // let the copy land before the CTA leaves
        }
        __syncthreads();
        return false;
      }
      return true;
    };
    // element nat of staged row c (0 = vector A, 1 = vector B)
    auto staged = [&](int c, int nat) -> float {
      const char* row = reinterpret_cast<const char*>(buf) + c * N * esz;
      if (p.dtype == DT_F32) return reinterpret_cast<const float*>(row)[nat];
      if (p.dtype == DT_F16) return __half2float(reinterpret_cast<const __half*>(row)[nat]);
      return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(row)[nat]);
    };

    // ---- load the pair in Makhoul order: position lt + j*T ----
    // (staged: the first greedy step's team reduction, or the transform's opening
    // barrier for single-warp teams, orders these reads before buf is written again)
    float2 r[E];
    float2 acc = make_float2(0.f, 0.f);
    if (p.bulk && !stage_rows(true)) return;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const int nat = nat_of<N>(lt + j * T);
      float a, b;
      if (p.bulk) {
        a = staged(0, nat);
        b = hasB ? staged(1, nat) : 0.f;
      } else {
        a = load_elem(w_in(), p.dtype, elem_index(p.layout, colA, nat, ld_in()));
        b = hasB ? load_elem(w_in(), p.dtype, elem_index(p.layout, colB, nat, ld_in())) : 0.f;
      }
      r[j] = make_float2(a, b);
      acc.x = __fadd_rn(acc.x, fabsf(a));
      acc.y = __fadd_rn(acc.y, fabsf(b));
    }
    float2 sum0 = team_sum<PL>(acc, red, lt, parity);
    // ---- exact power-of-two normalisation: c1 of each vector lands in [1, 2) ----
    int sA = 0, sB = 0;
    {
      const bool finA = isfinite(sum0.x), finB = isfinite(sum0.y);
      if (active && lt == 0 && (!finA || !finB)) atomicOr(p.status, 1u);
      const float cA = __fdiv_rn(sum0.x, (float)N), cB = __fdiv_rn(sum0.y, (float)N);
      if (finA && cA > 0.f) sA = max(-100, min(100, -ilogbf(cA)));
      if (finB && cB > 0.f) sB = max(-100, min(100, -ilogbf(cB)));
    }
    const float scA = pow2f(sA), scB = pow2f(sB);
    // An all-zero vector must stay exactly zero; the packed transform would
    // otherwise leak its partner's rounding error into it.
    const bool liveA = sum0.x > 0.f, liveB = sum0.y > 0.f;
    auto mask_dead = [&](float2(&v)[E]) {
      if (!liveA || !liveB) {
#pragma unroll
        for (int j = 0; j < E; ++j) v[j] = make_float2(liveA ? v[j].x : 0.f, liveB ? v[j].y : 0.f);
      }
    };
#pragma unroll
    for (int j = 0; j < E; ++j) r[j] = make_float2(__fmul_rn(r[j].x, scA), __fmul_rn(r[j].y, scB));
    sum0 = make_float2(__fmul_rn(sum0.x, scA), __fmul_rn(sum0.y, scB));

    if constexpr (PL::UMODE == UREG) {
#pragma unroll
      for (int j = 0; j < E; ++j) uu_reg[j] = make_float2(0.f, 0.f);
    } else {
#pragma unroll
      for (int j = 0; j < E; ++j) uslot[lt + j * T] = make_float2(0.f, 0.f);
    }
    float2 coef[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) coef[q] = make_float2(0.f, 0.f);

    const bool tracing = TRACE && active;
    int8_t* trA = nullptr;
    int8_t* trB = nullptr;
    if (TRACE && tracing) {
      trA = p.trace + colA * (int64_t)nsteps * N;
      trB = p.trace + colB * (int64_t)nsteps * N;
    }

    // One atomic greedy step on the values in r: lambda = ||r||_1 / N per vector,
    // r -= sign(r) lambda; the applied step is returned through `add` callback.
    auto greedy = [&](int step, bool have_sum, float2 presum, auto&& add) -> float2 {
      float2 s = presum;
      if (!have_sum) {
        float2 a = make_float2(0.f, 0.f);
#pragma unroll
        for (int j = 0; j < E; ++j) {
          a.x = __fadd_rn(a.x, fabsf(r[j].x));
          a.y = __fadd_rn(a.y, fabsf(r[j].y));
        }
        s = team_sum<PL>(a, red, lt, parity);
      }
      const float lA = __fdiv_rn(s.x, (float)N);
      const float lB = __fdiv_rn(s.y, (float)N);
#pragma unroll
      for (int j = 0; j < E; ++j) {
        if (TRACE && tracing) {
          const int nat = nat_of<N>(lt + j * T);
          const int64_t off = (int64_t)step * N + nat;
          trA[off] = (int8_t)((r[j].x > 0.f) - (r[j].x < 0.f));
          if (hasB) trB[off] = (int8_t)((r[j].y > 0.f) - (r[j].y < 0.f));
        }
        const float dA = signed_step(r[j].x, lA);
        const float dB = signed_step(r[j].y, lB);
        r[j].x = __fsub_rn(r[j].x, dA);
        r[j].y = __fsub_rn(r[j].y, dB);
        add(j, dA, dB);
      }
      return make_float2(lA, lB);
    };
    auto add_u = [&](int j, float dA, float dB) {
      if constexpr (PL::UMODE == UREG) {
        uu_reg[j].x = __fadd_rn(uu_reg[j].x, dA);
        uu_reg[j].y = __fadd_rn(uu_reg[j].y, dB);
      }
    };
    auto add_none = [&](int, float, float) {};

    const float isA = pow2f(-sA), isB = pow2f(-sB);
    auto u_at = [&](int j) -> float2 {
      if constexpr (PL::UMODE == UREG) {
        return uu_reg[j];
      } else {
        return uslot[lt + j * T];
      }
    };

    // Half-block hb: even = two greedy steps from Q_N (u), odd = two from P Q_N (vhat),
    // each followed by P; the last one (hb == 2k) forms x - u - r and its P gives vhat.
    // One call site for the transform keeps the kernel's code footprint small.
    int step = 0;
    const int HB = 2 * p.iters;
    for (int hb = 0; hb <= HB; ++hb) {
      if (hb == HB) {
        if (active && p.resid) {
#pragma unroll
          for (int j = 0; j < E; ++j) {
            const int nat = nat_of<N>(lt + j * T);
            p.resid[colA * N + nat] = __fmul_rn(r[j].x, isA);
            if (hasB) p.resid[colB * N + nat] = __fmul_rn(r[j].y, isB);
          }
        }
        if (p.bulk) {
          team_sync<PL>();  // the last transform's readers of buf are done
          if (!stage_rows(false)) return;
        }
#pragma unroll
        for (int j = 0; j < E; ++j) {
          const int nat = nat_of<N>(lt + j * T);
          float a, b;
          if (p.bulk) {
            a = __fmul_rn(staged(0, nat), scA);
            b = hasB ? __fmul_rn(staged(1, nat), scB) : 0.f;
          } else {
            a = __fmul_rn(load_elem(w_in(), p.dtype, elem_index(p.layout, colA, nat, ld_in())), scA);
            b = hasB ? __fmul_rn(load_elem(w_in(), p.dtype, elem_index(p.layout, colB, nat, ld_in())), scB) : 0.f;
          }
          const float2 uj = u_at(j);
          r[j] = make_float2(__fsub_rn(__fsub_rn(a, uj.x), r[j].x), __fsub_rn(__fsub_rn(b, uj.y), r[j].y));
        }
        if (p.iters == 0) {
#pragma unroll
          for (int j = 0; j < E; ++j) r[j] = make_float2(0.f, 0.f);
          break;
        }
        team_sync<PL>();  // the last transform's readers of buf (or of the staged x) are done
      } else if ((hb & 1) == 0) {
        // two greedy steps from Q_N (update u).  u outside registers (shared memory,
        // or the workspace slot for the longest vectors) is updated in place by both
        // steps: two roundings, as with two separate updates
        auto add_slot = [&](int j, float dA, float dB) {
          if constexpr (PL::UMODE == UREG) {
            add_u(j, dA, dB);
          } else {
            float2 uj = uslot[lt + j * T];
            uj.x = __fadd_rn(uj.x, dA);
            uj.y = __fadd_rn(uj.y, dB);
            uslot[lt + j * T] = uj;
          }
        };
        const float2 l1 = greedy(step, hb == 0, sum0, add_slot);
        ++step;
        const float2 l2 = greedy(step, false, sum0, add_slot);
        ++step;
        if (hb == 0) {
          coef[0] = l1;
          coef[1] = l2;
        }
      } else {
        // two greedy steps from P Q_N on y = P rho (vhat is implicit: P (x - u - r) at the end)
        const float2 l3 = greedy(step, false, sum0, add_none);
        ++step;
        const float2 l4 = greedy(step, false, sum0, add_none);
        ++step;
        if (hb == 1) {
          coef[2] = l3;
          coef[3] = l4;
        }
      }
      xf.apply(r);
      mask_dead(r);
    }
    float2(&vh)[E] = r;  // r now holds vhat

    // ---- optional dense factors (natural order, scaled back) ----
    if (active && (p.u || p.vhat)) {
#pragma unroll
      for (int j = 0; j < E; ++j) {
        const int nat = nat_of<N>(lt + j * T);
        const float2 uj = u_at(j);
        if (p.u) {
          p.u[colA * N + nat] = __fmul_rn(uj.x, isA);
          if (hasB) p.u[colB * N + nat] = __fmul_rn(uj.y, isB);
        }
        if (p.vhat) {
          p.vhat[colA * N + nat] = __fmul_rn(vh[j].x, isA);
          if (hasB) p.vhat[colB * N + nat] = __fmul_rn(vh[j].y, isB);
        }
      }
    }

    // ---- centres: closed form +-a1 +-a2 (Sec. 2.1), then optional Lloyd refinement ----
    // cen[f][c][q]: factor f (0 = u, 1 = vhat), vector c (0 = A, 1 = B), ascending centre q
    float cen[2][2][4];
    {
      const float a1[2][2] = {{coef[0].x, coef[0].y}, {coef[2].x, coef[2].y}};
      const float a2[2][2] = {{coef[1].x, coef[1].y}, {coef[3].x, coef[3].y}};
#pragma unroll
      for (int f = 0; f < 2; ++f)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const float outer = __fadd_rn(a1[f][c], a2[f][c]);
          const float inner = fabsf(__fsub_rn(a1[f][c], a2[f][c]));
          cen[f][c][0] = -outer;
          cen[f][c][1] = -inner;
          cen[f][c][2] = inner;
          cen[f][c][3] = outer;
        }
    }
    // decision boundaries: closed form uses -max(a1,a2), 0, +max(a1,a2) exactly
    float bnd[2][2][3];
#pragma unroll
    for (int f = 0; f < 2; ++f)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const float mm = fmaxf(f ? (c ? coef[2].y : coef[2].x) : (c ? coef[0].y : coef[0].x),
                               f ? (c ? coef[3].y : coef[3].x) : (c ? coef[1].y : coef[1].x));
        bnd[f][c][0] = -mm;
        bnd[f][c][1] = 0.f;
        bnd[f][c][2] = mm;
      }
    auto code_of = [](float x, const float (&b)[3]) -> int { return (x > b[0]) + (x > b[1]) + (x > b[2]); };
    auto val = [&](int j, int f, int c) -> float {
      if (f == 0) {
        const float2 uj = u_at(j);
        return c ? uj.y : uj.x;
      }
      return c ? vh[j].y : vh[j].x;
    };
    {
      for (int it = 0; it < p.kmeans_iters; ++it) {
        // one factor at a time.  Per vector c the thread accumulates, for each of the
        // three boundaries b_q, the sum and count of its values above b_q, plus the
        // total sum: cluster q holds the values above exactly q boundaries (ties
        // low, as the codes), so the per-cluster sums and counts are differences of
        // these -- 3 compare/select/add triples per value instead of 4.
#pragma unroll
        for (int f = 0; f < 2; ++f) {
          // [c*8 + q]: sum above b_q; [c*8 + 3 + q]: count above b_q; [c*8 + 6]: total
          float acc[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[i] = 0.f;
#pragma unroll
          for (int j = 0; j < E; ++j) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              const float x = val(j, f, c);
              if constexpr (TRACE) {
                if (tracing && (c == 0 || hasB)) {
                  const int nat = nat_of<N>(lt + j * T);
                  (c ? trB : trA)[(int64_t)(4 * p.iters + 2 * it + f) * N + nat] = (int8_t)code_of(x, bnd[f][c]);
                }
              }
              acc[c * 8 + 6] = __fadd_rn(acc[c * 8 + 6], x);
#pragma unroll
              for (int q = 0; q < 3; ++q) {
                const bool gt = x > bnd[f][c][q];
                acc[c * 8 + q] = __fadd_rn(acc[c * 8 + q], gt ? x : 0.f);
                acc[c * 8 + 3 + q] = __fadd_rn(acc[c * 8 + 3 + q], gt ? 1.f : 0.f);
              }
            }
          }
          float tot[16];
          team_sum_k<PL, 16>(acc, tot, reinterpret_cast<float*>(red), lt);
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const float* t = tot + c * 8;
            // counts are exact integers in fp32 (n <= 16384)
            const float sum[4] = {__fsub_rn(t[6], t[0]), __fsub_rn(t[0], t[1]), __fsub_rn(t[1], t[2]), t[2]};
            const float cnt[4] = {__fsub_rn((float)N, t[3]), __fsub_rn(t[3], t[4]), __fsub_rn(t[4], t[5]), t[5]};
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
              if (cnt[qq] > 0.f) cen[f][c][qq] = __fdiv_rn(sum[qq], cnt[qq]);
            }
#pragma unroll
            for (int qq = 0; qq < 3; ++qq)
              bnd[f][c][qq] = __fmul_rn(0.5f, __fadd_rn(cen[f][c][qq], cen[f][c][qq + 1]));
          }
        }
      }
    }

    // ---- 2-bit codes: nearest centre, ties low ----
    team_sync<PL>();  // everyone is done with buf
    uint8_t* cb = reinterpret_cast<uint8_t*>(buf);
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const int nat = nat_of<N>(lt + j * T);
      cb[0 * N + nat] = (uint8_t)code_of(val(j, 0, 0), bnd[0][0]);
      cb[1 * N + nat] = (uint8_t)code_of(val(j, 0, 1), bnd[0][1]);
      cb[2 * N + nat] = (uint8_t)code_of(val(j, 1, 0), bnd[1][0]);
      cb[3 * N + nat] = (uint8_t)code_of(val(j, 1, 1), bnd[1][1]);
    }
    team_sync<PL>();
    constexpr int WPV = N / 16;  // words per vector (N % 16 == 0 for every plan)
    static_assert(N % 16 == 0, "plans keep N a multiple of 16");
    if (active) {
      for (int wi = lt; wi < 4 * WPV; wi += T) {
        const int plane = wi / WPV;
        const int word = wi - plane * WPV;
        const uint4 q = *reinterpret_cast<const uint4*>(cb + plane * N + word * 16);
        const uint32_t qq[4] = {q.x, q.y, q.z, q.w};
        uint32_t packed = 0;
#pragma unroll
        for (int b4 = 0; b4 < 4; ++b4) {
#pragma unroll
          for (int by = 0; by < 4; ++by) packed |= ((qq[b4] >> (8 * by)) & 3u) << (2 * (4 * b4 + by));
        }
        const bool isB = (plane & 1) != 0;
        if (isB && !hasB) continue;
        const int64_t col = isB ? colB : colA;
        uint32_t* dst = (plane < 2) ? (batched ? bp.mat[mi].codes_u : p.codes_u)
                                    : (batched ? bp.mat[mi].codes_v : p.codes_v);
        dst[col * WPV + word] = packed;
      }
      if (lt == 0) {
        const float sc[2] = {isA, isB};
        for (int v2 = 0; v2 < (hasB ? 2 : 1); ++v2) {
          const int64_t col = v2 ? colB : colA;
          const float c1 = v2 ? coef[0].y : coef[0].x, c2 = v2 ? coef[1].y : coef[1].x;
          const float d1 = v2 ? coef[2].y : coef[2].x, d2 = v2 ? coef[3].y : coef[3].x;
          const float f = sc[v2];
          float* cu = (batched ? bp.mat[mi].centres_u : p.centres_u) + col * 4;
          float* cv = (batched ? bp.mat[mi].centres_v : p.centres_v) + col * 4;
          float* coeffs_out = batched ? bp.mat[mi].coeffs : p.coeffs;
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) {
            cu[qq] = __fmul_rn(cen[0][v2][qq], f);
            cv[qq] = __fmul_rn(cen[1][v2][qq], f);
          }
          if (coeffs_out) {
            float* co = coeffs_out + col * 4;
            co[0] = __fmul_rn(c1, f); co[1] = __fmul_rn(c2, f);
            co[2] = __fmul_rn(d1, f); co[3] = __fmul_rn(d2, f);
          }
        }
      }
    }
    team_sync<PL>();  // buf is reused by the next pair
  }
}

// ---------------------------------------------------------------------------
// kd_apply_p kernel: y_j = P x_j, fp32 vector-major.
// ---------------------------------------------------------------------------
struct ApplyParams {
  const float* x;
  float* y;
  int64_t n, m;
  const float2* twt;
  const uint32_t* eps;
  int64_t npairs;
};

// Several matrices of one vector length in one kd_apply_p launch (kd_apply_p_batch):
// matrix i owns the global pairs [pair0, pair0 + ceil(m / 2)) and the sign bits at
// eps + i * ceil(n / 32).
struct ApplyMat {
  const float* x;
  float* y;
  int64_t m, pair0;
};
struct ApplyBatch {
  int count;  // 0: the single matrix of ApplyParams
  ApplyMat mat[kMaxBatch];
};

template <class PL>
__global__ void __launch_bounds__(PL::THREADS, PL::MINB) apply_p_kernel(ApplyParams p,
                                                                        const __grid_constant__ ApplyBatch ab) {
  constexpr int N = PL::N;
  constexpr int T = PL::T;
  constexpr int E = PL::E;
  extern __shared__ __align__(16) float2 smem[];
  const int team = threadIdx.x / T;
  const int lt = threadIdx.x - team * T;
  const float2* tw;
  float2* buf = cta_setup<PL>(smem, p.twt, tw, team);
  Xform<PL, false> xf;  // scalar roots: no registers to spare for constant pairs
  xf.init(buf, tw, p.eps, lt);
  int cur_mat = 0;  // matrix whose sign set the transform holds (batch launches)
  for (int64_t base = (int64_t)blockIdx.x * PL::Q; base < p.npairs; base += (int64_t)gridDim.x * PL::Q) {
    const int64_t pair = base + team;
    const bool active = pair < p.npairs;
    int64_t pr = active ? pair : base;
    int mi = 0;
    const bool batched = PL::BATCH && ab.count > 0;
    if (batched) {
      while (mi + 1 < ab.count && pr >= ab.mat[mi + 1].pair0) ++mi;
      pr -= ab.mat[mi].pair0;
      if (mi != cur_mat) {  // uniform per team: Q == 1 whenever T > 32
        xf.set_eps(p.eps + (int64_t)mi * ((N + 31) / 32));
        cur_mat = mi;
      }
    }
    const float* x = batched ? ab.mat[mi].x : p.x;
    float* y = batched ? ab.mat[mi].y : p.y;
    const int64_t m_in = batched ? ab.mat[mi].m : p.m;
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < m_in;
    float2 v[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const int nat = nat_of<N>(lt + j * T);
      v[j] = make_float2(__ldg(&x[colA * N + nat]), hasB ? __ldg(&x[(colA + 1) * N + nat]) : 0.f);
    }
    team_sync<PL>();  // x and y may alias: all loads of this pair precede any store
    xf.apply(v);
    if (active) {
#pragma unroll
      for (int j = 0; j < E; ++j) {
        const int nat = nat_of<N>(lt + j * T);
        y[colA * N + nat] = v[j].x;
        if (hasB) y[(colA + 1) * N + nat] = v[j].y;
      }
    }
    team_sync<PL>();
  }
}

// ---------------------------------------------------------------------------
// kd_reconstruct kernel: W_hat_j = cu_j[code_u] + P(cv_j[code_v])   (App. C)
// ---------------------------------------------------------------------------
struct RecParams {
  int dtype, layout;
  // 1: every output row (KD_VEC_ROWS) starts 16-byte aligned and n * element size is a
  // multiple of 16: W_hat leaves in 16-byte stores
  int vec;
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  int64_t n, m, ld;
  void* out;
  const float2* twt;
  const uint32_t* eps;
  int64_t npairs;
};

// Several matrices of one vector length in one reconstruct launch
// (kd_reconstruct_batch): matrix i owns the global pairs [pair0, pair0 + ceil(m / 2))
// and the sign bits at eps + i * ceil(n / 32); dtype and layout are shared.
struct RecMat {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  void* out;
  int64_t m, ld, pair0;
};
struct RecBatch {
  int count;  // 0: the single matrix of RecParams
  RecMat mat[kMaxBatch];
};

template <class PL>
__global__ void __launch_bounds__(PL::THREADS, PL::MINB) reconstruct_kernel(RecParams p, const __grid_constant__ RecBatch rb) {
  constexpr int N = PL::N;
  constexpr int T = PL::T;
  constexpr int E = PL::E;
  constexpr int WPV = N / 16;
  constexpr int WPT = (WPV + T - 1) / T;  // code words per thread and plane/vector
  extern __shared__ __align__(16) float2 smem[];
  const int team = threadIdx.x / T;
  const int lt = threadIdx.x - team * T;
  const float2* tw;
  float2* buf = cta_setup<PL>(smem, p.twt, tw, team);
  Xform<PL, false> xf;  // scalar roots: no registers to spare for constant pairs
  xf.init(buf, tw, p.eps, lt);
  const bool batched = PL::BATCH && rb.count > 0;
  // global pair -> (matrix, pair within it)
  auto locate = [&](int64_t gp, int& mi, int64_t& pr) {
    mi = 0;
    pr = gp;
    if (batched) {
      while (mi + 1 < rb.count && pr >= rb.mat[mi + 1].pair0) ++mi;
      pr -= rb.mat[mi].pair0;
    }
  };
  // the pair's code words (uA, uB, vA, vB) of this thread, held in registers: the next
  // pair's are loaded while the current pair is transformed
  uint4 cw_next[WPT];
  auto load_codes = [&](int64_t gp) {
    int mi;
    int64_t pr;
    locate(gp, mi, pr);
    const uint32_t* codes_u = batched ? rb.mat[mi].codes_u : p.codes_u;
    const uint32_t* codes_v = batched ? rb.mat[mi].codes_v : p.codes_v;
    const int64_t m_in = batched ? rb.mat[mi].m : p.m;
    const int64_t cA = 2 * pr;
    const int64_t cB = (cA + 1) < m_in ? cA + 1 : cA;
#pragma unroll
    for (int k = 0; k < WPT; ++k) {
      const int w = lt + k * T;
      cw_next[k] = w < WPV ? make_uint4(__ldg(&codes_u[cA * WPV + w]), __ldg(&codes_u[cB * WPV + w]),
                                        __ldg(&codes_v[cA * WPV + w]), __ldg(&codes_v[cB * WPV + w]))
                           : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  const int64_t stride = (int64_t)gridDim.x * PL::Q;
  {
    const int64_t base0 = (int64_t)blockIdx.x * PL::Q;
    if (base0 < p.npairs) load_codes(base0 + team < p.npairs ? base0 + team : base0);
  }
  int cur_mat = 0;  // matrix whose sign set the transform holds (batch launches)
  for (int64_t base = (int64_t)blockIdx.x * PL::Q; base < p.npairs; base += stride) {
    const int64_t pair = base + team;
    const bool active = pair < p.npairs;
    int mi;
    int64_t pr;
    locate(active ? pair : base, mi, pr);
    if (batched && mi != cur_mat) {  // uniform per team: Q == 1 whenever T > 32
      xf.set_eps(p.eps + (int64_t)mi * ((N + 31) / 32));
      cur_mat = mi;
    }
    const float* centres_u = batched ? rb.mat[mi].centres_u : p.centres_u;
    const float* centres_v = batched ? rb.mat[mi].centres_v : p.centres_v;
    const int64_t m_in = batched ? rb.mat[mi].m : p.m;
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < m_in;
    const int64_t colB = hasB ? colA + 1 : colA;
    // the four centre sets of the pair (the same for the whole team: broadcast loads)
    const float4 cuA = __ldg(reinterpret_cast<const float4*>(centres_u) + colA);
    const float4 cuB = __ldg(reinterpret_cast<const float4*>(centres_u) + colB);
    const float4 cvA = __ldg(reinterpret_cast<const float4*>(centres_v) + colA);
    const float4 cvB = __ldg(reinterpret_cast<const float4*>(centres_v) + colB);
    auto pick = [](const float4& c, uint32_t q) -> float {
      const float lo = (q & 1u) ? c.y : c.x;
      const float hi = (q & 1u) ? c.w : c.z;
      return (q & 2u) ? hi : lo;
    };
    // code words of the pair staged in shared memory, word w as (uA, uB, vA, vB)
    uint4* cw = reinterpret_cast<uint4*>(buf);
#pragma unroll
    for (int k = 0; k < WPT; ++k) {
      const int w = lt + k * T;
      if (w < WPV) cw[w] = cw_next[k];
    }
    team_sync<PL>();
    float2 uq[E], vq[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const int nat = nat_of<N>(lt + j * T);
      const uint4 c = cw[nat >> 4];
      const int sh = 2 * (nat & 15);
      uq[j] = make_float2(pick(cuA, (c.x >> sh) & 3u), pick(cuB, (c.y >> sh) & 3u));
      vq[j] = make_float2(pick(cvA, (c.z >> sh) & 3u), pick(cvB, (c.w >> sh) & 3u));
    }
    // the next pair's code words, in flight during this pair's transform
    if (base + stride < p.npairs) load_codes(base + stride + team < p.npairs ? base + stride + team : base + stride);
    team_sync<PL>();  // the transform reuses buf
    xf.apply(vq);
    // W_hat = U_q + P V_q, staged in natural order so the stores are contiguous; one
    // spare slot per 16 keeps the 8-entry runs the 16-byte stores read conflict-free
    auto sp = [](int i) { return i + (i >> 4); };
    static_assert(N + N / 16 <= PL::BUF, "natural-order staging fits the exchange buffer");
    team_sync<PL>();
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const int nat = nat_of<N>(lt + j * T);
      buf[sp(nat)] = make_float2(__fadd_rn(uq[j].x, vq[j].x), __fadd_rn(uq[j].y, vq[j].y));
    }
    team_sync<PL>();
    if (active) {
      void* out = batched ? rb.mat[mi].out : p.out;
      const int64_t ld = batched ? rb.mat[mi].ld : p.ld;
      if (p.vec) {
        // 16-byte chunks of consecutive entries: 8 at 16-bit output, 4 at fp32
        const int per = p.dtype == DT_F32 ? 4 : 8;
        for (int i0 = per * lt; i0 < N; i0 += per * T) {
          float a[8], b[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float2 v = e < per ? buf[sp(i0 + e)] : make_float2(0.f, 0.f);
            a[e] = v.x;
            b[e] = v.y;
          }
          auto pack = [&](const float (&f)[8]) -> uint4 {
            if (p.dtype == DT_F32) {
              return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                                __float_as_uint(f[3]));
            }
            uint32_t w4[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              if (p.dtype == DT_F16) {
                const __half2 t = __floats2half2_rn(f[2 * h], f[2 * h + 1]);
                w4[h] = *reinterpret_cast<const uint32_t*>(&t);
              } else {
                const __nv_bfloat162 t = __floats2bfloat162_rn(f[2 * h], f[2 * h + 1]);
                w4[h] = *reinterpret_cast<const uint32_t*>(&t);
              }
            }
            return make_uint4(w4[0], w4[1], w4[2], w4[3]);
          };
          const int esz = p.dtype == DT_F32 ? 4 : 2;
          char* o = static_cast<char*>(out);
          *reinterpret_cast<uint4*>(o + (colA * ld + i0) * esz) = pack(a);
          if (hasB) *reinterpret_cast<uint4*>(o + (colB * ld + i0) * esz) = pack(b);
        }
      } else {
        for (int i = 2 * lt; i < N; i += 2 * T) {
          const float2 e0 = buf[sp(i)], e1 = buf[sp(i + 1)];   // entries i, i + 1 of (A, B)
          store_elem(out, p.dtype, elem_index(p.layout, colA, i, ld), e0.x);
          store_elem(out, p.dtype, elem_index(p.layout, colA, i + 1, ld), e1.x);
          if (hasB) {
            store_elem(out, p.dtype, elem_index(p.layout, colB, i, ld), e0.y);
            store_elem(out, p.dtype, elem_index(p.layout, colB, i + 1, ld), e1.y);
          }
        }
      }
    }
    team_sync<PL>();
  }
}

}  // namespace kd
