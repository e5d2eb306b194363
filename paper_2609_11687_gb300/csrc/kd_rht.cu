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
//
// Input staging: when every vector start is 16-byte aligned, one thread per CTA
// streams the next blocks into a ring of shared-memory stages with bulk copies
// (cp.async.bulk, completion counted on an mbarrier per stage) while the CTA
// transforms the current ones, so the loads stay in flight through the
// butterflies and barriers.  Every wait on a stage is bounded by a clock limit;
// on expiry the CTA records KD_RHT_ERR_TIMEOUT in the caller's status word, waits
// (bounded again) for the copies it issued, and returns.  Unaligned inputs take
// plain per-thread loads.

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "kashin.h"
#include "kd_bulk.cuh"
#include "kd_math.cuh"

namespace kd {
namespace {

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
  uint32_t* status;  // optional device word: KD_RHT_ERR_* bits
};

constexpr uint32_t kRhtErrTimeout = 1u;           // a stage's bulk copy did not complete in time

KD_HD constexpr int rht_threads(int log_b) { return ((1 << log_b) / 16) > 256 ? ((1 << log_b) / 16) : 256; }
// resident CTAs per SM the register budget is sized for (1024 threads: 64 registers each)
KD_HD constexpr int rht_min_blocks(int log_b) { return 1024 / rht_threads(log_b); }

// Shared-memory slot of block index i in the exchange between passes X and X+1.
// Exchange 0 (16-strided against 16-contiguous accesses): one pad word per 16
// entries.  Exchange X >= 1 (two 16-runs 16^(X+1) apart, or 32 contiguous): 16 pad
// words per 16^(X+1) entries, which moves the second run to the other 16 banks.
// Every warp access of every pass is then free of bank conflicts; both stay
// below B + B/16 slots.
template <int X>
__device__ __forceinline__ int rpad(int i) {
  if constexpr (X == 0) return i + (i >> 4);
  else return i + ((i >> (4 * X + 4)) << 4);
}
template <int X>
KD_HD constexpr int rpad_off(int o) {
  return X == 0 ? o + (o >> 4) : o + ((o >> (4 * X + 4)) << 4);
}

// radix of pass K: four index bits, fewer in the last pass when log2 b % 4 != 0
template <int LOG_B, int K>
KD_HD constexpr int rht_radix() {
  return (LOG_B - 4 * K) >= 4 ? 16 : (1 << (LOG_B - 4 * K));
}

// Block index held in register e of thread t during pass K (bits 4K .. 4K+3 of
// the index vary with e), split as base(t) + off(e).  Pass 0: 16 contiguous
// entries.  Full passes: stride S = 16^K inside a run of 16 S.  A short last pass
// (radix R < 16): 16/R groups of R entries at stride S, consecutive threads on
// consecutive groups.
template <int LOG_B, int K>
__device__ __forceinline__ int rht_base(int t) {
  constexpr int S = 1 << (4 * K);
  constexpr int R = rht_radix<LOG_B, K>();
  if constexpr (K == 0) return 16 * t;
  else if constexpr (R == 16) return (t & (S - 1)) + 16 * S * (t / S);
  else return t;
}

template <int LOG_B, int K>
KD_HD constexpr int rht_off(int e) {
  constexpr int TB = (1 << LOG_B) / 16;
  constexpr int S = 1 << (4 * K);
  constexpr int R = rht_radix<LOG_B, K>();
  return K == 0 ? e : (R == 16 ? S * e : TB * (e / R) + S * (e % R));
}

template <int LOG_B, int K>
__device__ __forceinline__ int rht_index(int t, int e) {
  return rht_base<LOG_B, K>(t) + rht_off<LOG_B, K>(e);
}

// padded slot of rht_index(t, e) in exchange X as rpad<X>(base) + a compile-time
// offset: base and offset never carry into the bits the padding reads
template <int LOG_B, int K, int X, int E>
__device__ __forceinline__ float* slot(float* buf, int pbase) {
  return buf + pbase + rpad_off<X>(rht_off<LOG_B, K>(E));
}

// Walsh-Hadamard butterflies on each group of R consecutive entries of the 16
// held as 8 float2 (entry e in v[e / 2], .x for even e).  Level 1 pairs the two
// halves of one float2 (scalar add and subtract); every level h >= 2 pairs float2
// with float2, one packed FFMA2 (multiplier +-1, so exactly the rounded sum or
// difference) per two butterflies.
template <int R>
__device__ __forceinline__ void fwht_groups(float2 (&v)[8]) {
  if constexpr (R >= 2) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float a = v[k].x, b = v[k].y;
      v[k] = make_float2(__fadd_rn(a, b), __fsub_rn(a, b));
    }
  }
  const float2 one = make_float2(1.f, 1.f), mone = make_float2(-1.f, -1.f);
#pragma unroll
  for (int h = 1; h < R / 2; h <<= 1) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if ((k & h) == 0) {
        const float2 a = v[k], b = v[k + h];
        v[k] = __ffma2_rn(b, one, a);
        v[k + h] = __ffma2_rn(b, mone, a);
      }
    }
  }
}

__device__ __forceinline__ float load_one(const void* x, int dtype, int64_t o) {
  if (dtype == KD_F32) return __ldg(static_cast<const float*>(x) + o);
  if (dtype == KD_F16) return __half2float(__ldg(static_cast<const __half*>(x) + o));
  return __bfloat162float(__ldg(static_cast<const __nv_bfloat16*>(x) + o));
}

// entries 2k, 2k+1 of a run times (s_i * scale): the sign bits 2k, 2k+1 of `bits`
// are moved into the sign of the scale factor, one packed multiply for the pair
template <int K>
__device__ __forceinline__ float2 sign_scale(float2 f, uint32_t bits, uint32_t scale_bits) {
  const float s0 = __uint_as_float(scale_bits | ((bits << (31 - 2 * K)) & 0x80000000u));
  const float s1 = __uint_as_float(scale_bits | ((bits << (30 - 2 * K)) & 0x80000000u));
  return __fmul2_rn(f, make_float2(s0, s1));
}

__device__ __forceinline__ float2 widen2(uint32_t w, int dtype) {
  if (dtype == KD_F16) return __half22float2(*reinterpret_cast<const __half2*>(&w));
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w));
}

// 16 contiguous entries from global memory starting at element offset o
__device__ __forceinline__ void load16(const RhtParams& p, int64_t o, float2 (&v)[8]) {
  if (p.vec_in) {
    if (p.dtype == KD_F32) {
      const float4* q = reinterpret_cast<const float4*>(static_cast<const float*>(p.x) + o);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float4 a = __ldg(q + c);
        v[2 * c] = make_float2(a.x, a.y);
        v[2 * c + 1] = make_float2(a.z, a.w);
      }
    } else {
      const uint4* q = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p.x) + o);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const uint4 a = __ldg(q + c);
        v[4 * c] = widen2(a.x, p.dtype);
        v[4 * c + 1] = widen2(a.y, p.dtype);
        v[4 * c + 2] = widen2(a.z, p.dtype);
        v[4 * c + 3] = widen2(a.w, p.dtype);
      }
    }
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = make_float2(load_one(p.x, p.dtype, o + 2 * k), load_one(p.x, p.dtype, o + 2 * k + 1));
  }
}

// All passes after the load (the first pass's butterflies included), the
// inverse's scale and sign flip, and the store of one unit.  Every thread of the
// CTA calls it (inactive teams too: it holds the CTA's barriers).  The forward
// data arrive already sign-flipped and scaled.  `after_first_barrier` runs once
// per unit right after the first CTA barrier, when every thread has finished
// reading what it loaded the unit from.
//
// UNIT_BAR: the caller passes a CTA barrier at the start of every unit, after the
// previous unit's last reads of buf.  Then the first exchange needs no barrier
// before its writes, and with three or more passes the exchange between passes 0
// and 1 stays inside a half-warp: pass 0's 16 contiguous entries of thread t and
// pass 1's 16-strided group of thread t both lie in the 256-entry run t / 16, which
// threads 16 (t / 16) .. +15 alone write and read (both paddings keep a run inside
// its own slots).  That exchange, and the writes of pass 1 into the next one, then
// need only warp barriers.
template <int LOG_B, bool INV, bool UNIT_BAR = false, class F>
__device__ __forceinline__ void transform_and_store(const RhtParams& p, float2 (&v)[8], float* buf, int t,
                                                    bool active, int64_t j, int64_t off, uint32_t run_bits,
                                                    F&& after_first_barrier) {
  constexpr int NPASS = (LOG_B + 3) / 4;
  constexpr bool LOCAL = UNIT_BAR && NPASS >= 3;
  // the step whose read barrier is the first CTA barrier (forward: the exchange 0 -> 1
  // is warp-local, so the second step's)
  constexpr int FIRST_CTA = (LOCAL && !INV) ? 2 : 1;
  if constexpr (NPASS == 1) {
    __syncthreads();
    after_first_barrier();
  }
  static_for<0, NPASS>([&](auto kk) {
    constexpr int KI = decltype(kk)::value;
    constexpr int K = INV ? NPASS - 1 - KI : KI;
    if constexpr (KI > 0) {
      constexpr int KP = INV ? K + 1 : K - 1;
      constexpr int X = K < KP ? K : KP;  // exchange between passes X and X + 1
      const int wbase = rpad<X>(rht_base<LOG_B, KP>(t));
      const int rbase = rpad<X>(rht_base<LOG_B, K>(t));
      // before the writes: the previous reads of the slots written here are done
      if constexpr (UNIT_BAR && KI == 1) {
        // the unit barrier ordered them
      } else if constexpr (LOCAL && KP == 1) {
        __syncwarp();  // pass 1's slots were read by this half-warp alone
      } else {
        __syncthreads();
      }
      if constexpr (!UNIT_BAR && KI == 1) after_first_barrier();
      static_for<0, 8>([&](auto kk) {
        constexpr int Q = decltype(kk)::value;
        *slot<LOG_B, KP, X, 2 * Q>(buf, wbase) = v[Q].x;
        *slot<LOG_B, KP, X, 2 * Q + 1>(buf, wbase) = v[Q].y;
      });
      if constexpr (LOCAL && X == 0) {
        __syncwarp();
      } else {
        __syncthreads();
      }
      if constexpr (UNIT_BAR && KI == FIRST_CTA) after_first_barrier();
      static_for<0, 8>([&](auto kk) {
        constexpr int Q = decltype(kk)::value;
        v[Q] = make_float2(*slot<LOG_B, K, X, 2 * Q>(buf, rbase), *slot<LOG_B, K, X, 2 * Q + 1>(buf, rbase));
      });
    }
    fwht_groups<rht_radix<LOG_B, K>()>(v);
  });

  if (!active) return;
  if constexpr (!INV) {
    float* yo = p.y + j * p.ldy + off + rht_base<LOG_B, NPASS - 1>(t);
    static_for<0, 8>([&](auto kk) {
      constexpr int Q = decltype(kk)::value;
      yo[rht_off<LOG_B, NPASS - 1>(2 * Q)] = v[Q].x;
      yo[rht_off<LOG_B, NPASS - 1>(2 * Q + 1)] = v[Q].y;
    });
  } else {
    const uint32_t sb = __float_as_uint(p.scale);
    static_for<0, 8>([&](auto kk) {
      constexpr int K = decltype(kk)::value;
      v[K] = sign_scale<K>(v[K], run_bits, sb);
    });
    float* yo = p.y + j * p.ldy + off + 16 * t;
    if (p.vec_out) {
      float4* q = reinterpret_cast<float4*>(yo);
#pragma unroll
      for (int c = 0; c < 4; ++c) q[c] = make_float4(v[2 * c].x, v[2 * c].y, v[2 * c + 1].x, v[2 * c + 1].y);
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        yo[2 * k] = v[k].x;
        yo[2 * k + 1] = v[k].y;
      }
    }
  }
}

// sign bits of the vector, once per CTA (entry j: bit j % 32 of word j / 32)
__device__ __forceinline__ void stage_sign_bits(uint32_t* sbits, int64_t n, uint64_t seed, int nthreads) {
  const int words = (int)((n + 31) / 32);
  for (int wd = threadIdx.x; wd < words; wd += nthreads) {
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; ++bb) {
      const int64_t j = (int64_t)wd * 32 + bb;
      if (j >= n) break;
      bits |= (uint32_t)(splitmix64_mix(seed + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull) >> 63) << bb;
    }
    sbits[wd] = bits;
  }
}

template <int LOG_B, bool INV>
__global__ void __launch_bounds__(rht_threads(LOG_B)) rht_kernel(RhtParams p) {
  constexpr int B = 1 << LOG_B;
  constexpr int TB = B / 16;
  constexpr int THREADS = rht_threads(LOG_B);
  constexpr int TEAMS = THREADS / TB;
  constexpr int NPASS = (LOG_B + 3) / 4;
  constexpr int SLOTS = B + B / 16;  // every rpad<X>(B - 1) < SLOTS
  extern __shared__ __align__(16) float smem[];
  const int words = (int)((p.n + 31) / 32);
  uint32_t* sbits = reinterpret_cast<uint32_t*>(smem);
  const int team = threadIdx.x / TB;
  const int t = threadIdx.x % TB;
  float* buf = smem + ((words + 3) & ~3) + team * SLOTS;

  stage_sign_bits(sbits, p.n, p.seed, THREADS);
  __syncthreads();

  // this team's unit, walked as (vector j, block bi) without a division per unit
  const int64_t nblk = p.n / B;
  const int64_t step = (int64_t)gridDim.x * TEAMS;
  const int64_t dj = step / nblk, db = step - dj * nblk;
  int64_t unit = (int64_t)blockIdx.x * TEAMS + team;
  int64_t jv = unit / nblk, bi = unit - jv * nblk;
  for (int64_t base = (int64_t)blockIdx.x * TEAMS; base < p.units; base += step, unit += step) {
    const bool active = unit < p.units;
    const int64_t j = active ? jv : 0;
    const int64_t off = active ? bi * B : 0;  // block start inside the vector
    jv += dj;
    bi += db;
    if (bi >= nblk) {
      bi -= nblk;
      ++jv;
    }
    float2 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = make_float2(0.f, 0.f);
    // contiguous run of this thread in pass 0: entries off + 16 t .. + 15 (one sign half-word)
    const int64_t run = off + 16 * t;
    const uint32_t run_bits = (sbits[run >> 5] >> (run & 16)) & 0xFFFFu;

    if (active) {
      if constexpr (!INV) {
        load16(p, j * p.ldx + run, v);
        const uint32_t sb = __float_as_uint(p.scale);
        static_for<0, 8>([&](auto kk) {
          constexpr int K = decltype(kk)::value;
          v[K] = sign_scale<K>(v[K], run_bits, sb);
        });
      } else {
        const int64_t o = j * p.ldx + off;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          v[k] = make_float2(load_one(p.x, p.dtype, o + rht_index<LOG_B, NPASS - 1>(t, 2 * k)),
                             load_one(p.x, p.dtype, o + rht_index<LOG_B, NPASS - 1>(t, 2 * k + 1)));
      }
    }

    transform_and_store<LOG_B, INV>(p, v, buf, t, active, j, off, run_bits, [] {});
  }
}

// ---------------------------------------------------------------------------
// Bulk-copy staged variant
// ---------------------------------------------------------------------------
template <int LOG_B>
KD_HD constexpr int rht_stages() { return LOG_B >= 14 ? 2 : 3; }

// Shared memory of the staged kernel:
//   [mbarriers (64 B)][sign bits][STAGES x THREADS*16 entries of the input dtype][exchange]
KD_HD constexpr size_t rht_staged_smem(int log_b, int stages, int64_t n, int esz) {
  return 64 + (((size_t)((n + 31) / 32) * 4 + 15) & ~size_t(15)) +
         (size_t)stages * rht_threads(log_b) * 16 * esz +
         (size_t)(rht_threads(log_b) / ((1 << log_b) / 16)) * ((1 << log_b) + (1 << log_b) / 16) * 4;
}

template <int LOG_B, bool INV>
__global__ void __launch_bounds__(rht_threads(LOG_B), rht_min_blocks(LOG_B)) rht_staged_kernel(RhtParams p) {
  constexpr int B = 1 << LOG_B;
  constexpr int TB = B / 16;
  constexpr int THREADS = rht_threads(LOG_B);
  constexpr int TEAMS = THREADS / TB;
  constexpr int NPASS = (LOG_B + 3) / 4;
  constexpr int SLOTS = B + B / 16;
  constexpr int STAGES = rht_stages<LOG_B>();
  extern __shared__ __align__(128) unsigned char smem_raw[];
  const int esz = p.dtype == KD_F32 ? 4 : 2;
  const int words = (int)((p.n + 31) / 32);
  uint64_t* mbar = reinterpret_cast<uint64_t*>(smem_raw);
  uint32_t* sbits = reinterpret_cast<uint32_t*>(smem_raw + 64);
  unsigned char* stage0 = smem_raw + 64 + (((size_t)words * 4 + 15) & ~size_t(15));
  const size_t stage_bytes = (size_t)THREADS * 16 * esz;  // TEAMS blocks of B entries
  const int tid = threadIdx.x;
  const int team = tid / TB;
  const int t = tid % TB;
  float* buf = reinterpret_cast<float*>(stage0 + STAGES * stage_bytes) + team * SLOTS;

  const int64_t nblk = p.n / B;
  const int64_t per_iter = (int64_t)gridDim.x * TEAMS;
  const int64_t first = (int64_t)blockIdx.x * TEAMS;
  const int64_t n_iter = first < p.units ? (p.units - first + per_iter - 1) / per_iter : 0;

  // producer: the blocks of iteration i into stage s (thread 0 only)
  auto issue = [&](int64_t i, int s) {
    const int64_t base = first + i * per_iter;
    const int64_t left = p.units - base;
    const int cnt = (int)(left < TEAMS ? left : TEAMS);
    const uint32_t blk_bytes = (uint32_t)(B * esz);
    mbar_arrive_expect_tx(&mbar[s], blk_bytes * (uint32_t)cnt);
    // one copy per run of address-contiguous blocks (a whole stage when ldx == n)
    int64_t jj = base / nblk;
    int64_t bi = base - jj * nblk;
    for (int k = 0; k < cnt;) {
      int len = cnt - k;
      if (p.ldx != p.n && (int64_t)len > nblk - bi) len = (int)(nblk - bi);
      const unsigned char* src = static_cast<const unsigned char*>(p.x) + (jj * p.ldx + bi * B) * esz;
      bulk_copy_g2s(stage0 + s * stage_bytes + (size_t)k * blk_bytes, src, blk_bytes * (uint32_t)len, &mbar[s]);
      k += len;
      bi += len;
      while (bi >= nblk) {
        bi -= nblk;
        ++jj;
      }
    }
  };

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&mbar[s], 1);
    mbar_init_fence();
  }
  stage_sign_bits(sbits, p.n, p.seed, THREADS);
  __syncthreads();
  if (tid == 0) {
    for (int64_t i = 0; i < STAGES && i < n_iter; ++i) issue(i, (int)i);
  }

  // this team's unit, walked as (vector j, block bi) without a division per unit
  const int64_t dj = per_iter / nblk, db = per_iter - dj * nblk;
  int64_t unit = first + team;
  int64_t jv = unit / nblk, bi = unit - jv * nblk;
  int s = 0;
  uint32_t parity = 0;
  for (int64_t i = 0; i < n_iter; ++i, unit += per_iter) {
    const bool ok = mbar_wait_bounded(&mbar[s], parity);
    if (__syncthreads_or(!ok)) {
      // a copy did not land in time: report, let this CTA's copies finish, leave
      if (tid == 0) {
        if (p.status) atomicOr(p.status, kRhtErrTimeout);
        const int64_t issued = (i + STAGES < n_iter) ? i + STAGES : n_iter;
        int ks = s;
        uint32_t kp = parity;
        for (int64_t k = i; k < issued; ++k) {
          mbar_wait_bounded(&mbar[ks], kp);
          if (++ks == STAGES) {
            ks = 0;
            kp ^= 1u;
          }
        }
      }
      __syncthreads();
      return;
    }
    const bool active = unit < p.units;
    const int64_t j = active ? jv : 0;
    const int64_t off = active ? bi * B : 0;
    jv += dj;
    bi += db;
    if (bi >= nblk) {
      bi -= nblk;
      ++jv;
    }
    const int64_t run = off + 16 * t;
    const uint32_t run_bits = (sbits[run >> 5] >> (run & 16)) & 0xFFFFu;
    const unsigned char* blk = stage0 + s * stage_bytes + (size_t)team * B * esz;
    float2 v[8];
    if constexpr (!INV) {
      // 16 contiguous 16-bit entries = two 16-byte words at byte 32 tid; lanes
      // 4..7 of each quarter-warp read their two words in the other order so the
      // quarter covers all 32 banks once per access
      const uint4* q = reinterpret_cast<const uint4*>(blk) + 2 * t;
      const int sw = (tid >> 2) & 1;
      const uint4 a = q[sw];
      const uint4 b = q[sw ^ 1];
      const uint4 lo = sw ? b : a;
      const uint4 hi = sw ? a : b;
      const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
      const uint32_t sb = __float_as_uint(p.scale);
      static_for<0, 8>([&](auto kk) {
        constexpr int K = decltype(kk)::value;
        v[K] = sign_scale<K>(widen2(w[K], p.dtype), run_bits, sb);
      });
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        float e2[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int idx = rht_index<LOG_B, NPASS - 1>(t, 2 * k + h);
          if (esz == 4) {
            e2[h] = reinterpret_cast<const float*>(blk)[idx];
          } else if (p.dtype == KD_F16) {
            e2[h] = __half2float(reinterpret_cast<const __half*>(blk)[idx]);
          } else {
            e2[h] = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(blk)[idx]);
          }
        }
        v[k] = make_float2(e2[0], e2[1]);
      }
    }
    const int s_now = s;
    if (++s == STAGES) {
      s = 0;
      parity ^= 1u;
    }
    // after the first barrier every read of stage s_now is done: refill it
    transform_and_store<LOG_B, INV, true>(p, v, buf, t, active, j, off, run_bits, [&] {
      if (tid == 0 && i + STAGES < n_iter) {
        fence_proxy_async_smem();
        issue(i + STAGES, s_now);
      }
    });
  }
}

size_t rht_smem_bytes(int log_b, int64_t n) {
  const int B = 1 << log_b;
  const int teams = rht_threads(log_b) / (B / 16);
  const size_t words = (size_t)((n + 31) / 32);
  return ((words + 3) & ~size_t(3)) * 4 + (size_t)teams * (B + B / 16) * 4;
}

template <class K>
cudaError_t launch_persistent(K kernel, int threads, int teams, size_t smem, const RhtParams& p, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kernel, threads, smem)) != cudaSuccess) return e;
  if (per < 1) return cudaErrorInvalidConfiguration;
  const int64_t want = (p.units + teams - 1) / teams;
  const int64_t cap = (int64_t)per * sms;
  const int grid = (int)(want < cap ? want : cap);
  kernel<<<grid, threads, smem, s>>>(p);
  return cudaGetLastError();
}

template <int LOG_B, bool INV>
cudaError_t launch_rht(const RhtParams& p, cudaStream_t s) {
  constexpr int THREADS = rht_threads(LOG_B);
  constexpr int TEAMS = THREADS / ((1 << LOG_B) / 16);
  const int esz = p.dtype == KD_F32 ? 4 : 2;
  // staged: every block start 16-byte aligned, and not an fp32 forward load (its
  // 64-byte runs per thread would be bank-conflicted in the stage)
  const bool staged = p.vec_in && (INV || esz == 2);
  if (staged)
    return launch_persistent(rht_staged_kernel<LOG_B, INV>, THREADS, TEAMS,
                             rht_staged_smem(LOG_B, rht_stages<LOG_B>(), p.n, esz), p, s);
  return launch_persistent(rht_kernel<LOG_B, INV>, THREADS, TEAMS, rht_smem_bytes(LOG_B, p.n), p, s);
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
                            int inverse, float* y, int64_t ldy, uint32_t* status, void* stream) {
  if (kd_rht_block(n) == 0) return KD_ERR_UNSUPPORTED_N;
  if (m < 0 || ldx < n || ldy < n || (dtype != KD_F32 && dtype != KD_F16 && dtype != KD_BF16) ||
      (inverse != 0 && inverse != 1))
    return KD_ERR_INVALID_ARG;
  if (m == 0) return KD_OK;
  if (!x || !y) return KD_ERR_INVALID_ARG;
  // elements are read and written at least one at a time: aligned to their size
  if (reinterpret_cast<uintptr_t>(x) % (dtype == KD_F32 ? 4 : 2) != 0 || reinterpret_cast<uintptr_t>(y) % 4 != 0 ||
      reinterpret_cast<uintptr_t>(status) % 4 != 0)
    return KD_ERR_INVALID_ARG;
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
  p.status = status;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const cudaError_t e = inverse ? kd::dispatch_rht<true>(log_b, p, s) : kd::dispatch_rht<false>(log_b, p, s);
  return e == cudaSuccess ? KD_OK : KD_ERR_CUDA;
}
