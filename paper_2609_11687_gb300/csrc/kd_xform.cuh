// The sign-randomised DCT operator P on a pair of vectors held by one team
// (Sec. 3.1: P z = IDCT(eps * DCT(z)); Alg. 1 applies it twice per block).
//
// With both vectors in Makhoul's even/odd order and packed as one complex
// vector z (vector 2j in the real part, 2j+1 in the imaginary part),
//     P' z = IDFT( M( DFT(z) ) ),
//     M: Z'_k = e+_k Z_k + e-_k exp(i pi k/N) Z_{N-k},  e+-_k = (eps_k +- eps_{N-k}) / 2,
// (the DCT's per-coefficient scale cancels between DCT and IDCT).  Exactly one of
// e+_k, e-_k is non-zero: either Z'_k = eps_k Z_k, or Z'_k = eps_k exp(i pi k/N) Z_{N-k}.
//
// DFT: in-place mixed-radix decimation in frequency over shared memory (natural
// order in, digit-reversed out); IDFT: the mirror passes (digit-reversed in,
// natural out).  Pass 0 works on the thread's own registers (the vector stays
// register-resident between transforms).  Inter-pass twiddles come from a table
// laid out in the order the threads read it (conflict-free in shared memory).
//
// M runs in one of two forms:
//  * paired (last radix == first radix, one last-pass group per thread): the
//    thread owning frequency group K and the one owning N/R0 - K sit at lanes
//    l and l ^ H of one warp; each gets its partner's values by shuffle and
//    applies M in registers between the last forward and first inverse pass;
//  * slot order (all other plans): each thread reads its own slots and their
//    partners' from shared memory (conflict-free: partners of consecutive slots
//    are consecutive slots in reverse), then writes its own.
// All per-frequency quantities (partner slot, eps bits, exp(i pi k/N)) reduce to
// a few per-thread constants computed once per CTA.
#pragma once

#include <type_traits>

#include "kd_math.cuh"

namespace kd {

enum { UREG = 0, UGMEM = 1, USMEM = 2 };

// Padded slot: one spare float2 per 16 and per 256 slots, so that accesses with
// lane strides 1, 16 and 256 fall in distinct bank pairs.
KD_HD constexpr int pad(int i) { return i + (i >> 4) + (i >> 8); }

// True when pad(base + j*stride) == pad(base) + pad(j*stride) for every base the
// access pattern produces (checked exhaustively at compile time), so element
// addresses are a per-thread padded base plus compile-time offsets.
KD_HD constexpr bool sep_strided(int nbase, int base_mul, int base_add_max, int count, int stride) {
  // bases: b = q * base_mul + a, q < nbase, a < base_add_max
  for (int q = 0; q < nbase; ++q)
    for (int a = 0; a < base_add_max; ++a) {
      const int b = q * base_mul + a;
      for (int j = 0; j < count; ++j)
        if (pad(b + j * stride) != pad(b) + pad(j * stride)) return false;
    }
  return true;
}

// Twiddle read that the compiler may not hoist out of the block loop: every
// thread's twiddles are loop-invariant, and keeping them all in registers would
// spill.  SMEM selects a shared-memory (else read-only global) load.
template <bool SMEM>
__device__ __forceinline__ float2 ld_tw(const float2* p) {
  float2 v;
  if constexpr (SMEM) {
    const unsigned a = (unsigned)__cvta_generic_to_shared(p);
    asm volatile("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a));
  } else {
    asm volatile("ld.global.nc.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "l"(p));
  }
  return v;
}



// Two consecutive table entries (16-byte aligned) in one 128-bit load.
template <bool SMEM>
__device__ __forceinline__ float4 ld_tw4(const float2* p) {
  float4 v;
  if constexpr (SMEM) {
    const unsigned a = (unsigned)__cvta_generic_to_shared(p);
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
  } else {
    asm volatile("ld.global.nc.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
  }
  return v;
}

// Plans that apply the DFTs' constant roots in packed FP32x2 form (kd_math.cuh
// mul_root): opted in per plan (kd_plans.cuh) where the registers allow it and it
// measured faster.
template <class PL>
struct PackedRoots {
  static constexpr bool value = false;
};

template <int N_, int T_, int Q_, int UMODE_, int MINB_, int... Rs>
struct Plan {
  static constexpr int N = N_;
  static constexpr int T = T_;
  static constexpr int Q = Q_;
  static constexpr int UMODE = UMODE_;
  static constexpr int MINB = MINB_;  // CTAs per SM the register budget must allow
  static constexpr int NP = sizeof...(Rs);
  static constexpr int Rv[NP] = {Rs...};
  static constexpr int E = Rv[0];
  static constexpr int RL = Rv[NP - 1];
  static constexpr int THREADS = T * Q;
  // batched launches (kd_decompose_batch) compiled in: the lengths whose matrices can
  // be too small to fill the GPU alone (longer ones run one launch per matrix)
  static constexpr bool BATCH = N_ <= 8192;
  static constexpr int NW = (T + 31) / 32;  // warps per team
  static constexpr int BUF = (N + N / 16 + N / 256 + 8 + 15) / 16 * 16;  // padded float2 slots per team
  // float2 reduction slots per team: ping-pong partials of team_sum, or the
  // 16-value reduction of the k-means refinement (16 (NW + 1) floats = 8 (NW + 1) float2)
  static constexpr int RED = (4 * NW > 8 * (NW + 1)) ? 4 * NW : 8 * (NW + 1);
  static constexpr int USL = (UMODE_ == 2) ? N : 0;            // float2 slots of u per team (shared)
  static constexpr int MBS = 2;  // float2 slots holding the team's mbarrier (bulk-copy staging)
  // M in registers: one last-pass group per thread, partner at lane ^ HALF
  static constexpr bool PAIRED = (RL == E) && (N / RL == T);
  static constexpr int HALF = (T < 32 ? T : 32) / 2;

  KD_HD static constexpr int R(int i) { return Rv[i]; }
  KD_HD static constexpr int B(int i) {  // sub-transform length entering pass i
    int b = N;
    for (int j = 0; j < i; ++j) b /= Rv[j];
    return b;
  }
  KD_HD static constexpr int S(int i) { return B(i) / Rv[i]; }  // stride of pass i's digit
  // access-ordered twiddle table: pass 0 [j][t] (N entries), pass i>=1 [j][np] (B(i) entries)
  KD_HD static constexpr int tw_off(int i) {
    int o = 0;
    for (int j = 0; j < i; ++j) o += B(j);
    return o;
  }
  static constexpr int TWN = tw_off(NP - 1);

  // stage the table in shared memory when MINB CTAs per SM still fit
  static constexpr int TEAM = BUF + RED + USL + MBS;  // float2 slots of shared memory per team
  static constexpr bool TW_SMEM = (size_t)TWN * 8 + (size_t)Q * TEAM * 8 <= (size_t)(227 * 1024) / MINB - 1024;
  static constexpr size_t SMEM_TW = TW_SMEM ? (size_t)TWN * sizeof(float2) : 0;
  // paired twiddle layout (table staged in shared memory, every twiddled pass of even
  // radix): rows 2a and 2a + 1 of a pass table are interleaved per column
  // ([a][column][2]), so one 128-bit load fetches a column's twiddles of both rows
  KD_HD static constexpr bool tw2_ok() {
    for (int i = 0; i < NP - 1; ++i)
      if (Rv[i] % 2 != 0) return false;
    return TW_SMEM;
  }
  static constexpr bool TW2 = tw2_ok();
  // table position of row j, column c of pass i (rows of length L)
  KD_HD static constexpr int tw_pos(int i, int L, int j, int c) {
    return tw_off(i) + (TW2 ? (j / 2) * 2 * L + 2 * c + (j % 2) : j * L + c);
  }
  static constexpr size_t SMEM = SMEM_TW + (size_t)Q * TEAM * sizeof(float2);

  // pass 0 / inverse pass 0 and slot-order M: slots base + j*T with base < T
  static constexpr bool SEP0 = sep_strided(1, 0, T, E, T);
  // paired last pass: group of frequencies K + (N/RL) j sits at slot_low(K) + j
  KD_HD static constexpr int slot_low_c(int K) {
    int s = 0;
    for (int i = 0; i < NP - 1; ++i) {
      s += (K % Rv[i]) * (B(i) / Rv[i]);
      K /= Rv[i];
    }
    return s;
  }
  KD_HD static constexpr bool sep_last() {
    for (int K = 0; K < N / RL; ++K)
      for (int j = 0; j < RL; ++j)
        if (pad(slot_low_c(K) + j) != pad(slot_low_c(K)) + pad(j)) return false;
    return true;
  }
  KD_HD static constexpr bool sep_pass(int i) {
    // groups of pass i: base = blk * B(i) + np (blk < N/B(i), np < S(i)), stride S(i)
    return sep_strided(N / B(i), B(i), S(i), Rv[i], S(i));
  }
  KD_HD static constexpr bool valid() {
    int p = 1;
    for (int i = 0; i < NP; ++i) p *= Rv[i];
    return p == N && N == T * E && (N % 16 == 0) && NP >= 2 &&
           (T <= 32 ? (32 % T == 0) : (T % 32 == 0 && Q == 1));
  }
  static_assert(valid(), "inconsistent plan");
};

template <class PL>
__device__ __forceinline__ void team_sync() {
  if constexpr (PL::T <= 32) {
    __syncwarp();
  } else {
    __syncthreads();
  }
}

__device__ __forceinline__ bool eps_neg(const uint32_t* __restrict__ eb, int k) {
  return (__ldg(&eb[k >> 5]) >> (k & 31)) & 1u;
}

// exp(i pi a / b) in double, rounded
__device__ __forceinline__ float2 expi_pi(long long a, long long b) {
  double s, c;
  sincospi((double)a / (double)b, &s, &c);
  return make_float2((float)c, (float)s);
}

// Digit-reversed slot of X over passes 1..NP-1: X = sum x_i prod_{1<=j<i} R_j  ->  sum x_i S_i
template <class PL>
__device__ __forceinline__ int slot_rest(int X) {
  int s = 0;
  static_for<1, PL::NP>([&](auto ii) {
    constexpr int I = decltype(ii)::value;
    const int xi = X % PL::R(I);
    X /= PL::R(I);
    s += xi * PL::S(I);
  });
  return s;
}

// Slot of the first element of the last-pass group that holds frequencies
// K + (N/RL) j: the digits of K over passes 0..NP-2 placed at their strides.
template <class PL>
__device__ __forceinline__ int slot_low(int K) {
  int s = 0;
  static_for<0, PL::NP - 1>([&](auto ii) {
    constexpr int I = decltype(ii)::value;
    const int ki = K % PL::R(I);
    K /= PL::R(I);
    s += ki * PL::S(I);
  });
  return s;
}

// Inverse of slot_rest for a slot below T (digits of passes 1..NP-1).
template <class PL>
__device__ __forceinline__ int rest_of_slot(int s) {
  int X = 0, mul = 1;
  static_for<1, PL::NP>([&](auto ii) {
    constexpr int I = decltype(ii)::value;
    const int xi = (s / PL::S(I)) % PL::R(I);
    X += xi * mul;
    mul *= PL::R(I);
  });
  return X;
}

// ---------------------------------------------------------------------------
// PKX: packed constant roots in the DFTs (the plan's choice by default)
template <class PL, bool PKX = PackedRoots<PL>::value>
struct Xform {
  static constexpr int N = PL::N, T = PL::T, E = PL::E, NP = PL::NP;
  float2* buf;                 // team's padded exchange buffer (shared)
  const float2* tw;            // access-ordered twiddles (shared or global)
  int lt;
  float2 cw;                   // M twiddle base
  using Mask = typename std::conditional<(E > 32), uint64_t, uint32_t>::type;
  Mask ek, em;                 // eps_k < 0 / eps_{-k} < 0 for each owned frequency (bit index)
  Mask dm;                     // ek ^ em: frequencies whose M takes the partner value
  static constexpr float kInvN = 1.0f / (float)N;
  static constexpr bool PK = PKX;
  // Warp-local middle passes (16 x 16 x 16 with 256 threads): after pass 0 the
  // vector falls into 16 blocks of 256 slots (one per pass-0 output digit b), and the
  // M partner of every last-pass group of block b lies in block 16 - b (blocks 0 and
  // 8 pair with themselves).  Warp w owns blocks {w, 16 - w} ({0, 8} for w = 0) for
  // pass 1, the last pass and the inverse pass 1, so only the exchanges into and
  // out of pass 0 cross warps: two CTA barriers per P instead of four.
  static constexpr bool WL = NP == 3 && PL::PAIRED && E == 16 && PL::R(1) == 16 && PL::RL == 16 && T == 256;
  // Slot-order plans of shape R0 x 16 x 16 (n = 11008): the 16 pass-1 groups and the
  // 16 last-pass groups of a 256-slot block are taken by the same 16 consecutive
  // threads (group g goes to thread g mod T in both passes), so the exchange between
  // passes 1 and 2, forward and inverse, stays inside a half-warp.
  static constexpr bool L12 = NP == 3 && !PL::PAIRED && PL::R(1) == 16 && PL::S(1) == 16 && PL::RL == 16 &&
                              T % 16 == 0;
  // Warp-local units for an odd first radix (n = 11008 = 43 x 16 x 16): after pass 0
  // the vector falls into E blocks of 256 slots, and the M partner of every frequency
  // of block b lies in block E - b (block 0 pairs with itself).  Unit 0 is block 0,
  // unit u >= 1 the blocks u and E - u; warp w takes units w, w + NW, ...  In a unit,
  // lane l < 16 takes group i = l of the first block and lane l >= 16 group 31 - l of
  // the second, in pass 1, the last pass and their inverses; M then pairs lane l with
  // lane l ^ 16 (register 15 - k2) in registers, as the paired plans do (unit 0: lane l
  // with lane 16 - l, lane 0 with itself).  Only the exchanges into pass 1 and out of
  // the inverse pass 1 cross warps: two CTA barriers per P instead of five.
  static constexpr bool WLU = NP == 3 && !PL::PAIRED && (E % 2 == 1) && PL::R(1) == 16 && PL::RL == 16 &&
                              PL::S(1) == 16 && T == 256;
  static constexpr int NU = (E + 1) / 2;  // units
  static constexpr int NWT = T >= 32 ? T / 32 : 1;  // warps of the team
  static constexpr int UPW = (NU + NWT - 1) / NWT;  // units per warp, at most
  float2 ucw[WLU ? UPW : 1];              // per unit: exp(i pi K / N) of the lane's group K
  uint32_t umk[WLU ? UPW : 1];            // per unit: eps_k < 0 bits (low 16), eps_{N-k} < 0 bits (high 16)
  int g1;                      // warp-local: this thread's pass-1 group
  int p0, p1;                  // slot-order M: partner slot constants
  int pb0;                     // pad(lt): base of the pass-0 slots lt + j T
  int pbp0, pbp1;              // slot-order M: pad(p0), pad(p1)
  int kgrp;                    // paired M: own frequency group (k = kgrp + (N/RL) j)
  int lbase;                   // paired M: slot of that group's first element
  int self;                    // paired M: 0 regular, 1 group 0, 2 group N/(2 R0)

  __device__ __forceinline__ void init(float2* b, const float2* t, const uint32_t* __restrict__ eb, int lane_t) {
    buf = b;
    tw = t;
    lt = lane_t;
    pb0 = pad(lt);
    if constexpr (PL::PAIRED) {
      constexpr int H = PL::HALF;
      constexpr int L = T;
      const int w = lt / (2 * H), l = lt % (2 * H), h = l / H, i = l % H;
      // partner groups K and T - K at lanes l and l ^ H (K = 0 and T/2 pair with
      // themselves, at lanes 0 and H of warp 0)
      int bb;
      if constexpr (WL) {
        // last-pass group K = b + 16 k1 (b: pass-0 digit = block, k1: pass-1 digit);
        // warp w >= 1 holds blocks w and 16 - w, warp 0 blocks 0 and 8
        bb = (w == 0) ? (i < 8 ? 16 * i : 16 * i - 120) : w + 16 * i;
        g1 = ((w == 0) ? 8 * h : (h ? 16 - w : w)) * 16 + i;
      } else {
        bb = H * w + i;
        g1 = 0;
      }
      kgrp = h ? (bb ? L - bb : L / 2) : bb;
      self = (bb == 0) ? (h == 0 ? 1 : 2) : 0;
      lbase = slot_low<PL>(kgrp);
      cw = expi_pi(kgrp, N);
      p0 = p1 = pbp0 = pbp1 = 0;
    } else if constexpr (WLU) {
#pragma unroll
      for (int q = 0; q < UPW; ++q) {
        int b, i;
        bool act;
        unit_of(q, b, i, act);
        ucw[q] = expi_pi(b + (long long)E * i, N);
      }
      cw = make_float2(0.f, 0.f);
      p0 = p1 = pbp0 = pbp1 = kgrp = self = lbase = g1 = 0;
    } else {
      const int Kp = rest_of_slot<PL>(lt);
      p0 = slot_rest<PL>((T - Kp) % T);
      p1 = slot_rest<PL>(T - 1 - Kp);
      pbp0 = pad(p0);
      pbp1 = pad(p1);
      cw = expi_pi((long long)E * Kp, N);
      kgrp = self = lbase = g1 = 0;
    }
    set_eps(eb);
  }

  // warp-local units: this lane's block b and group index i in its unit q (act false
  // for the idle half of unit 0 and for units past the last)
  __device__ __forceinline__ void unit_of(int q, int& b, int& i, bool& act) const {
    const int w = lt >> 5, l = lt & 31;
    const int u = w + NWT * q;
    if (u == 0) {
      b = 0;
      i = l & 15;
      act = l < 16;
    } else {
      b = l < 16 ? u : E - u;
      i = l < 16 ? l : 31 - l;
      act = u < NU;
    }
  }

  // the sign set's bits at this thread's frequencies (and their mirrors)
  __device__ __forceinline__ void set_eps(const uint32_t* __restrict__ eb) {
    ek = em = 0;
    if constexpr (PL::PAIRED) {
#pragma unroll
      for (int kp = 0; kp < E; ++kp) {
        const int k = kgrp + T * kp;
        ek |= (Mask)eps_neg(eb, k) << kp;
        em |= (Mask)eps_neg(eb, (N - k) % N) << kp;
      }
    } else if constexpr (WLU) {
#pragma unroll
      for (int q = 0; q < UPW; ++q) {
        int b, i;
        bool act;
        unit_of(q, b, i, act);
        uint32_t m = 0;
        if (b + E * i < N) {
          for (int kp = 0; kp < 16; ++kp) {
            const int k = b + E * i + (N / 16) * kp;
            m |= (uint32_t)eps_neg(eb, k) << kp;
            m |= (uint32_t)eps_neg(eb, (N - k) % N) << (16 + kp);
          }
        }
        umk[q] = m;
      }
    } else {
      const int Kp = rest_of_slot<PL>(lt);
#pragma unroll
      for (int r = 0; r < E; ++r) {
        const int k = r + E * Kp;
        ek |= (Mask)eps_neg(eb, k) << r;
        em |= (Mask)eps_neg(eb, (N - k) % N) << r;
      }
    }
    dm = ek ^ em;
  }

  // padded address of pass-0 slot lt + j T (base + compile-time offset when separable)
  template <int J>
  __device__ __forceinline__ int a0() const {
    if constexpr (PL::SEP0) return pb0 + pad(J * T);
    else return pad(lt + J * T);
  }

  // M on one frequency: own value a, partner value b; returns Z'_k (1/N folded in).
  // eps_k == eps_{N-k}: Z'_k = eps_k a / N;  otherwise Z'_k = eps_k exp(i pi k/N) b / N.
  template <long long RNUM, long long RDEN, int BIT>
  __device__ __forceinline__ float2 mfreq(float2 a, float2 b) const {
    // exp(i pi k / N) = cw * exp(i pi RNUM / RDEN)
    const float2 wk = mul_root<+1, RNUM, 2 * RDEN, PK>(cw);
    const float2 t = cmul(b, wk);
    const bool diff = (dm >> BIT) & 1u;
    const float2 sel = diff ? t : a;
    // +-1/N with the sign of eps_k taken straight from its bit
    const uint32_t sgn = (uint32_t)((ek >> BIT) & 1u) << 31;
    const float f = __uint_as_float(__float_as_uint(kInvN) | sgn);
    return __fmul2_rn(sel, make_float2(f, f));
  }

  // mfreq with explicit per-group constants (warp-local units): c = exp(i pi K / N),
  // m = the eps bits of the group's frequencies (low 16) and of their mirrors (high 16)
  template <int KP>
  __device__ __forceinline__ float2 mfreq_u(float2 a, float2 b, float2 c, uint32_t m) const {
    const float2 wk = mul_root<+1, KP, 2 * 16, PK>(c);
    const float2 t = cmul(b, wk);
    const bool diff = ((m ^ (m >> 16)) >> KP) & 1u;
    const float2 sel = diff ? t : a;
    const uint32_t sgn = ((m >> KP) & 1u) << 31;
    const float f = __uint_as_float(__float_as_uint(kInvN) | sgn);
    return __fmul2_rn(sel, make_float2(f, f));
  }

  // v[j] *= W (DIR < 0) or conj(W) (DIR > 0) for j = 1 .. R-1, W = the entry (j, c)
  // of pass I's twiddle table (rows of length L)
  template <int I, int L, int R, int DIR>
  __device__ __forceinline__ void twiddle(float2 (&v)[R], int c) const {
    auto mul = [](float2 a, float2 w) { return DIR < 0 ? cmul(a, w) : cmulc(a, w); };
    if constexpr (PL::TW2) {
      static_assert(R % 2 == 0, "paired twiddles need an even radix");
      static_for<0, R / 2>([&](auto pc) {
        constexpr int P = decltype(pc)::value;
        constexpr int O = PL::tw_pos(I, L, 2 * P, 0);
        const float2* q = tw + O + 2 * c;
        if constexpr (P == 0) {
          v[1] = mul(v[1], ld_tw<PL::TW_SMEM>(q + 1));
        } else {
          const float4 w = ld_tw4<PL::TW_SMEM>(q);
          v[2 * P] = mul(v[2 * P], make_float2(w.x, w.y));
          v[2 * P + 1] = mul(v[2 * P + 1], make_float2(w.z, w.w));
        }
      });
    } else {
      constexpr int O = PL::tw_off(I);
#pragma unroll
      for (int j = 1; j < R; ++j) v[j] = mul(v[j], ld_tw<PL::TW_SMEM>(tw + O + j * L + c));
    }
  }

  // forward pass 0 from registers
  __device__ __forceinline__ void fwd0(float2 (&v)[E]) {
    if constexpr (kd_is_big_prime<E>()) {
      static_assert(!PL::TW2, "row-major pass-0 table");
      dft_prime_pass<E, -1>([&](auto jc) { return v[decltype(jc)::value]; },
                              [&](auto kc, float2 x) {
                                constexpr int K = decltype(kc)::value;
                                if constexpr (K > 0) x = cmul(x, ld_tw<PL::TW_SMEM>(tw + K * T + lt));  // row-major: E odd
                                buf[a0<K>()] = x;
                              });
    } else {
      Dft<E, -1, PK>::run(v);
      twiddle<0, T, E, -1>(v, lt);
      static_for<0, E>([&](auto jc) { buf[a0<decltype(jc)::value>()] = v[decltype(jc)::value]; });
    }
  }

  // inverse pass 0 into registers
  __device__ __forceinline__ void inv0(float2 (&v)[E]) {
    if constexpr (kd_is_big_prime<E>()) {
      // outputs go back to the thread's own slots (already read), then to registers
      dft_prime_pass<E, +1>(
          [&](auto jc) {
            constexpr int J = decltype(jc)::value;
            float2 x = buf[a0<J>()];
            if constexpr (J > 0) x = cmulc(x, ld_tw<PL::TW_SMEM>(tw + J * T + lt));  // row-major: E odd
            return x;
          },
          [&](auto kc, float2 x) { buf[a0<decltype(kc)::value>()] = x; });
      static_for<0, E>([&](auto jc) { v[decltype(jc)::value] = buf[a0<decltype(jc)::value>()]; });
    } else {
      static_for<0, E>([&](auto jc) { v[decltype(jc)::value] = buf[a0<decltype(jc)::value>()]; });
      twiddle<0, T, E, +1>(v, lt);
      Dft<E, +1, PK>::run(v);
    }
  }

  // shared-memory pass I (1 <= I <= NP-1), forward (DIR < 0) or inverse
  template <int I, int DIR>
  __device__ __forceinline__ void pass() {
    constexpr int R = PL::R(I);
    constexpr int Bk = PL::B(I);
    constexpr int S = Bk / R;
    constexpr int G = N / R;
    constexpr bool LAST = (I == NP - 1);
    constexpr int OFF = PL::tw_off(I);
    constexpr bool SEP = PL::sep_pass(I);
    // warp-local plans: pass 1 has one group per thread, in one of the warp's blocks
    constexpr bool ONE = WL && I == 1;
    for (int g = ONE ? g1 : lt; ONE || g < G; g += T) {
      pass_group<I, DIR>(g);
      if constexpr (ONE) break;
    }
  }

  // one group g of pass I: blk = g / S, np = g % S, slots blk B(I) + np + j S
  template <int I, int DIR>
  __device__ __forceinline__ void pass_group(int g) {
    constexpr int R = PL::R(I);
    constexpr int Bk = PL::B(I);
    constexpr int S = Bk / R;
    constexpr bool LAST = (I == NP - 1);
    constexpr bool SEP = PL::sep_pass(I);
    const int blk = g / S;
    const int np = g - blk * S;
    const int base = blk * Bk + np;
    const int pb = pad(base);
    auto addr = [&](int j) { return SEP ? pb + pad(j * S) : pad(base + j * S); };
    float2 v[R];
#pragma unroll
    for (int j = 0; j < R; ++j) v[j] = buf[addr(j)];
    if constexpr (DIR < 0) {
      Dft<R, -1, PK>::run(v);
      if constexpr (!LAST) twiddle<I, S, R, -1>(v, np);
    } else {
      if constexpr (!LAST) twiddle<I, S, R, +1>(v, np);
      Dft<R, +1, PK>::run(v);
    }
#pragma unroll
    for (int j = 0; j < R; ++j) buf[addr(j)] = v[j];
  }

  // warp-local unit q: pass 1, the last pass with M in registers, their inverses
  __device__ __forceinline__ void unit(int q) {
    constexpr int R = 16;
    int b, i;
    bool act;
    unit_of(q, b, i, act);
    const bool selfu = (lt >> 5) == 0 && q == 0;  // unit 0: block 0 pairs with itself
    // this unit's constants (selects, not an indexed array: stays in registers)
    float2 c = ucw[0];
    uint32_t m = umk[0];
#pragma unroll
    for (int qq = 1; qq < UPW; ++qq)
      if (q == qq) {
        c = ucw[qq];
        m = umk[qq];
      }
    if (act) pass_group<1, -1>(16 * b + i);
    __syncwarp();
    // last pass: the group (b, k1 = i) at slots 256 b + 16 i + k2, frequencies
    // b + E i + (N / 16) k2
    constexpr bool SEP = PL::sep_pass(2);
    const int base = PL::B(1) * b + R * i;
    const int pb = pad(base);
    auto addr = [&](int j) { return SEP ? pb + pad(j) : pad(base + j); };
    float2 v[R];
#pragma unroll
    for (int j = 0; j < R; ++j) v[j] = act ? buf[addr(j)] : make_float2(0.f, 0.f);
    Dft<R, -1, PK>::run(v);
    auto body = [&](auto selfc) {
      constexpr bool SELF = decltype(selfc)::value;
      const int src = SELF ? (((lt & 31) < 16) ? ((16 - (lt & 31)) & 15) : (lt & 31)) : ((lt & 31) ^ 16);
      const bool own = SELF && (lt & 31) == 0;  // frequency group 0: partners in its own registers
      if constexpr (SELF) {
        if (own) {
#pragma unroll
          for (int j = 0; j < R; ++j) buf[addr(j)] = v[j];
        }
      }
      static_for<0, R / 2>([&](auto kk) {
        constexpr int K1 = decltype(kk)::value;
        constexpr int K2 = R - 1 - K1;
        const float2 s1 = v[K2], s2 = v[K1];
        float2 q1, q2;
        q1.x = __shfl_sync(0xffffffffu, s1.x, src);
        q1.y = __shfl_sync(0xffffffffu, s1.y, src);
        q2.x = __shfl_sync(0xffffffffu, s2.x, src);
        q2.y = __shfl_sync(0xffffffffu, s2.y, src);
        if constexpr (SELF) {
          if (own) {
            q1 = buf[addr((R - K1) % R)];
            q2 = buf[addr((R - K2) % R)];
          }
        }
        const float2 o1 = mfreq_u<K1>(s2, q1, c, m);
        const float2 o2 = mfreq_u<K2>(s1, q2, c, m);
        v[K1] = o1;
        v[K2] = o2;
      });
    };
    if (selfu) {
      body(std::true_type{});
    } else {
      body(std::false_type{});
    }
    Dft<R, +1, PK>::run(v);
    if (act) {
#pragma unroll
      for (int j = 0; j < R; ++j) buf[addr(j)] = v[j];
    }
    __syncwarp();
    if (act) pass_group<1, +1>(16 * b + i);
  }

  // paired last pass: forward DFT of own group, M with the partner lane, inverse DFT.
  // M runs in place, two mirrored indices (KP, R-1-KP) at a time: the partner lane's
  // value for index KP is its v[R-1-KP], so each step exchanges both of a mirrored
  // pair's sources before overwriting them (no second array of R values is live).
  __device__ __forceinline__ void last_paired() {
    constexpr int R = PL::RL;
    constexpr int H = PL::HALF;
    constexpr bool SEP = PL::sep_last();
    const int base = lbase;
    const int pb = pad(base);
    auto addr = [&](int j) { return SEP ? pb + pad(j) : pad(base + j); };
    float2 v[R];
#pragma unroll
    for (int j = 0; j < R; ++j) v[j] = buf[addr(j)];
    Dft<R, -1, PK>::run(v);
    // Only the warp holding groups 0 and N/(2 RL) (self-paired) needs the local-value
    // selects; every other warp takes the shuffle-only path (warp-uniform branch).
    // Group 0 pairs index KP with its own (R - KP) % R, which the in-place order may
    // already have overwritten: its lane keeps the transformed values in its own slots.
    auto body = [&](auto slowc) {
      constexpr bool SLOW = decltype(slowc)::value;
      if constexpr (SLOW) {
        if (self == 1) {
#pragma unroll
          for (int j = 0; j < R; ++j) buf[addr(j)] = v[j];
        }
      }
      static_for<0, R / 2>([&](auto kk) {
        constexpr int K1 = decltype(kk)::value;
        constexpr int K2 = R - 1 - K1;
        const float2 s1 = v[K2], s2 = v[K1];
        float2 q1, q2;
        q1.x = __shfl_xor_sync(0xffffffffu, s1.x, H);
        q1.y = __shfl_xor_sync(0xffffffffu, s1.y, H);
        q2.x = __shfl_xor_sync(0xffffffffu, s2.x, H);
        q2.y = __shfl_xor_sync(0xffffffffu, s2.y, H);
        if constexpr (SLOW) {
          if (self == 1) {
            q1 = buf[addr((R - K1) % R)];
            q2 = buf[addr((R - K2) % R)];
          } else if (self == 2) {
            q1 = s1;
            q2 = s2;
          }
        }
        // k = K + (N/R) KP: exp(i pi k/N) = exp(i pi K/N) exp(i pi KP/R)
        const float2 o1 = mfreq<K1, R, K1>(s2, q1);
        const float2 o2 = mfreq<K2, R, K2>(s1, q2);
        v[K1] = o1;
        v[K2] = o2;
      });
    };
    if (__any_sync(0xffffffffu, self != 0)) {
      body(std::true_type{});
    } else {
      body(std::false_type{});
    }
    Dft<R, +1, PK>::run(v);
#pragma unroll
    for (int j = 0; j < R; ++j) buf[addr(j)] = v[j];
  }

  // slot-order M (own slots lt + T r, partners from constants); v is scratch
  __device__ __forceinline__ void middle_slots(float2 (&v)[E]) {
    static_for<0, E>([&](auto rr) {
      constexpr int RR = decltype(rr)::value;
      int pa;
      if constexpr (RR == 0) pa = pbp0;
      else if constexpr (PL::SEP0) pa = pbp1 + pad((E - RR) * T);
      else pa = pad((E - RR) * T + p1);
      // k = RR + E K': exp(i pi k/N) = exp(i pi E K'/N) exp(i pi RR/N)
      v[RR] = mfreq<RR, N, RR>(buf[a0<RR>()], buf[pa]);
    });
    team_sync<PL>();
    static_for<0, E>([&](auto rr) { buf[a0<decltype(rr)::value>()] = v[decltype(rr)::value]; });
  }

  // y = P' v
  __device__ __forceinline__ void apply(float2 (&v)[E]) {
    if constexpr (T <= 32) team_sync<PL>();  // earlier readers of buf are done
    fwd0(v);
    team_sync<PL>();
    if constexpr (PL::PAIRED) {
      static_for<1, NP - 1>([&](auto ii) {
        pass<decltype(ii)::value, -1>();
        if constexpr (WL) __syncwarp();
        else team_sync<PL>();
      });
      last_paired();
      if constexpr (WL) __syncwarp();
      else team_sync<PL>();
      static_for<1, NP - 1>([&](auto ii) {
        pass<NP - 1 - decltype(ii)::value, +1>();
        team_sync<PL>();
      });
    } else if constexpr (WLU) {
#pragma unroll 1
      for (int q = 0; q < UPW; ++q) {
        if ((lt >> 5) + NWT * q < NU) unit(q);  // warp-uniform
      }
      team_sync<PL>();
    } else {
      static_for<1, NP>([&](auto ii) {
        constexpr int I = decltype(ii)::value;
        pass<I, -1>();
        if constexpr (L12 && I == 1) __syncwarp();
        else team_sync<PL>();
      });
      middle_slots(v);
      team_sync<PL>();
      static_for<1, NP>([&](auto ii) {
        constexpr int I = decltype(ii)::value;
        pass<NP - I, +1>();
        if constexpr (L12 && I == 1) __syncwarp();
        else team_sync<PL>();
      });
    }
    inv0(v);
  }
};

// ---------------------------------------------------------------------------
// Table set-up for one plan: access-ordered twiddles (double-precision sincospi,
// rounded), the sign bits (SplitMix64 of seed + (j+1)*gamma, bit 63 set ->
// eps_j = -1) and the cleared status word.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 root_w(long long m, long long b) {  // exp(-2 pi i m / b)
  double s, c;
  sincospi(2.0 * (double)m / (double)b, &s, &c);
  return make_float2((float)c, (float)(-s));
}

template <class PL>
__global__ void setup_kernel(float2* twt, uint32_t* eps, uint32_t* status, uint64_t seed) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int stride = gridDim.x * blockDim.x;
  if (tid == 0) *status = 0u;
  for (int e = tid; e < PL::TWN; e += stride) {
    long long m = 0, b = 1;
    static_for<0, PL::NP - 1>([&](auto ii) {
      constexpr int I = decltype(ii)::value;
      constexpr int OFF = PL::tw_off(I);
      constexpr int LEN = PL::B(I);
      if (e >= OFF && e < OFF + LEN) {
        const int r = e - OFF;
        // row j, column c: pass 0 W_N^{c j} (c = thread), pass I W_B^{c j} (c = np)
        constexpr int L = (I == 0) ? PL::T : PL::S(I);
        int j, c;
        if constexpr (PL::TW2) {  // [j / 2][c][j % 2]
          j = 2 * (r / (2 * L)) + (r % 2);
          c = (r % (2 * L)) / 2;
        } else {                  // [j][c]
          j = r / L;
          c = r % L;
        }
        m = (long long)c * j;
        b = (I == 0) ? PL::N : LEN;
      }
    });
    twt[e] = root_w(m, b);
  }
  constexpr int words = (PL::N + 31) / 32;
  for (int wd = tid; wd < words; wd += stride) {
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; ++bb) {
      const int j = wd * 32 + bb;
      if (j >= PL::N) break;
      const uint64_t z = splitmix64_mix(seed + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull);
      bits |= (uint32_t)(z >> 63) << bb;
    }
    eps[wd] = bits;
  }
}

}  // namespace kd
