// Device arithmetic for the Kashin-DCT kernels: complex helpers, compile-time
// trigonometric constants, and in-register small DFTs.
//
// All floating-point operations here use explicit round-to-nearest intrinsics
// (the library is compiled with --fmad=false), so every instantiation of a kernel
// performs the same operations in the same order: the trace build and the
// timed build are bitwise identical.
#pragma once

#include <cstdint>
#include <type_traits>
#include <cuda_runtime.h>

#define KD_HD __host__ __device__

namespace kd {

// SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014): the sign of
// entry j of a seeded sign set is bit 63 of mix(seed + (j + 1) * 0x9E3779B97F4A7C15).
__device__ __forceinline__ uint64_t splitmix64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// ---------------------------------------------------------------------------
// Compile-time cos / sin of 2*pi*a/b (double), from the Taylor series after an
// exact rational reduction of the angle to [-pi/4, pi/4].
// ---------------------------------------------------------------------------
constexpr double kPi = 3.141592653589793238462643383279502884;

KD_HD constexpr double taylor_sin(double x) {
  double term = x, sum = x;
  for (int k = 1; k < 16; ++k) {
    term *= -x * x / ((2.0 * k) * (2.0 * k + 1.0));
    sum += term;
  }
  return sum;
}

KD_HD constexpr double taylor_cos(double x) {
  double term = 1.0, sum = 1.0;
  for (int k = 1; k < 16; ++k) {
    term *= -x * x / ((2.0 * k - 1.0) * (2.0 * k));
    sum += term;
  }
  return sum;
}

// angle 2*pi*a/b: a reduced mod b, q = nearest quarter turn, remainder exact.
KD_HD constexpr long long kd_mod(long long a, long long b) { return ((a % b) + b) % b; }

KD_HD constexpr double cos2pi(long long a, long long b) {
  long long r = kd_mod(a, b);
  long long q = (4 * r * 2 + b) / (2 * b);  // round(4r/b)
  double f = kPi * (double)(4 * r - q * b) / (2.0 * (double)b);
  switch (q & 3) {
    case 0: return taylor_cos(f);
    case 1: return -taylor_sin(f);
    case 2: return -taylor_cos(f);
    default: return taylor_sin(f);
  }
}

KD_HD constexpr double sin2pi(long long a, long long b) {
  long long r = kd_mod(a, b);
  long long q = (4 * r * 2 + b) / (2 * b);
  double f = kPi * (double)(4 * r - q * b) / (2.0 * (double)b);
  switch (q & 3) {
    case 0: return taylor_sin(f);
    case 1: return taylor_cos(f);
    case 2: return -taylor_sin(f);
    default: return -taylor_cos(f);
  }
}

// ---------------------------------------------------------------------------
// Complex helpers (float2 = re, im)
// ---------------------------------------------------------------------------
// Complex add / subtract as one packed FP32x2 fused multiply-add with +-1 (the
// same rounding as separate adds: b * 1 is exact), half the issue slots.
__device__ __forceinline__ float2 cadd(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(1.f, 1.f), a);
}
__device__ __forceinline__ float2 csub(float2 a, float2 b) {
  return __ffma2_rn(b, make_float2(-1.f, -1.f), a);
}
// Complex products stay scalar: a packed form needs a sign-flipped copy of one
// operand, one more FMA-pipe instruction than the four scalar ones (measured).
// a * b
__device__ __forceinline__ float2 cmul(float2 a, float2 b) {
  return make_float2(__fmaf_rn(a.x, b.x, __fmul_rn(-a.y, b.y)),
                     __fmaf_rn(a.x, b.y, __fmul_rn(a.y, b.x)));
}
// a * conj(b)
__device__ __forceinline__ float2 cmulc(float2 a, float2 b) {
  return make_float2(__fmaf_rn(a.x, b.x, __fmul_rn(a.y, b.y)),
                     __fmaf_rn(a.y, b.x, __fmul_rn(-a.x, b.y)));
}
__device__ __forceinline__ float2 cscale(float2 a, float s) {
  return make_float2(__fmul_rn(a.x, s), __fmul_rn(a.y, s));
}
// -i * a   (exact)
__device__ __forceinline__ float2 mul_mi(float2 a) { return make_float2(a.y, -a.x); }
// +i * a   (exact)
__device__ __forceinline__ float2 mul_pi(float2 a) { return make_float2(-a.y, a.x); }
// a + i b and a - i b as two scalar adds (the packed forms below, one instruction each,
// are used by the plans with packed constant roots and by Rader's form).
__device__ __forceinline__ float2 add_ib(float2 a, float2 b) {
  return make_float2(__fsub_rn(a.x, b.y), __fadd_rn(a.y, b.x));
}
__device__ __forceinline__ float2 sub_ib(float2 a, float2 b) {
  return make_float2(__fadd_rn(a.x, b.y), __fsub_rn(a.y, b.x));
}
// swapped pair: packed FP32x2 instructions read either half of a register pair for
// either lane, so (a.y, a.x) as an operand costs no instruction (measured on sm_103a)
__device__ __forceinline__ float2 swp(float2 a) { return make_float2(a.y, a.x); }
// a + i b and a - i b as one packed FMA on the swapped pair (b times +-1 is exact, so
// each lane rounds once, exactly as the scalar forms)
__device__ __forceinline__ float2 add_ib_pk(float2 a, float2 b) {
  return __ffma2_rn(swp(b), make_float2(-1.f, 1.f), a);
}
__device__ __forceinline__ float2 sub_ib_pk(float2 a, float2 b) {
  return __ffma2_rn(swp(b), make_float2(1.f, -1.f), a);
}

// Multiply by the compile-time root W_R^E = exp(DIR * 2 pi i E / R), DIR = -1 forward.
// Quarter turns are exact; eighth turns use one constant; others a full product.
// PK selects packed forms on the swapped pair (two FP32x2 instructions instead of
// four scalar ones, the same FMA-pipe cycles): fewer issue slots, but the constant
// pairs occupy registers, so a plan opts in only where registers are to spare.
template <int DIR, long long E, long long R, bool PK = false>
__device__ __forceinline__ float2 mul_root(float2 a) {
  constexpr long long e = kd_mod(E, R);
  if constexpr (e == 0) {
    return a;
  } else if constexpr ((4 * e) % R == 0) {
    constexpr long long qtr = (4 * e) / R;  // 1, 2, 3 quarter turns (counter-clockwise for DIR=+1)
    constexpr long long q = (DIR > 0) ? qtr : (4 - qtr) % 4;
    if constexpr (q == 1) return mul_pi(a);
    else if constexpr (q == 2) return make_float2(-a.x, -a.y);
    else return mul_mi(a);
  } else if constexpr ((8 * e) % R == 0) {
    constexpr float h = (float)0.70710678118654752440084436210484903928;
    constexpr long long o = (8 * e) / R;  // odd octant 1,3,5,7
    constexpr long long oo = (DIR > 0) ? o : (8 - o);
    // exp(i*pi*oo/4) = (c, s) with |c| = |s| = h
    constexpr float c = (oo == 1 || oo == 7) ? h : -h;
    constexpr float s = (oo == 1 || oo == 3) ? h : -h;
    // (a.x + i a.y)(c + i s) = c (a.x - (s/c) a.y, a.y + (s/c) a.x) with s/c = +-1 exact:
    // one packed FMA on the swapped pair, one packed multiply
    if constexpr (PK) {
      constexpr float q = (c > 0) == (s > 0) ? 1.f : -1.f;
      return __fmul2_rn(__ffma2_rn(swp(a), make_float2(-q, q), a), make_float2(c, c));
    } else if constexpr ((c > 0) == (s > 0)) {
      return make_float2(__fmul_rn(c, __fsub_rn(a.x, a.y)), __fmul_rn(c, __fadd_rn(a.y, a.x)));
    } else {
      return make_float2(__fmul_rn(c, __fadd_rn(a.x, a.y)), __fmul_rn(c, __fsub_rn(a.y, a.x)));
    }
  } else {
    constexpr float c = (float)cos2pi(e, R);
    constexpr float s = (float)((DIR > 0 ? 1.0 : -1.0) * sin2pi(e, R));
    if constexpr (PK) {
      // a (c, c) + swap(a) (-s, s)
      return __ffma2_rn(swp(a), make_float2(-s, s), __fmul2_rn(a, make_float2(c, c)));
    } else {
      return make_float2(__fmaf_rn(a.x, c, __fmul_rn(-a.y, s)), __fmaf_rn(a.x, s, __fmul_rn(a.y, c)));
    }
  }
}

// ---------------------------------------------------------------------------
// Compile-time loop: f(std::integral_constant<int, I>{}) for I in [B, E).
// ---------------------------------------------------------------------------
template <int I>
using ic = std::integral_constant<int, I>;

template <int B, int E, class F>
__device__ __forceinline__ void static_for(F&& f) {
  if constexpr (B < E) {
    f(ic<B>{});
    static_for<B + 1, E>(f);
  }
}

// ---------------------------------------------------------------------------
// In-register DFT of size R (DIR = -1 forward, +1 inverse, unnormalised):
//   X[k] = sum_n x[n] exp(DIR * 2 pi i n k / R), natural order in and out.
// ---------------------------------------------------------------------------
template <int R>
struct SmallestFactor {
  static constexpr int value = (R % 4 == 0 && R > 4) ? 4 : (R % 2 == 0) ? 2 : (R % 3 == 0) ? 3
                             : (R % 5 == 0) ? 5 : (R % 7 == 0) ? 7 : R;
};

template <int R, int DIR, bool PK = false>
struct Dft;

template <int DIR, bool PK>
struct Dft<1, DIR, PK> {
  template <class A>
  __device__ __forceinline__ static void run(A&) {}
};

template <int DIR, bool PK>
struct Dft<2, DIR, PK> {
  template <class A>
  __device__ __forceinline__ static void run(A& v) {
    float2 a = v[0], b = v[1];
    v[0] = cadd(a, b);
    v[1] = csub(a, b);
  }
};

template <int DIR, bool PK>
struct Dft<4, DIR, PK> {
  template <class A>
  __device__ __forceinline__ static void run(A& v) {
    float2 s02 = cadd(v[0], v[2]), d02 = csub(v[0], v[2]);
    float2 s13 = cadd(v[1], v[3]), d13 = csub(v[1], v[3]);
    // forward: X1 = d02 - i d13, X3 = d02 + i d13 ; inverse: signs swapped
    v[0] = cadd(s02, s13);
    v[2] = csub(s02, s13);
    if constexpr (PK) {
      v[1] = DIR < 0 ? sub_ib_pk(d02, d13) : add_ib_pk(d02, d13);
      v[3] = DIR < 0 ? add_ib_pk(d02, d13) : sub_ib_pk(d02, d13);
    } else if constexpr (DIR < 0) {
      v[1] = sub_ib(d02, d13);
      v[3] = add_ib(d02, d13);
    } else {
      v[1] = add_ib(d02, d13);
      v[3] = sub_ib(d02, d13);
    }
  }
};

// Odd prime R: symmetric direct form.  a_n = x_n + x_{R-n}, b_n = x_n - x_{R-n};
// X_k = x_0 + sum a_n cos(2 pi n k / R) -+ i sum b_n sin(2 pi n k / R).
template <int R, int DIR, bool PK = false>
struct DftPrime {
  template <class Arr>
  __device__ __forceinline__ static void run(Arr& v) {
    constexpr int H = (R - 1) / 2;
    float2 a[H + 1], b[H + 1];
    const float2 x0 = v[0];
    float2 sum = x0;
#pragma unroll
    for (int n = 1; n <= H; ++n) {
      a[n] = cadd(v[n], v[R - n]);
      b[n] = csub(v[n], v[R - n]);
      sum = cadd(sum, a[n]);
    }
    v[0] = sum;
    static_for<1, H + 1>([&](auto kk) {
      constexpr int K = decltype(kk)::value;
      float2 ak = x0;
      float2 bk = make_float2(0.f, 0.f);
      static_for<1, H + 1>([&](auto nn) {
        constexpr int NN = decltype(nn)::value;
        constexpr float c = (float)cos2pi((long long)NN * K, R);
        constexpr float s = (float)sin2pi((long long)NN * K, R);
        ak = __ffma2_rn(a[NN], make_float2(c, c), ak);
        bk = __ffma2_rn(b[NN], make_float2(s, s), bk);
      });
      // forward: X_k = ak - i bk, X_{R-k} = ak + i bk ; inverse: the reverse
      if constexpr (PK) {
        v[K] = DIR < 0 ? sub_ib_pk(ak, bk) : add_ib_pk(ak, bk);
        v[R - K] = DIR < 0 ? add_ib_pk(ak, bk) : sub_ib_pk(ak, bk);
      } else if constexpr (DIR < 0) {
        v[K] = sub_ib(ak, bk);
        v[R - K] = add_ib(ak, bk);
      } else {
        v[K] = add_ib(ak, bk);
        v[R - K] = sub_ib(ak, bk);
      }
    });
  }
};

// Odd prime R, streaming form: inputs come from load(n) (each read once), outputs
// leave through store(k, X) as soon as they are formed, so only the symmetric
// sums a_n, b_n stay live (used where R is too large to hold inputs and outputs
// in registers at once).
template <int R, int DIR, class Load, class Store>
__device__ __forceinline__ void dft_prime_stream(Load&& load, Store&& store) {
  constexpr int H = (R - 1) / 2;
  float2 a[H + 1], b[H + 1];
  const float2 x0 = load(ic<0>{});
  float2 sum = x0;
  static_for<1, H + 1>([&](auto nc) {
    constexpr int NN = decltype(nc)::value;
    const float2 p = load(ic<NN>{}), q = load(ic<R - NN>{});
    a[NN] = cadd(p, q);
    b[NN] = csub(p, q);
    sum = cadd(sum, a[NN]);
  });
  store(ic<0>{}, sum);
  static_for<1, H + 1>([&](auto kk) {
    constexpr int K = decltype(kk)::value;
    float2 ak = x0;
    float2 bk = make_float2(0.f, 0.f);
    static_for<1, H + 1>([&](auto nn) {
      constexpr int NN = decltype(nn)::value;
      constexpr float c = (float)cos2pi((long long)NN * K, R);
      constexpr float sn = (float)sin2pi((long long)NN * K, R);
      // one packed FMA per complex term (both lanes round exactly like two FFMAs)
      ak = __ffma2_rn(a[NN], make_float2(c, c), ak);
      bk = __ffma2_rn(b[NN], make_float2(sn, sn), bk);
    });
    if constexpr (DIR < 0) {
      store(ic<K>{}, sub_ib(ak, bk));
      store(ic<R - K>{}, add_ib(ak, bk));
    } else {
      store(ic<K>{}, add_ib(ak, bk));
      store(ic<R - K>{}, sub_ib(ak, bk));
    }
  });
}

template <int R>
KD_HD constexpr bool kd_is_big_prime() {
  if (R < 11 || R % 2 == 0) return false;
  for (int d = 3; d * d <= R; d += 2)
    if (R % d == 0) return false;
  return true;
}

// ---------------------------------------------------------------------------
// Odd prime R by Rader's mapping (C. M. Rader, Proc. IEEE 56, 1968), split in halves.
//
// With g a primitive root mod R and H = (R-1)/2 (so g^H = -1 mod R), take inputs in
// the order n_q = g^-q and outputs k_m = g^m.  Then n_q k_m = g^(m-q) and, with
//   u_q = x(n_q) + x(-n_q),   v_q = x(n_q) - x(-n_q)          (q = 0 .. H-1),
//   C_j = cos(2 pi g^j / R)   (period H in j),
//   S_j = sin(2 pi g^j / R)   (S_(j+H) = -S_j),
// the outputs are
//   X(k_m) = x_0 + P_m + DIR i Q_m,   X(-k_m) = x_0 + P_m - DIR i Q_m,   X_0 = x_0 + sum u,
// where P = u (*) C is a cyclic convolution of length H and Q = v (*) S a negacyclic
// one.  For odd H the negacyclic one turns cyclic by alternating signs:
// J_j = (-1)^j S_j has period H and Q_m = (-1)^m [((-1)^q v_q) (*) J]_m.  Both cyclic
// convolutions run through length-H DFTs against the constant spectra
// C^_k = DFT_H(C)_k / H and J^_k = DFT_H(J)_k / H; x_0 enters as the zero-frequency
// term of the inverse.  With H = A B, gcd(A, B) = 1, each length-H DFT is a
// prime-factor (Good-Thomas) A x B DFT without twiddles.
//
// Per point of a 43-point DFT this is about 35 FMA-pipe operations against 46 for the
// symmetric direct form, with independent butterflies instead of 21-term chains.  The
// spectrum products and the final a +- i b run as packed FP32x2 instructions, which keeps
// the code (and the instruction-cache footprint of the kernel) small.
// ---------------------------------------------------------------------------
KD_HD constexpr long long kd_powmod(long long b, long long e, long long m) {
  long long r = 1;
  b = kd_mod(b, m);
  while (e > 0) {
    if (e & 1) r = r * b % m;
    b = b * b % m;
    e >>= 1;
  }
  return r;
}

KD_HD constexpr int kd_primitive_root(int R) {
  for (int g = 2; g < R; ++g) {
    bool full = true;
    for (int e = 1; e < R - 1 && full; ++e)
      if (kd_powmod(g, e, R) == 1) full = false;
    if (full) return g;
  }
  return 0;
}

KD_HD constexpr int kd_smallest_factor(int h) {
  for (int d = 2; d * d <= h; ++d)
    if (h % d == 0) return d;
  return h;
}

// Rader's mapping applies when H = (R-1)/2 is odd and splits into two coprime factors.
template <int R>
KD_HD constexpr bool kd_rader_split() {
  if (!kd_is_big_prime<R>()) return false;
  const int h = (R - 1) / 2;
  if (h % 2 == 0) return false;
  const int a = kd_smallest_factor(h);
  return a != h && (h / a) % a != 0;
}

// (1/H) sum_j f_j exp(-2 pi i j k / H), f_j = C_j (KIND 0) or J_j (KIND 1); IM picks the part
template <int R, int KIND, bool IM>
KD_HD constexpr double kd_rader_spectrum(int k) {
  const int h = (R - 1) / 2;
  const long long g = kd_primitive_root(R);
  double s = 0.0;
  for (int j = 0; j < h; ++j) {
    const long long gj = kd_powmod(g, j, R);
    const double f = KIND == 0 ? cos2pi(gj, R) : ((j & 1) ? -1.0 : 1.0) * sin2pi(gj, R);
    s += f * (IM ? -sin2pi((long long)j * k, h) : cos2pi((long long)j * k, h));
  }
  return s / h;
}

// in-register prime-factor DFT of size A*B (gcd 1), sign SGN, natural order in and out:
// input n = (B n1 + A n2) mod AB, output k = (B (B^-1 mod A) k1 + A (A^-1 mod B) k2) mod AB
template <int A, int B, int SGN, class Arr>
__device__ __forceinline__ void dft_pfa(Arr& y) {
  constexpr int N = A * B;
  constexpr int ka = B * (int)kd_powmod(B, A == 2 ? 0 : A - 2, A) % N;   // B (B^-1 mod A), A prime
  constexpr int kb = A * (int)kd_powmod(A, B == 2 ? 0 : B - 2, B) % N;   // A (A^-1 mod B), B prime
  float2 t[N];
  static_for<0, B>([&](auto n2c) {
    constexpr int N2 = decltype(n2c)::value;
    float2 s[A];
    static_for<0, A>([&](auto n1c) { s[decltype(n1c)::value] = y[(B * decltype(n1c)::value + A * N2) % N]; });
    Dft<A, SGN, true>::run(s);
    static_for<0, A>([&](auto k1c) { t[decltype(k1c)::value * B + N2] = s[decltype(k1c)::value]; });
  });
  static_for<0, A>([&](auto k1c) {
    constexpr int K1 = decltype(k1c)::value;
    float2 s[B];
    static_for<0, B>([&](auto n2c) { s[decltype(n2c)::value] = t[K1 * B + decltype(n2c)::value]; });
    Dft<B, SGN, true>::run(s);
    static_for<0, B>([&](auto k2c) { y[(ka * K1 + kb * decltype(k2c)::value) % N] = s[decltype(k2c)::value]; });
  });
}

// a * (c + i s) with compile-time c, s: two packed operations on the swapped pair (the
// constants carry the sign, so no operand needs negating)
template <int R, int KIND, int K>
__device__ __forceinline__ float2 mul_rader_spectrum(float2 a) {
  constexpr float c = (float)kd_rader_spectrum<R, KIND, false>(K);
  constexpr float s = (float)kd_rader_spectrum<R, KIND, true>(K);
  return __ffma2_rn(swp(a), make_float2(-s, s), __fmul2_rn(a, make_float2(c, c)));
}

// Streaming form, the same interface as dft_prime_stream: every input is read once
// through load(n), every output leaves once through store(k, X).
template <int R, int DIR, class Load, class Store>
__device__ __forceinline__ void dft_prime_rader(Load&& load, Store&& store) {
  static_assert(kd_rader_split<R>(), "Rader split needs (R-1)/2 odd with two coprime factors");
  constexpr int H = (R - 1) / 2;
  constexpr int FA = kd_smallest_factor(H);
  constexpr int FB = H / FA;
  static_assert(kd_smallest_factor(FB) == FB, "second factor must be prime");
  constexpr long long g = kd_primitive_root(R);
  constexpr long long gi = kd_powmod(g, R - 2, R);
  float2 u[H], w[H];
  const float2 x0 = load(ic<0>{});
  static_for<0, H>([&](auto qc) {
    constexpr int Q = decltype(qc)::value;
    constexpr int n = (int)kd_powmod(gi, Q, R);
    const float2 p = load(ic<n>{}), m = load(ic<R - n>{});
    u[Q] = cadd(p, m);
    w[Q] = (Q & 1) ? csub(m, p) : csub(p, m);   // (-1)^q v_q
  });
  dft_pfa<FA, FB, -1>(u);
  dft_pfa<FA, FB, -1>(w);
  store(ic<0>{}, cadd(x0, u[0]));
  {
    constexpr float c0 = (float)kd_rader_spectrum<R, 0, false>(0);   // real: C and J are real
    constexpr float j0 = (float)kd_rader_spectrum<R, 1, false>(0);
    u[0] = __ffma2_rn(u[0], make_float2(c0, c0), x0);
    w[0] = __fmul2_rn(w[0], make_float2(j0, j0));
  }
  static_for<1, H>([&](auto kc) {
    constexpr int K = decltype(kc)::value;
    u[K] = mul_rader_spectrum<R, 0, K>(u[K]);
    w[K] = mul_rader_spectrum<R, 1, K>(w[K]);
  });
  dft_pfa<FA, FB, +1>(u);
  dft_pfa<FA, FB, +1>(w);
  static_for<0, H>([&](auto mc) {
    constexpr int M = decltype(mc)::value;
    constexpr int k = (int)kd_powmod(g, M, R);
    // X(k_m) = P_m + s i Q'_m with s = DIR (-1)^m
    if constexpr ((DIR < 0) != ((M & 1) != 0)) {
      store(ic<k>{}, sub_ib_pk(u[M], w[M]));
      store(ic<R - k>{}, add_ib_pk(u[M], w[M]));
    } else {
      store(ic<k>{}, add_ib_pk(u[M], w[M]));
      store(ic<R - k>{}, sub_ib_pk(u[M], w[M]));
    }
  });
}

// the big-prime pass: Rader's form where it applies, else the symmetric direct form
template <int R, int DIR, class Load, class Store>
__device__ __forceinline__ void dft_prime_pass(Load&& load, Store&& store) {
  if constexpr (kd_rader_split<R>()) {
    dft_prime_rader<R, DIR>(load, store);
  } else {
    dft_prime_stream<R, DIR>(load, store);
  }
}

// Composite R = A * B (A = smallest factor, 4 preferred): decimation in frequency.
//   n = B*n1 + n2 ; k = k1 + A*k2
//   step 1: for each n2, size-A DFT over n1 -> k1 ; multiply by W_R^{n2*k1}
//   step 2: for each k1, size-B DFT over n2 -> k2.
template <int R, int DIR, bool PK>
struct DftComposite {
  static constexpr int A = SmallestFactor<R>::value;
  static constexpr int B = R / A;
  template <class Arr>
  __device__ __forceinline__ static void run(Arr& v) {
    float2 t[R];
    static_for<0, B>([&](auto n2c) {
      constexpr int N2 = decltype(n2c)::value;
      float2 s[A];
#pragma unroll
      for (int n1 = 0; n1 < A; ++n1) s[n1] = v[B * n1 + N2];
      Dft<A, DIR, PK>::run(s);
      static_for<0, A>([&](auto k1c) {
        constexpr int K1 = decltype(k1c)::value;
        t[K1 * B + N2] = mul_root<DIR, (long long)N2 * K1, R, PK>(s[K1]);
      });
    });
#pragma unroll
    for (int k1 = 0; k1 < A; ++k1) {
      float2 s[B];
#pragma unroll
      for (int n2 = 0; n2 < B; ++n2) s[n2] = t[k1 * B + n2];
      Dft<B, DIR, PK>::run(s);
#pragma unroll
      for (int k2 = 0; k2 < B; ++k2) v[k1 + A * k2] = s[k2];
    }
  }
};

template <int R, int DIR, bool PK>
struct Dft {
  template <class A>
  __device__ __forceinline__ static void run(A& v) {
    if constexpr (SmallestFactor<R>::value == R) {
      DftPrime<R, DIR, PK>::run(v);
    } else {
      DftComposite<R, DIR, PK>::run(v);
    }
  }
};

}  // namespace kd
