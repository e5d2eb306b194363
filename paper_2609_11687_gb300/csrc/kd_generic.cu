// Run-time-length path: the vector lengths without a compiled plan.
//
// Any n with 1 <= n <= 16384 whose prime factors all lie in {2, 3, 5, 7, 11, 13, 43}
// runs here with the same method and outputs as the per-length plans (Algorithm 1,
// the closed-form centres of Sec. 2.1, the optional k-means refinement, the 2-bit
// codes of App. C; P, and the dense re-materialisation).  What changes is the
// transform's shape, which is chosen when the call is made:
//  - the pair (two vectors packed as one complex vector, Makhoul order) lives in a
//    padded shared-memory buffer for the whole of Algorithm 1, and every radix
//    pass of the complex FFT is a shared-memory pass (radices 16, 8, 4, 2, 9, 3, 5,
//    7, 11, 13, 43, chosen from the factorisation of n);
//  - the frequency pairs (k, n - k) of the middle operator M are found through a
//    slot table instead of per-thread constants;
//  - u lives in a per-CTA workspace slot (L2-resident), one CTA of 256 threads per
//    vector pair.
// Makhoul's reordering and the middle operator hold for odd n as well (the even
// positions take the first ceil(n/2) slots); the code words of a vector are
// ceil(n/16), the last one padded with zero codes.
#include <map>
#include <mutex>

#include "kd_kernels.cuh"
#include "kd_ops.h"

namespace kd {
namespace {

constexpr int kGenMaxPasses = 16;
constexpr int kGenThreads = 256;
constexpr int64_t kGenMaxN = 16384;
constexpr int kGenRedFloats = 160;  // >= 16 (warps + 1) (k-means sums) and 4 warps (l1 sums)

// Team shape for the shared reduction helpers: the whole CTA is one team.
struct GenTeam {
  static constexpr int T = kGenThreads;
  static constexpr int NW = kGenThreads / 32;
};

// Radix passes of one length: pass i splits sub-transforms of length B[i] into
// R[i] interleaved ones of length S[i] = B[i] / R[i] (decimation in frequency).
struct GenPlan {
  int n, np;
  int R[kGenMaxPasses], S[kGenMaxPasses], B[kGenMaxPasses];
  int tw[kGenMaxPasses];  // float2 offset of pass i's twiddles [j][s] = W_{B[i]}^{s j} (not the last pass)
  int woff;               // float2 offset of exp(i pi k / n), k = 0 .. n/2
  int permoff;            // float2 offset of the slot of frequency k (int32), k < n
  int twn;                // float2 units of the whole table
};

bool gen_plan(int64_t n, GenPlan* g) {
  if (n < 1 || n > kGenMaxN) return false;
  static const int radices[] = {16, 8, 4, 2, 9, 3, 5, 7, 11, 13, 43};
  int rem = (int)n, np = 0;
  for (int r : radices) {
    while (rem % r == 0) {
      if (np == kGenMaxPasses) return false;
      g->R[np++] = r;
      rem /= r;
    }
  }
  if (rem != 1) return false;
  g->n = (int)n;
  g->np = np;
  int b = (int)n, off = 0;
  for (int i = 0; i < np; ++i) {
    g->B[i] = b;
    g->S[i] = b / g->R[i];
    g->tw[i] = off;
    if (i < np - 1) off += b;
    b = g->S[i];
  }
  g->woff = off;
  g->permoff = g->woff + (int)n / 2 + 1;
  g->twn = g->permoff + ((int)n + 1) / 2;
  return true;
}

size_t gen_smem(int64_t n) {
  const size_t bufn = (size_t)((n + n / 16 + n / 256 + 8 + 15) / 16 * 16);
  const size_t ps = (size_t)((n + 15) / 16 * 16);  // code bytes per plane
  return bufn * sizeof(float2) + kGenRedFloats * sizeof(float) + 4 * ps;
}

// Natural index of Makhoul slot s, and its inverse (any n).
__device__ __forceinline__ int gen_nat(int s, int n) { return s < ((n + 1) >> 1) ? 2 * s : 2 * n - 1 - 2 * s; }
__device__ __forceinline__ int gen_slot(int nat, int n) { return (nat & 1) ? n - ((nat + 1) >> 1) : nat >> 1; }

// One shared-memory radix pass over all groups of the pair buffer.  Forward (DIR < 0):
// DFT then the twiddles of the next level; inverse: conjugate twiddles then IDFT.
template <int R, int DIR>
__device__ __forceinline__ void gen_pass_r(float2* buf, const float2* __restrict__ tw, int n, int S, int Bk, bool last,
                                           int lt) {
  const int G = n / R;
  for (int g = lt; g < G; g += kGenThreads) {
    const int blk = g / S;
    const int sp = g - blk * S;
    const int base = blk * Bk + sp;
    if constexpr (kd_is_big_prime<R>()) {
      // streaming form (Rader's for 43, direct otherwise): every load precedes the first store
      if constexpr (DIR < 0) {
        dft_prime_pass<R, -1>([&](auto jc) { return buf[pad(base + decltype(jc)::value * S)]; },
                                [&](auto kc, float2 x) {
                                  constexpr int K = decltype(kc)::value;
                                  if (K > 0 && !last) x = cmul(x, __ldg(&tw[K * S + sp]));
                                  buf[pad(base + K * S)] = x;
                                });
      } else {
        dft_prime_pass<R, +1>(
            [&](auto jc) {
              constexpr int J = decltype(jc)::value;
              float2 x = buf[pad(base + J * S)];
              if (J > 0 && !last) x = cmulc(x, __ldg(&tw[J * S + sp]));
              return x;
            },
            [&](auto kc, float2 x) { buf[pad(base + decltype(kc)::value * S)] = x; });
      }
    } else {
      float2 v[R];
#pragma unroll
      for (int j = 0; j < R; ++j) v[j] = buf[pad(base + j * S)];
      if constexpr (DIR < 0) {
        Dft<R, -1>::run(v);
        if (!last) {
#pragma unroll
          for (int j = 1; j < R; ++j) v[j] = cmul(v[j], __ldg(&tw[j * S + sp]));
        }
      } else {
        if (!last) {
#pragma unroll
          for (int j = 1; j < R; ++j) v[j] = cmulc(v[j], __ldg(&tw[j * S + sp]));
        }
        Dft<R, +1>::run(v);
      }
#pragma unroll
      for (int j = 0; j < R; ++j) buf[pad(base + j * S)] = v[j];
    }
  }
}

template <int DIR>
__device__ void gen_pass(const GenPlan& g, int i, float2* buf, const float2* __restrict__ tab, int lt) {
  const bool last = (i == g.np - 1);
  const float2* tw = tab + g.tw[i];
  const int n = g.n, S = g.S[i], Bk = g.B[i];
  switch (g.R[i]) {
    case 16: gen_pass_r<16, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 8: gen_pass_r<8, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 4: gen_pass_r<4, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 2: gen_pass_r<2, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 9: gen_pass_r<9, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 3: gen_pass_r<3, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 5: gen_pass_r<5, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 7: gen_pass_r<7, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 11: gen_pass_r<11, DIR>(buf, tw, n, S, Bk, last, lt); break;
    case 13: gen_pass_r<13, DIR>(buf, tw, n, S, Bk, last, lt); break;
    default: gen_pass_r<43, DIR>(buf, tw, n, S, Bk, last, lt); break;
  }
}

// M between the forward and inverse FFT (1/n folded in): for each frequency pair
// (k, n - k), if eps_k == eps_{n-k}:  Z'_k = eps_k Z_k / n,  Z'_{n-k} = eps_k Z_{n-k} / n;
// otherwise Z'_k = eps_k w_k Z_{n-k} / n,  Z'_{n-k} = eps_k conj(w_k) Z_k / n  (w_k = exp(i pi k/n)).
// Frequencies 0 and n/2 pair with themselves: Z'_k = eps_k Z_k / n.
__device__ void gen_middle(const GenPlan& g, float2* buf, const float2* __restrict__ tab,
                           const uint32_t* __restrict__ eb, int lt) {
  const int n = g.n;
  const float2* wk = tab + g.woff;
  const int* perm = reinterpret_cast<const int*>(tab + g.permoff);
  const float inv = __fdiv_rn(1.f, (float)n);
  for (int k = lt; 2 * k <= n; k += kGenThreads) {
    const int kk = (k == 0) ? 0 : n - k;
    const int sa = pad(__ldg(&perm[k]));
    const float2 a = buf[sa];
    const bool ek = eps_neg(eb, k);
    const float f = ek ? -inv : inv;
    if (kk == k) {
      buf[sa] = make_float2(__fmul_rn(a.x, f), __fmul_rn(a.y, f));
      continue;
    }
    const int sb = pad(__ldg(&perm[kk]));
    const float2 b = buf[sb];
    float2 za = a, zb = b;
    if (ek != eps_neg(eb, kk)) {
      const float2 w = __ldg(&wk[k]);
      za = cmul(b, w);
      zb = cmulc(a, w);
    }
    buf[sa] = make_float2(__fmul_rn(za.x, f), __fmul_rn(za.y, f));
    buf[sb] = make_float2(__fmul_rn(zb.x, f), __fmul_rn(zb.y, f));
  }
}

// buf <- P' buf (both packed vectors, Makhoul order in and out).  Starts with a
// barrier (callers have just written their own slots) and ends with one.
__device__ void gen_apply(const GenPlan& g, float2* buf, const float2* __restrict__ tab,
                          const uint32_t* __restrict__ eb, int lt) {
  __syncthreads();
  for (int i = 0; i < g.np; ++i) {
    gen_pass<-1>(g, i, buf, tab, lt);
    __syncthreads();
  }
  gen_middle(g, buf, tab, eb, lt);
  __syncthreads();
  for (int i = g.np - 1; i >= 0; --i) {
    gen_pass<+1>(g, i, buf, tab, lt);
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Decomposition: the steps, normalisation, centres, refinement and codes of the
// per-length kernel, over shared-memory slots s = lt + j * 256.
// ---------------------------------------------------------------------------
template <bool TRACE>
__global__ void __launch_bounds__(kGenThreads, 2) gen_decompose_kernel(DecParams p, const __grid_constant__ GenPlan g) {
  extern __shared__ __align__(16) float2 smem[];
  constexpr int T = kGenThreads;
  const int n = g.n;
  const int lt = threadIdx.x;
  const int bufn = (n + n / 16 + n / 256 + 8 + 15) / 16 * 16;
  float2* buf = smem;
  float2* red = smem + bufn;
  uint8_t* cb = reinterpret_cast<uint8_t*>(reinterpret_cast<float*>(red) + kGenRedFloats);
  const int WPV = (n + 15) / 16;
  const int PS = WPV * 16;  // code bytes per plane
  const float2* tab = p.twt;
  float2* uslot = p.uslots + (int64_t)blockIdx.x * n;
  int parity = 0;
  const int nsteps = 4 * p.iters + 2 * p.kmeans_iters;

  for (int64_t pr = blockIdx.x; pr < p.npairs; pr += gridDim.x) {
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < p.m;
    const int64_t colB = hasB ? colA + 1 : colA;

    float2 acc = make_float2(0.f, 0.f);
    for (int s = lt; s < n; s += T) {
      const int nat = gen_nat(s, n);
      const float a = load_elem(p.w, p.dtype, elem_index(p.layout, colA, nat, p.ld));
      const float b = hasB ? load_elem(p.w, p.dtype, elem_index(p.layout, colB, nat, p.ld)) : 0.f;
      buf[pad(s)] = make_float2(a, b);
      acc.x = __fadd_rn(acc.x, fabsf(a));
      acc.y = __fadd_rn(acc.y, fabsf(b));
    }
    float2 sum0 = team_sum<GenTeam>(acc, red, lt, parity);
    int sA = 0, sB = 0;
    {
      const bool finA = isfinite(sum0.x), finB = isfinite(sum0.y);
      if (lt == 0 && (!finA || !finB)) atomicOr(p.status, 1u);
      const float cA = __fdiv_rn(sum0.x, (float)n), cB = __fdiv_rn(sum0.y, (float)n);
      if (finA && cA > 0.f) sA = max(-100, min(100, -ilogbf(cA)));
      if (finB && cB > 0.f) sB = max(-100, min(100, -ilogbf(cB)));
    }
    const float scA = pow2f(sA), scB = pow2f(sB);
    const float isA = pow2f(-sA), isB = pow2f(-sB);
    const bool liveA = sum0.x > 0.f, liveB = sum0.y > 0.f;
    for (int s = lt; s < n; s += T) {
      const float2 x = buf[pad(s)];
      buf[pad(s)] = make_float2(__fmul_rn(x.x, scA), __fmul_rn(x.y, scB));
      uslot[s] = make_float2(0.f, 0.f);
    }
    sum0 = make_float2(__fmul_rn(sum0.x, scA), __fmul_rn(sum0.y, scB));
    float2 coef[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) coef[q] = make_float2(0.f, 0.f);

    int8_t* trA = nullptr;
    int8_t* trB = nullptr;
    if (TRACE) {
      trA = p.trace + colA * (int64_t)nsteps * n;
      trB = p.trace + colB * (int64_t)nsteps * n;
    }

    // one atomic greedy step on the pair's residual (see the per-length kernel)
    auto greedy = [&](int step, bool have_sum, bool upd_u) -> float2 {
      float2 sm = sum0;
      if (!have_sum) {
        float2 a = make_float2(0.f, 0.f);
        for (int s = lt; s < n; s += T) {
          const float2 r = buf[pad(s)];
          a.x = __fadd_rn(a.x, fabsf(r.x));
          a.y = __fadd_rn(a.y, fabsf(r.y));
        }
        sm = team_sum<GenTeam>(a, red, lt, parity);
      }
      const float lA = __fdiv_rn(sm.x, (float)n);
      const float lB = __fdiv_rn(sm.y, (float)n);
      for (int s = lt; s < n; s += T) {
        float2 r = buf[pad(s)];
        if (TRACE) {
          const int64_t off = (int64_t)step * n + gen_nat(s, n);
          trA[off] = (int8_t)((r.x > 0.f) - (r.x < 0.f));
          if (hasB) trB[off] = (int8_t)((r.y > 0.f) - (r.y < 0.f));
        }
        const float dA = signed_step(r.x, lA);
        const float dB = signed_step(r.y, lB);
        r.x = __fsub_rn(r.x, dA);
        r.y = __fsub_rn(r.y, dB);
        buf[pad(s)] = r;
        if (upd_u) {
          float2 uj = uslot[s];
          uj.x = __fadd_rn(uj.x, dA);
          uj.y = __fadd_rn(uj.y, dB);
          uslot[s] = uj;
        }
      }
      return make_float2(lA, lB);
    };

    int step = 0;
    const int HB = 2 * p.iters;
    for (int hb = 0; hb <= HB; ++hb) {
      if (hb == HB) {
        // r -> x - u - r: its P is vhat (P^2 = I)
        for (int s = lt; s < n; s += T) {
          const int nat = gen_nat(s, n);
          const float2 r = buf[pad(s)];
          if (p.resid) {
            p.resid[colA * n + nat] = __fmul_rn(r.x, isA);
            if (hasB) p.resid[colB * n + nat] = __fmul_rn(r.y, isB);
          }
          const float a = __fmul_rn(load_elem(p.w, p.dtype, elem_index(p.layout, colA, nat, p.ld)), scA);
          const float b = hasB ? __fmul_rn(load_elem(p.w, p.dtype, elem_index(p.layout, colB, nat, p.ld)), scB) : 0.f;
          const float2 uj = uslot[s];
          buf[pad(s)] = (p.iters == 0) ? make_float2(0.f, 0.f)
                                       : make_float2(__fsub_rn(__fsub_rn(a, uj.x), r.x), __fsub_rn(__fsub_rn(b, uj.y), r.y));
        }
        if (p.iters == 0) break;
      } else if ((hb & 1) == 0) {
        const float2 l1 = greedy(step++, hb == 0, true);
        const float2 l2 = greedy(step++, false, true);
        if (hb == 0) {
          coef[0] = l1;
          coef[1] = l2;
        }
      } else {
        const float2 l3 = greedy(step++, false, false);
        const float2 l4 = greedy(step++, false, false);
        if (hb == 1) {
          coef[2] = l3;
          coef[3] = l4;
        }
      }
      gen_apply(g, buf, tab, p.eps, lt);
      if (!liveA || !liveB) {
        for (int s = lt; s < n; s += T) {
          const float2 v = buf[pad(s)];
          buf[pad(s)] = make_float2(liveA ? v.x : 0.f, liveB ? v.y : 0.f);
        }
      }
    }
    // buf now holds vhat (own slots written last by this thread or read after a barrier)
    __syncthreads();

    if (p.u || p.vhat) {
      for (int s = lt; s < n; s += T) {
        const int nat = gen_nat(s, n);
        const float2 uj = uslot[s];
        const float2 vj = buf[pad(s)];
        if (p.u) {
          p.u[colA * n + nat] = __fmul_rn(uj.x, isA);
          if (hasB) p.u[colB * n + nat] = __fmul_rn(uj.y, isB);
        }
        if (p.vhat) {
          p.vhat[colA * n + nat] = __fmul_rn(vj.x, isA);
          if (hasB) p.vhat[colB * n + nat] = __fmul_rn(vj.y, isB);
        }
      }
    }

    // closed-form centres (Sec. 2.1) and boundaries, as in the per-length kernel
    float cen[2][2][4];
    float bnd[2][2][3];
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
          const float mm = fmaxf(a1[f][c], a2[f][c]);
          bnd[f][c][0] = -mm;
          bnd[f][c][1] = 0.f;
          bnd[f][c][2] = mm;
        }
    }
    auto code_of = [](float x, const float (&b)[3]) -> int { return (x > b[0]) + (x > b[1]) + (x > b[2]); };
    auto val = [&](int s, int f, int c) -> float {
      const float2 v = f ? buf[pad(s)] : uslot[s];
      return c ? v.y : v.x;
    };
    for (int it = 0; it < p.kmeans_iters; ++it) {
#pragma unroll
      for (int f = 0; f < 2; ++f) {
        // [c*8 + q]: sum above b_q; [c*8 + 3 + q]: count above b_q; [c*8 + 6]: total
        float acc16[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) acc16[i] = 0.f;
        for (int s = lt; s < n; s += T) {
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const float x = val(s, f, c);
            if (TRACE && (c == 0 || hasB))
              (c ? trB : trA)[(int64_t)(4 * p.iters + 2 * it + f) * n + gen_nat(s, n)] = (int8_t)code_of(x, bnd[f][c]);
            acc16[c * 8 + 6] = __fadd_rn(acc16[c * 8 + 6], x);
#pragma unroll
            for (int q = 0; q < 3; ++q) {
              const bool gt = x > bnd[f][c][q];
              acc16[c * 8 + q] = __fadd_rn(acc16[c * 8 + q], gt ? x : 0.f);
              acc16[c * 8 + 3 + q] = __fadd_rn(acc16[c * 8 + 3 + q], gt ? 1.f : 0.f);
            }
          }
        }
        float tot[16];
        team_sum_k<GenTeam, 16>(acc16, tot, reinterpret_cast<float*>(red), lt);
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const float* t = tot + c * 8;
          const float sum[4] = {__fsub_rn(t[6], t[0]), __fsub_rn(t[0], t[1]), __fsub_rn(t[1], t[2]), t[2]};
          const float cnt[4] = {__fsub_rn((float)n, t[3]), __fsub_rn(t[3], t[4]), __fsub_rn(t[4], t[5]), t[5]};
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            if (cnt[qq] > 0.f) cen[f][c][qq] = __fdiv_rn(sum[qq], cnt[qq]);
#pragma unroll
          for (int qq = 0; qq < 3; ++qq) bnd[f][c][qq] = __fmul_rn(0.5f, __fadd_rn(cen[f][c][qq], cen[f][c][qq + 1]));
        }
      }
    }

    // 2-bit codes: nearest centre (ties low), one byte per entry, packed 16 per word
    for (int s = lt; s < n; s += T) {
      const int nat = gen_nat(s, n);
      cb[0 * PS + nat] = (uint8_t)code_of(val(s, 0, 0), bnd[0][0]);
      cb[1 * PS + nat] = (uint8_t)code_of(val(s, 0, 1), bnd[0][1]);
      cb[2 * PS + nat] = (uint8_t)code_of(val(s, 1, 0), bnd[1][0]);
      cb[3 * PS + nat] = (uint8_t)code_of(val(s, 1, 1), bnd[1][1]);
    }
    for (int i = n + lt; i < PS; i += T) {
#pragma unroll
      for (int plane = 0; plane < 4; ++plane) cb[plane * PS + i] = 0;
    }
    __syncthreads();
    for (int wi = lt; wi < 4 * WPV; wi += T) {
      const int plane = wi / WPV;
      const int word = wi - plane * WPV;
      const bool isB = (plane & 1) != 0;
      if (isB && !hasB) continue;
      const uint4 q = *reinterpret_cast<const uint4*>(cb + plane * PS + word * 16);
      const uint32_t qq[4] = {q.x, q.y, q.z, q.w};
      uint32_t packed = 0;
#pragma unroll
      for (int b4 = 0; b4 < 4; ++b4) {
#pragma unroll
        for (int by = 0; by < 4; ++by) packed |= ((qq[b4] >> (8 * by)) & 3u) << (2 * (4 * b4 + by));
      }
      uint32_t* dst = (plane < 2) ? p.codes_u : p.codes_v;
      dst[(isB ? colB : colA) * WPV + word] = packed;
    }
    if (lt == 0) {
      const float sc[2] = {isA, isB};
      for (int v2 = 0; v2 < (hasB ? 2 : 1); ++v2) {
        const int64_t col = v2 ? colB : colA;
        const float f = sc[v2];
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          p.centres_u[col * 4 + qq] = __fmul_rn(cen[0][v2][qq], f);
          p.centres_v[col * 4 + qq] = __fmul_rn(cen[1][v2][qq], f);
        }
        if (p.coeffs) {
          float* co = p.coeffs + col * 4;
          co[0] = __fmul_rn(v2 ? coef[0].y : coef[0].x, f);
          co[1] = __fmul_rn(v2 ? coef[1].y : coef[1].x, f);
          co[2] = __fmul_rn(v2 ? coef[2].y : coef[2].x, f);
          co[3] = __fmul_rn(v2 ? coef[3].y : coef[3].x, f);
        }
      }
    }
    __syncthreads();  // buf and the code bytes are reused by the next pair
  }
}

// y_j = P x_j (fp32, vector-major rows of length n)
__global__ void __launch_bounds__(kGenThreads, 2) gen_apply_kernel(ApplyParams p, const __grid_constant__ GenPlan g) {
  extern __shared__ __align__(16) float2 smem[];
  constexpr int T = kGenThreads;
  const int n = g.n;
  const int lt = threadIdx.x;
  float2* buf = smem;
  for (int64_t pr = blockIdx.x; pr < p.npairs; pr += gridDim.x) {
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < p.m;
    for (int s = lt; s < n; s += T) {
      const int nat = gen_nat(s, n);
      buf[pad(s)] = make_float2(__ldg(&p.x[colA * n + nat]), hasB ? __ldg(&p.x[(colA + 1) * n + nat]) : 0.f);
    }
    gen_apply(g, buf, p.twt, p.eps, lt);  // its first barrier orders every load before any store (x, y may alias)
    for (int s = lt; s < n; s += T) {
      const int nat = gen_nat(s, n);
      const float2 v = buf[pad(s)];
      p.y[colA * n + nat] = v.x;
      if (hasB) p.y[(colA + 1) * n + nat] = v.y;
    }
    __syncthreads();
  }
}

// W_hat_j = cu_j[code_u] + P(cv_j[code_v])  (App. C)
__global__ void __launch_bounds__(kGenThreads, 2) gen_reconstruct_kernel(RecParams p, const __grid_constant__ GenPlan g) {
  extern __shared__ __align__(16) float2 smem[];
  constexpr int T = kGenThreads;
  const int n = g.n;
  const int WPV = (n + 15) / 16;
  const int lt = threadIdx.x;
  float2* buf = smem;
  auto pick = [](const float4& c, uint32_t q) -> float {
    const float lo = (q & 1u) ? c.y : c.x;
    const float hi = (q & 1u) ? c.w : c.z;
    return (q & 2u) ? hi : lo;
  };
  for (int64_t pr = blockIdx.x; pr < p.npairs; pr += gridDim.x) {
    const int64_t colA = 2 * pr;
    const bool hasB = (colA + 1) < p.m;
    const int64_t colB = hasB ? colA + 1 : colA;
    const float4 cuA = __ldg(reinterpret_cast<const float4*>(p.centres_u) + colA);
    const float4 cuB = __ldg(reinterpret_cast<const float4*>(p.centres_u) + colB);
    const float4 cvA = __ldg(reinterpret_cast<const float4*>(p.centres_v) + colA);
    const float4 cvB = __ldg(reinterpret_cast<const float4*>(p.centres_v) + colB);
    auto code = [&](const uint32_t* planes, int64_t col, int nat) -> uint32_t {
      return (__ldg(&planes[col * WPV + (nat >> 4)]) >> (2 * (nat & 15))) & 3u;
    };
    for (int s = lt; s < n; s += T) {
      const int nat = gen_nat(s, n);
      buf[pad(s)] = make_float2(pick(cvA, code(p.codes_v, colA, nat)), pick(cvB, code(p.codes_v, colB, nat)));
    }
    gen_apply(g, buf, p.twt, p.eps, lt);
    for (int nat = lt; nat < n; nat += T) {
      const float2 v = buf[pad(gen_slot(nat, n))];
      const float a = __fadd_rn(pick(cuA, code(p.codes_u, colA, nat)), v.x);
      store_elem(p.out, p.dtype, elem_index(p.layout, colA, nat, p.ld), a);
      if (hasB) {
        const float b = __fadd_rn(pick(cuB, code(p.codes_u, colB, nat)), v.y);
        store_elem(p.out, p.dtype, elem_index(p.layout, colB, nat, p.ld), b);
      }
    }
    __syncthreads();
  }
}

// Tables of one call: pass twiddles, exp(i pi k/n), frequency slots, sign bits
// (SplitMix64, as the per-length set-up) and the cleared status word.
__global__ void gen_setup_kernel(float2* tab, uint32_t* eps, uint32_t* status, uint64_t seed,
                                 const __grid_constant__ GenPlan g) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int stride = gridDim.x * blockDim.x;
  const int n = g.n;
  if (tid == 0) *status = 0u;
  for (int e = tid; e < g.woff; e += stride) {
    int i = 0;
    while (i + 1 < g.np - 1 && e >= g.tw[i + 1]) ++i;
    const int r = e - g.tw[i];
    const int sp = r % g.S[i], j = r / g.S[i];
    tab[e] = root_w((long long)sp * j, g.B[i]);
  }
  for (int k = tid; 2 * k <= n; k += stride) tab[g.woff + k] = expi_pi(k, n);
  int* perm = reinterpret_cast<int*>(tab + g.permoff);
  for (int k = tid; k < n; k += stride) {
    int x = k, s = 0;
    for (int i = 0; i < g.np; ++i) {
      s += (x % g.R[i]) * g.S[i];
      x /= g.R[i];
    }
    perm[k] = s;
  }
  const int words = (n + 31) / 32;
  for (int wd = tid; wd < words; wd += stride) {
    uint32_t bits = 0;
    for (int bb = 0; bb < 32; ++bb) {
      const int j = wd * 32 + bb;
      if (j >= n) break;
      bits |= (uint32_t)(splitmix64_mix(seed + (uint64_t)(j + 1) * 0x9E3779B97F4A7C15ull) >> 63) << bb;
    }
    eps[wd] = bits;
  }
}

// ---------------------------------------------------------------------------
// Host side: PlanOps for one run-time length
// ---------------------------------------------------------------------------
template <class K>
int gen_occupancy(K kernel, int64_t n) {
  const size_t smem = gen_smem(n);
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) return 0;
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, kGenThreads, smem) != cudaSuccess) return 0;
  return nb;
}

int gen_ctas(int which, int64_t n) {
  if (which == 0) return gen_occupancy(gen_decompose_kernel<false>, n);
  if (which == 1) return gen_occupancy(gen_apply_kernel, n);
  return gen_occupancy(gen_reconstruct_kernel, n);
}

cudaError_t gen_decompose(const DecParams& p, const BatchParams* bp, int grid, cudaStream_t s) {
  GenPlan g;
  if (bp || !gen_plan(p.n, &g)) return cudaErrorInvalidValue;
  auto k = p.trace ? gen_decompose_kernel<true> : gen_decompose_kernel<false>;
  const size_t smem = gen_smem(p.n);
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<grid, kGenThreads, smem, s>>>(p, g);
  return cudaGetLastError();
}

cudaError_t gen_apply_launch(const ApplyParams& p, const ApplyBatch*, int grid, cudaStream_t s) {
  GenPlan g;
  if (!gen_plan(p.n, &g)) return cudaErrorInvalidValue;
  const size_t smem = gen_smem(p.n);
  cudaError_t e = cudaFuncSetAttribute(gen_apply_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  gen_apply_kernel<<<grid, kGenThreads, smem, s>>>(p, g);
  return cudaGetLastError();
}

cudaError_t gen_reconstruct(const RecParams& p, const RecBatch* rb, int grid, cudaStream_t s) {
  GenPlan g;
  if (rb || !gen_plan(p.n, &g)) return cudaErrorInvalidValue;
  const size_t smem = gen_smem(p.n);
  cudaError_t e = cudaFuncSetAttribute(gen_reconstruct_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  gen_reconstruct_kernel<<<grid, kGenThreads, smem, s>>>(p, g);
  return cudaGetLastError();
}

cudaError_t gen_setup(float2* tab, uint32_t* eps, uint32_t* status, uint64_t seed, int64_t n, cudaStream_t s) {
  GenPlan g;
  if (!gen_plan(n, &g)) return cudaErrorInvalidValue;
  const int work = g.twn > n ? g.twn : (int)n;
  const int blocks = (work + 255) / 256;
  gen_setup_kernel<<<blocks, 256, 0, s>>>(tab, eps, status, seed, g);
  return cudaGetLastError();
}

}  // namespace

bool generic_length(int64_t n) {
  GenPlan g;
  return gen_plan(n, &g);
}

const PlanOps* generic_plan_ops(int64_t n) {
  GenPlan g;
  if (!gen_plan(n, &g)) return nullptr;
  static std::mutex mu;
  static std::map<int64_t, PlanOps> cache;  // node addresses stay valid
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(n);
  if (it != cache.end()) return &it->second;
  const PlanOps o{(int)n, kGenThreads, 1, gen_smem(n), true, false, g.twn,
                  &gen_ctas, &gen_decompose, &gen_apply_launch, &gen_reconstruct, &gen_setup};
  return &cache.emplace(n, o).first->second;
}

}  // namespace kd
