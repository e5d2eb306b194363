// Transform plans per supported vector length N.
//   Plan<N, T, Q, u-storage, min CTAs per SM, radices...>
//   T threads own one vector pair (E = R0 complex values each, positions t + j*T);
//   Q pairs per CTA (Q > 1 only when a team fits in one warp).
//   Plans whose last radix equals the first (one last-pass group per thread) apply
//   the middle operator in registers (Plan::PAIRED).
#pragma once
#include "kd_kernels.cuh"

namespace kd {
using Plan16 = Plan<16, 4, 8, UREG, 8, 4, 4>;
using Plan32 = Plan<32, 4, 8, UREG, 8, 8, 4>;
using Plan64 = Plan<64, 8, 4, UREG, 8, 8, 8>;
using Plan128 = Plan<128, 8, 4, UREG, 8, 16, 8>;
using Plan256 = Plan<256, 16, 4, USMEM, 8, 16, 16>;
using Plan512 = Plan<512, 32, 2, USMEM, 8, 16, 32>;
using Plan768 = Plan<768, 32, 2, USMEM, 6, 24, 32>;
using Plan1024 = Plan<1024, 64, 1, USMEM, 8, 16, 8, 8>;
using Plan1536 = Plan<1536, 96, 1, USMEM, 5, 16, 12, 8>;
using Plan2048 = Plan<2048, 128, 1, USMEM, 4, 16, 16, 8>;
using Plan3072 = Plan<3072, 192, 1, USMEM, 2, 16, 12, 16>;
using Plan4096 = Plan<4096, 256, 1, USMEM, 2, 16, 16, 16>;
using Plan8192 = Plan<8192, 512, 1, USMEM, 1, 16, 32, 16>;
// u (88 KB) in shared memory; the twiddle table then no longer fits beside it and
// is read through L1/L2
using Plan11008 = Plan<11008, 256, 1, USMEM, 1, 43, 16, 16>;
using Plan14336 = Plan<14336, 512, 1, UGMEM, 1, 28, 16, 32>;
using Plan16384 = Plan<16384, 512, 1, UGMEM, 1, 32, 32, 16>;

// packed constant roots (2.5 % faster at n = 4096; at n = 11008 the constant pairs
// cost spills and 9 %)
template <>
struct PackedRoots<Plan4096> {
  static constexpr bool value = true;
};
}  // namespace kd
