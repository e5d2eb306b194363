// Kernel instantiations for vector length N = 128.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_128() { return Ops<Plan128>::ops(); }
}  // namespace kd
