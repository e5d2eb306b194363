// Kernel instantiations for vector length N = 16.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_16() { return Ops<Plan16>::ops(); }
}  // namespace kd
