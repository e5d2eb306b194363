// Kernel instantiations for vector length N = 64.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_64() { return Ops<Plan64>::ops(); }
}  // namespace kd
