// Kernel instantiations for vector length N = 2048.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_2048() { return Ops<Plan2048>::ops(); }
}  // namespace kd
