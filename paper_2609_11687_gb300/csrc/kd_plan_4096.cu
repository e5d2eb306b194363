// Kernel instantiations for vector length N = 4096.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_4096() { return Ops<Plan4096>::ops(); }
}  // namespace kd
