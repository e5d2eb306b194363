// Kernel instantiations for vector length N = 16384.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_16384() { return Ops<Plan16384>::ops(); }
}  // namespace kd
