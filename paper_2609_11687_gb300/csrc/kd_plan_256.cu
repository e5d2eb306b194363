// Kernel instantiations for vector length N = 256.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_256() { return Ops<Plan256>::ops(); }
}  // namespace kd
