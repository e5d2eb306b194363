// Kernel instantiations for vector length N = 512.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_512() { return Ops<Plan512>::ops(); }
}  // namespace kd
