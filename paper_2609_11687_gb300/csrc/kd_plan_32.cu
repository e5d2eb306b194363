// Kernel instantiations for vector length N = 32.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_32() { return Ops<Plan32>::ops(); }
}  // namespace kd
