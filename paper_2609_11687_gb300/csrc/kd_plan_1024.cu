// Kernel instantiations for vector length N = 1024.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_1024() { return Ops<Plan1024>::ops(); }
}  // namespace kd
