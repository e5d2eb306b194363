// Kernel instantiations for vector length N = 768.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_768() { return Ops<Plan768>::ops(); }
}  // namespace kd
