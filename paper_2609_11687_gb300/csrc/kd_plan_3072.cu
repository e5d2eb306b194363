// Kernel instantiations for vector length N = 3072.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_3072() { return Ops<Plan3072>::ops(); }
}  // namespace kd
