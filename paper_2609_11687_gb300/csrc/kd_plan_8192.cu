// Kernel instantiations for vector length N = 8192.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_8192() { return Ops<Plan8192>::ops(); }
}  // namespace kd
