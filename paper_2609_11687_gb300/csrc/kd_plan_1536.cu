// Kernel instantiations for vector length N = 1536.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_1536() { return Ops<Plan1536>::ops(); }
}  // namespace kd
