// Kernel instantiations for vector length N = 11008.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_11008() { return Ops<Plan11008>::ops(); }
}  // namespace kd
