// Kernel instantiations for vector length N = 14336.
#include "kd_launch.cuh"
#include "kd_plans.cuh"

namespace kd {
const PlanOps* plan_ops_14336() { return Ops<Plan14336>::ops(); }
}  // namespace kd
