// fp32-replica instances of the bulk-copy synchronisation pass.
#include "aloco_sync_tma.cuh"

namespace aloco {
cudaError_t plan_sync_tma_f32(int M, int64_t nvec, int sm_count,
                              LaunchPlan *plan) {
    return plan_tma_dispatch<false>(M, nvec, sm_count, kTmaSmemBudget, plan);
}
}  // namespace aloco
