// bf16-replica instances of the fused synchronisation pass.
#include "aloco_sync_kernel.cuh"

namespace aloco {
cudaError_t plan_sync_bf16(int M, int64_t work_items, int sm_count,
                           int blocks_per_sm, LaunchPlan *plan) {
    return plan_dispatch<true>(M, work_items, sm_count, blocks_per_sm, plan);
}
}  // namespace aloco
