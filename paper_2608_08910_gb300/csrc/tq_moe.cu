// Mixture-of-experts entry points (work in progress).
#include "tq_launch.h"
#include "tqfx4.h"

extern "C" {
size_t tqfx4_moe_workspace_bytes(const tqfx4_experts *, const tqfx4_router *, int64_t, int) { return 0; }
tqfx4_status tqfx4_moe_ffn(const tqfx4_experts *, const tqfx4_router *, const float *, float *, int32_t *,
                           float *, void *, size_t, void *) { return TQFX4_EINVAL; }
tqfx4_status tqfx4_moe_grouped(const tqfx4_experts *, const tqfx4_router *, const float *, int64_t, float *,
                               int32_t *, float *, int, void *, size_t, void *) { return TQFX4_EINVAL; }
int tqfx4_moe_stage_count(int, int) { return 0; }
const char *tqfx4_moe_stage_name(int, int, int) { return ""; }
tqfx4_status tqfx4_moe_ffn_traced(const tqfx4_experts *, const tqfx4_router *, const float *, float *,
                                  int32_t *, float *, void *, size_t, void *, void *const *) {
    return TQFX4_EINVAL;
}
tqfx4_status tqfx4_moe_grouped_traced(const tqfx4_experts *, const tqfx4_router *, const float *, int64_t,
                                      float *, int32_t *, float *, int, void *, size_t, void *,
                                      void *const *) {
    return TQFX4_EINVAL;
}
tqfx4_status tqfx4_moe_workspace_views(const tqfx4_experts *, const tqfx4_router *, int64_t, int, int,
                                       tqfx4_moe_views *) {
    return TQFX4_EINVAL;
}
}
