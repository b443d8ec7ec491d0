// Host-side launchers of the tqfx4 kernels (internal to libtqfx4; the public
// interface is include/tqfx4.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tqfx4.h"

namespace tq {

int num_sms();
int max_smem_optin();
cudaError_t allow_max_smem(const void *kernel, unsigned char *flags);

cudaError_t launch_pack(int src, const void *a, const int8_t *t2, const uint16_t *scales, int64_t n, int64_t k,
                        void *blocks, int *status, cudaStream_t st);
cudaError_t launch_validate(const void *blocks, int64_t n, int64_t k, int *status, cudaStream_t st);
cudaError_t launch_quantize(const float *x, int64_t m, int64_t k, int8_t *q, float *da, int32_t *bsum,
                            int *status, cudaStream_t st);
cudaError_t launch_gemv_x(const void *blocks, int64_t n, int64_t k, const float *x, int8_t *q, float *da,
                          int32_t *bsum, float *y, int *status, cudaStream_t st);
cudaError_t launch_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                        const int32_t *bsum, float *y, int32_t *block_sums, int *status, cudaStream_t st);

tqfx4_status api_fail(tqfx4_status s, const char *msg);

struct MoeArgs;
struct MoeLayout;
bool moe_decode_args(const tqfx4_experts *ex, const tqfx4_router *rt, void *ws, MoeArgs &a, MoeLayout &L);
cudaError_t launch_copy_f32(float *dst, const float *src, int64_t n, cudaStream_t st);
cudaError_t launch_moe_decode(const MoeArgs &a, const float *x, float *out, int32_t *sel_idx, float *sel_w,
                              cudaStream_t st, void *const *events);
int gate_up_smem(const MoeArgs &a);
int64_t mxfp4_bytes(int64_t n, int64_t k);
cudaError_t launch_mxfp4_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                              int32_t *block_sums, int *status, cudaStream_t st);
// Records a stage event on `st`; inside a stream capture it becomes an
// external event node, so that the event keeps its timing meaning on replay.
inline cudaError_t record_stage_event(cudaEvent_t ev, cudaStream_t st) {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    cudaStreamIsCapturing(st, &cap);
    return cudaEventRecordWithFlags(ev, st, cap == cudaStreamCaptureStatusActive ? cudaEventRecordExternal
                                                                                  : cudaEventRecordDefault);
}
int mxfp4_gemv_smem(int64_t k, int acts);
int64_t free_bytes(int64_t n, int64_t k);
int gemv_free_smem(int64_t k);
cudaError_t launch_pack_free(const int8_t *t1, const int8_t *t2, const uint16_t *a1, const uint16_t *a2, int64_t n,
                             int64_t k, void *out, int *status, cudaStream_t st);
cudaError_t launch_gemv_free(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                             const int32_t *bsum, float *y, int32_t *S1, int32_t *S2, int *status, cudaStream_t st);
cudaError_t launch_moe_mxfp4_experts(const MoeArgs &a, float *out, cudaStream_t st, const cudaEvent_t *ev);
cudaError_t launch_moe_route(const MoeArgs &a, const float *x, int32_t *sel_idx, float *sel_w, cudaStream_t st);
cudaError_t launch_moe_experts(const MoeArgs &a, const void *const *ptrs, float *out, cudaStream_t st);
cudaError_t launch_expert_ffn(const MoeArgs &a, const float *x, float *out, cudaStream_t st, void *const *events);
bool expert_ffn_one_launch(const MoeArgs &a);  // launch_expert_ffn takes the one-launch kernel

struct GroupedArgs;
bool grouped_args(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t T, void *ws, GroupedArgs &a,
                  MoeLayout &L);
cudaError_t launch_moe_grouped(const GroupedArgs &a, const float *X, float *OUT, int32_t *sel_idx, float *sel_w,
                               cudaStream_t st, void *const *events);
cudaError_t launch_tc_gemm(const GroupedArgs &a, bool down, cudaStream_t st);
// Largest chunk (pairs) the streaming small-group pass takes for these
// shapes and buffers, 0 if it takes none; the pass itself, run after the
// tensor-core pass of the same projection.
int small_groups_max(const GroupedArgs &a);
cudaError_t launch_small_groups(const GroupedArgs &a, bool down, cudaStream_t st);
int grouped_stage_count();
const char *grouped_stage_name(int s);
int down_smem(const MoeArgs &a);
cudaError_t launch_selftest_timeout(int *status, cudaStream_t st);

// kernel<<<grid, block, smem, st>>>(args...) as a programmatic dependent of
// the previous kernel in the stream: its CTAs may become resident while that
// kernel drains. Every kernel launched this way executes griddepcontrol.wait
// before its first access to global memory, so the order of the stream
// holds.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                    Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

}  // namespace tq
