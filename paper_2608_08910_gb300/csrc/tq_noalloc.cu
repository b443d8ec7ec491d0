// tqfx4_moe_ffn_noalloc: the one-token MoE layer of tqfx4_moe_ffn for callers
// that cannot allocate device memory, running on a scratch area that the
// library itself holds as a file-scope device array.
#include <cstdio>

#include "tq_launch.h"
#include "tq_moe_common.cuh"
#include "tqfx4.h"

namespace {

// The scratch every call uses (workspace of tqfx4_moe_ffn). Each GPU that
// loads the library holds these bytes until the process exits.
__device__ __align__(256) unsigned char g_noalloc_scratch[TQFX4_NOALLOC_SCRATCH_BYTES];

}  // namespace

extern "C" tqfx4_status tqfx4_moe_ffn_noalloc(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x,
                                              float *out, int32_t *sel_idx, float *sel_w, void *stream) {
    if (tqfx4_moe_workspace_bytes(ex, rt, 1, TQFX4_PATH_AUTO) == 0)
        return tqfx4_moe_ffn(ex, rt, x, out, sel_idx, sel_w, nullptr, 0, stream);  // reports the shape error
    // the bound tqfx4_moe_ffn checks: the one-token (decode) layout
    const tq::MoeLayout L = tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, 1, false, true);
    if (L.total > TQFX4_NOALLOC_SCRATCH_BYTES) {
        char msg[200];
        snprintf(msg, sizeof(msg),
                 "tqfx4_moe_ffn_noalloc: these shapes need %zu bytes of scratch; the library holds %d "
                 "(use tqfx4_moe_ffn with a caller workspace)",
                 L.total, TQFX4_NOALLOC_SCRATCH_BYTES);
        return tq::api_fail(TQFX4_EWORKSPACE, msg);
    }
    // In host code g_noalloc_scratch only names a host-side stand-in; the
    // device address is looked up in the current context on every call (no
    // cached copy), so it stays right after a device reset, which reloads
    // the library's device code, and under a context other than the
    // device's primary one.
    void *ws = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ws, g_noalloc_scratch);
    if (e != cudaSuccess || !ws)
        return tq::api_fail(TQFX4_ECUDA, "tqfx4_moe_ffn_noalloc: cudaGetSymbolAddress failed");
    // The status word and the counters must start every call at zero; the
    // rest of the scratch is fully rewritten by the call.
    e = cudaMemsetAsync(ws, 0, L.ctr + 4 * L.n_ctr, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return tq::api_fail(TQFX4_ECUDA, "tqfx4_moe_ffn_noalloc: clearing the scratch failed");
    return tqfx4_moe_ffn(ex, rt, x, out, sel_idx, sel_w, ws, TQFX4_NOALLOC_SCRATCH_BYTES, stream);
}
