// C ABI of libtqfx4 (declared in include/tqfx4.h): argument checks on the
// host, then asynchronous launches on the caller's stream.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include <nvtx3/nvToolsExt.h>

#include "tq_launch.h"
#include "tq_moe_common.cuh"
#include "tqfx4.h"

namespace {

// One NVTX range per call that enqueues work, named after the entry point,
// so that a profiler shows the library's calls on the host timeline (the
// header-only NVTX API returns at once when no tool is attached).
struct TqRange {
    explicit TqRange(const char *name) { nvtxRangePushA(name); }
    ~TqRange() { nvtxRangePop(); }
    TqRange(const TqRange &) = delete;
    TqRange &operator=(const TqRange &) = delete;
};
#define TQ_RANGE() TqRange tq_range_(__func__)

thread_local char g_err[512] = "";

tqfx4_status fail(tqfx4_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

tqfx4_status ok() {
    g_err[0] = '\0';
    return TQFX4_OK;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// The debug build (TQFX4_DEBUG) checks every tq2_0_fx4 matrix an entry point
// reads against the format before its kernels run; the release build does
// nothing here.
cudaError_t debug_validate(const void *blocks, int64_t n, int64_t k, void *ws, void *stream) {
#ifdef TQFX4_DEBUG
    if (!blocks || n <= 0 || k <= 0) return cudaSuccess;
    return tq::launch_validate(blocks, n, k, static_cast<int *>(ws), static_cast<cudaStream_t>(stream));
#else
    (void)blocks, (void)n, (void)k, (void)ws, (void)stream;
    return cudaSuccess;
#endif
}

// The device address of page-locked host memory (the same pointer under
// unified addressing), or null for pageable memory or an unaligned pointer.
static void *mapped(const void *host, size_t align) {
    if (!host || reinterpret_cast<uintptr_t>(host) % align) return nullptr;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, host) != cudaSuccess) {
        cudaGetLastError();  // not sticky: clear it for the launches that follow
        return nullptr;
    }
    return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}


tqfx4_status cuda_fail(cudaError_t e, const char *what) {
    return fail(TQFX4_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

tqfx4_status check_ws(void *ws, size_t ws_bytes, size_t need, const char *fn) {
    if (!ws) return fail(TQFX4_EINVAL, "%s: workspace is NULL", fn);
    if (!aligned(ws, 256)) return fail(TQFX4_EALIGN, "%s: workspace must be 256-byte aligned", fn);
    if (ws_bytes < need)
        return fail(TQFX4_EWORKSPACE, "%s: workspace has %zu bytes, needs %zu", fn, ws_bytes, need);
    return TQFX4_OK;
}

tqfx4_status check_nk(int64_t n, int64_t k, const char *fn) {
    if (n < 0 || k < 0) return fail(TQFX4_EINVAL, "%s: negative size (n=%lld, k=%lld)", fn, (long long)n, (long long)k);
    if (n % 4) return fail(TQFX4_ESHAPE, "%s: n=%lld is not a multiple of 4", fn, (long long)n);
    if (k % 256) return fail(TQFX4_ESHAPE, "%s: k=%lld is not a multiple of 256", fn, (long long)k);
    return TQFX4_OK;
}

}  // namespace

namespace tq {
// Record a failure message for tqfx4_last_error() from other translation
// units of the library.
tqfx4_status api_fail(tqfx4_status s, const char *msg) { return fail(s, "%s", msg); }
}  // namespace tq

extern "C" {

int64_t tqfx4_matrix_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || n % 4 || k % 256) return -1;
    return (n / 4) * (k / 256) * 520;
}

size_t tqfx4_basic_workspace_bytes(void) { return TQFX4_STATUS_BYTES; }

tqfx4_status tqfx4_pack(int src, const void *a, const int8_t *t2, const uint16_t *scales_f16, int64_t n,
                        int64_t k, void *blocks, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    tqfx4_status s = check_nk(n, k, "tqfx4_pack");
    if (s) return s;
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, "tqfx4_pack"))) return s;
    if (n == 0 || k == 0) return ok();
    if (!a || !blocks) return fail(TQFX4_EINVAL, "tqfx4_pack: NULL input or output");
    if (!aligned(blocks, 16)) return fail(TQFX4_EALIGN, "tqfx4_pack: blocks must be 16-byte aligned");
    if (src == TQFX4_SRC_F32_RTN || src == TQFX4_SRC_F32_TIED) {
        if (t2 || scales_f16) return fail(TQFX4_EINVAL, "tqfx4_pack: t2/scales must be NULL for F32 sources");
        if (!aligned(a, 16)) return fail(TQFX4_EALIGN, "tqfx4_pack: W must be 16-byte aligned");
    } else if (src == TQFX4_SRC_TRITS) {
        if (!t2 || !scales_f16) return fail(TQFX4_EINVAL, "tqfx4_pack: TRITS needs t2 and scales");
        if (!aligned(a, 16) || !aligned(t2, 16) || !aligned(scales_f16, 2))
            return fail(TQFX4_EALIGN, "tqfx4_pack: t1/t2 must be 16-byte aligned");
    } else {
        return fail(TQFX4_EINVAL, "tqfx4_pack: unknown source %d", src);
    }
    cudaError_t e = tq::launch_pack(src, a, t2, scales_f16, n, k, blocks, static_cast<int *>(ws),
                                    static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_pack");
    return ok();
}

tqfx4_status tqfx4_quantize_act(const float *x, int64_t m, int64_t k, int8_t *q, float *da, int32_t *bsum,
                                void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    tqfx4_status s = check_nk(0, k, "tqfx4_quantize_act");
    if (s) return s;
    if (m < 0) return fail(TQFX4_EINVAL, "tqfx4_quantize_act: negative m");
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, "tqfx4_quantize_act"))) return s;
    if (m == 0 || k == 0) return ok();
    if (!x || !q || !da || !bsum) return fail(TQFX4_EINVAL, "tqfx4_quantize_act: NULL pointer");
    if (!aligned(x, 16) || !aligned(q, 16) || !aligned(da, 4) || !aligned(bsum, 4))
        return fail(TQFX4_EALIGN, "tqfx4_quantize_act: x and q must be 16-byte aligned");
    cudaError_t e = tq::launch_quantize(x, m, k, q, da, bsum, static_cast<int *>(ws),
                                        static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_quantize_act");
    return ok();
}

tqfx4_status tqfx4_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                        const int32_t *bsum, float *y, int32_t *block_sums, void *ws, size_t ws_bytes,
                        void *stream) {
    TQ_RANGE();
    tqfx4_status s = check_nk(n, k, "tqfx4_gemv");
    if (s) return s;
    if (k > TQFX4_MAX_K) return fail(TQFX4_ESHAPE, "tqfx4_gemv: k=%lld exceeds %d", (long long)k, TQFX4_MAX_K);
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, "tqfx4_gemv"))) return s;
    if (n == 0) return ok();
    if (!y) return fail(TQFX4_EINVAL, "tqfx4_gemv: y is NULL");
    if (k > 0 && (!blocks || !q || !da || !bsum)) return fail(TQFX4_EINVAL, "tqfx4_gemv: NULL input");
    if (k > 0 && (!aligned(blocks, 16) || !aligned(q, 16) || !aligned(da, 4) || !aligned(bsum, 4)))
        return fail(TQFX4_EALIGN, "tqfx4_gemv: blocks and q must be 16-byte aligned");
    if (!aligned(y, 4) || !aligned(block_sums, 4)) return fail(TQFX4_EALIGN, "tqfx4_gemv: misaligned output");
    cudaError_t e = debug_validate(blocks, n, k, ws, stream);
    if (e == cudaSuccess)
        e = tq::launch_gemv(blocks, n, k, q, da, bsum, y, block_sums, static_cast<int *>(ws),
                            static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_gemv");
    return ok();
}

tqfx4_status tqfx4_gemv_x(const void *blocks, int64_t n, int64_t k, const float *x, float *y, int8_t *q, float *da,
                          int32_t *bsum, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_gemv_x";
    tqfx4_status s = check_nk(n, k, fn);
    if (s) return s;
    if (k == 0 || k % 512 || k > TQFX4_MAX_K)
        return fail(TQFX4_ESHAPE, "%s: k=%lld must be a multiple of 512 in 512..%d", fn, (long long)k, TQFX4_MAX_K);
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, fn))) return s;
    if (n == 0) return ok();
    if (!blocks || !x || !y) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    if ((q == nullptr) != (da == nullptr) || (q == nullptr) != (bsum == nullptr))
        return fail(TQFX4_EINVAL, "%s: q, da and bsum all or none", fn);
    if (!aligned(blocks, 16) || !aligned(x, 16) || !aligned(y, 4) || !aligned(q, 16) || !aligned(da, 4) ||
        !aligned(bsum, 4))
        return fail(TQFX4_EALIGN, "%s: blocks, x and q must be 16-byte aligned", fn);
    cudaError_t e = debug_validate(blocks, n, k, ws, stream);
    if (e == cudaSuccess)
        e = tq::launch_gemv_x(blocks, n, k, x, q, da, bsum, y, static_cast<int *>(ws),
                              static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

size_t tqfx4_gemv_x_host_workspace_bytes(int64_t n, int64_t k) {
    if (n < 0 || k <= 0 || k % 512 || k > TQFX4_MAX_K || n % 4) return 0;
    return tq::align256(tq::align256(TQFX4_STATUS_BYTES + 4 * static_cast<size_t>(k)) + 4 * static_cast<size_t>(n));
}

tqfx4_status tqfx4_gemv_x_host(const void *blocks, int64_t n, int64_t k, const float *x_host, float *y_host,
                               void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_gemv_x_host";
    tqfx4_status s = check_nk(n, k, fn);
    if (s) return s;
    const size_t need = tqfx4_gemv_x_host_workspace_bytes(n, k);
    if (need == 0)
        return fail(TQFX4_ESHAPE, "%s: k=%lld must be a multiple of 512 in 512..%d", fn, (long long)k, TQFX4_MAX_K);
    if ((s = check_ws(ws, ws_bytes, need, fn))) return s;
    if (n == 0) return ok();
    if (!blocks || !x_host || !y_host) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    // page-locked buffers in place (the kernel reads x and writes y through
    // their device addresses); others through staging after the status word
    uint8_t *base = static_cast<uint8_t *>(ws);
    float *xd = reinterpret_cast<float *>(base + TQFX4_STATUS_BYTES);
    float *yd = reinterpret_cast<float *>(base + tq::align256(TQFX4_STATUS_BYTES + 4 * static_cast<size_t>(k)));
    const float *xm = static_cast<const float *>(mapped(x_host, 16));
    float *ym = static_cast<float *>(mapped(y_host, 4));
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    if (!xm) e = cudaMemcpyAsync(xd, x_host, 4 * static_cast<size_t>(k), cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    if ((s = tqfx4_gemv_x(blocks, n, k, xm ? xm : xd, ym ? ym : yd, nullptr, nullptr, nullptr, ws, ws_bytes,
                          stream)))
        return s;
    if (!ym) e = cudaMemcpyAsync(y_host, yd, 4 * static_cast<size_t>(n), cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_validate_blocks(const void *blocks, int64_t n, int64_t k, void *ws, size_t ws_bytes,
                                   void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_validate_blocks";
    tqfx4_status s = check_nk(n, k, fn);
    if (s) return s;
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, fn))) return s;
    if (n == 0 || k == 0) return ok();
    if (!blocks) return fail(TQFX4_EINVAL, "%s: NULL blocks", fn);
    if (!aligned(blocks, 16)) return fail(TQFX4_EALIGN, "%s: blocks must be 16-byte aligned", fn);
    cudaError_t e = tq::launch_validate(blocks, n, k, static_cast<int *>(ws), static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

int64_t tqfx4_free_bytes(int64_t n, int64_t k) { return tq::free_bytes(n, k); }

tqfx4_status tqfx4_pack_free(const int8_t *t1, const int8_t *t2, const uint16_t *a1_f16, const uint16_t *a2_f16,
                             int64_t n, int64_t k, void *blocks, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_pack_free";
    tqfx4_status s = check_nk(n, k, fn);
    if (s) return s;
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, fn))) return s;
    if (n == 0 || k == 0) return ok();
    if (!t1 || !t2 || !a1_f16 || !a2_f16 || !blocks) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    if (!aligned(t1, 16) || !aligned(t2, 16) || !aligned(a1_f16, 2) || !aligned(a2_f16, 2) || !aligned(blocks, 16))
        return fail(TQFX4_EALIGN, "%s: t1, t2 and blocks must be 16-byte aligned", fn);
    cudaError_t e = tq::launch_pack_free(t1, t2, a1_f16, a2_f16, n, k, blocks, static_cast<int *>(ws),
                                         static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_gemv_free(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                             const int32_t *bsum, float *y, int32_t *S1, int32_t *S2, void *ws, size_t ws_bytes,
                             void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_gemv_free";
    tqfx4_status s = check_nk(n, k, fn);
    if (s) return s;
    if (k == 0 || k > TQFX4_MAX_K) return fail(TQFX4_ESHAPE, "%s: k=%lld must be in 256..%d", fn, (long long)k,
                                               TQFX4_MAX_K);
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, fn))) return s;
    if (n == 0) return ok();
    if (!blocks || !q || !da || !bsum || !y) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    if ((S1 == nullptr) != (S2 == nullptr)) return fail(TQFX4_EINVAL, "%s: S1 and S2 both or neither", fn);
    if (!aligned(blocks, 16) || !aligned(q, 16) || !aligned(da, 4) || !aligned(bsum, 4) || !aligned(y, 4) ||
        !aligned(S1, 4) || !aligned(S2, 4))
        return fail(TQFX4_EALIGN, "%s: blocks and q must be 16-byte aligned", fn);
    if (tq::gemv_free_smem(k) > tq::max_smem_optin())
        return fail(TQFX4_ESHAPE, "%s: k too large for shared memory", fn);
    cudaError_t e = tq::launch_gemv_free(blocks, n, k, q, da, bsum, y, S1, S2, static_cast<int *>(ws),
                                         static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

int64_t tqfx4_mxfp4_bytes(int64_t n, int64_t k) { return tq::mxfp4_bytes(n, k); }

tqfx4_status tqfx4_gemv_mxfp4(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                              int32_t *block_sums, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_gemv_mxfp4";
    if (n < 0 || k <= 0 || k % 512 || k > TQFX4_MAX_K)
        return fail(TQFX4_ESHAPE, "%s: k=%lld must be a positive multiple of 512 <= %d", fn, (long long)k,
                    TQFX4_MAX_K);
    tqfx4_status s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, fn);
    if (s) return s;
    if (n == 0) return ok();
    if (!blocks || !q || !da || !y) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    if (!aligned(blocks, 16) || !aligned(q, 16) || !aligned(da, 4) || !aligned(y, 4) || !aligned(block_sums, 4))
        return fail(TQFX4_EALIGN, "%s: blocks and q must be 16-byte aligned", fn);
    cudaError_t e = tq::launch_mxfp4_gemv(blocks, n, k, q, da, y, block_sums, static_cast<int *>(ws),
                                          static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

// ---------------------------------------------------------------- MoE

namespace {

tqfx4_status check_moe_shapes(const tqfx4_experts *ex, const tqfx4_router *rt, const char *fn) {
    if (!ex || !rt) return fail(TQFX4_EINVAL, "%s: NULL experts or router", fn);
    if (ex->n_experts < 1 || ex->n_experts > TQFX4_MAX_EXPERTS)
        return fail(TQFX4_ESHAPE, "%s: n_experts=%lld outside 1..%d", fn, (long long)ex->n_experts,
                    TQFX4_MAX_EXPERTS);
    if (ex->hidden <= 0 || ex->inter <= 0 || ex->hidden % 256 || ex->inter % 256 || ex->hidden > TQFX4_MAX_K ||
        ex->inter > TQFX4_MAX_K)
        return fail(TQFX4_ESHAPE, "%s: hidden=%lld, inter=%lld must be positive multiples of 256 <= %d", fn,
                    (long long)ex->hidden, (long long)ex->inter, TQFX4_MAX_K);
    if (rt->top_k < 1 || rt->top_k > TQFX4_MAX_TOP_K || rt->top_k > ex->n_experts)
        return fail(TQFX4_ESHAPE, "%s: top_k=%d outside 1..min(n_experts, %d)", fn, rt->top_k, TQFX4_MAX_TOP_K);
    return TQFX4_OK;
}

tqfx4_status check_moe_ptrs(const tqfx4_experts *ex, const tqfx4_router *rt, const char *fn) {
    if (!ex->gate || !ex->up || !ex->down || !rt->weight) return fail(TQFX4_EINVAL, "%s: NULL weights", fn);
    if (!aligned(ex->gate, 16) || !aligned(ex->up, 16) || !aligned(ex->down, 16) || !aligned(rt->weight, 16) ||
        !aligned(rt->bias, 4))
        return fail(TQFX4_EALIGN, "%s: expert and router weights must be 16-byte aligned", fn);
    return TQFX4_OK;
}

}  // namespace

size_t tqfx4_moe_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t tokens, int path) {
    (void)path;
    if (check_moe_shapes(ex, rt, "tqfx4_moe_workspace_bytes") || tokens < 0) return 0;
    const int64_t T = tokens < 1 ? 1 : tokens;
    const size_t dec = tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, 1, false, true).total;
    const size_t grp = tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, T, true, true).total;
    return tokens <= 1 ? (dec > grp ? dec : grp) : grp;
}

int tqfx4_moe_stage_count(int grouped, int path) {
    (void)path;
    if (grouped == 2) return 4;
    return grouped ? tq::grouped_stage_count() : 3;
}

const char *tqfx4_moe_stage_name(int grouped, int path, int stage) {
    (void)path;
    static const char *dec[] = {"router", "gate_up", "down"};
    static const char *mx[] = {"router", "gate_up", "down", "combine"};
    if (grouped == 2) return (stage >= 0 && stage < 4) ? mx[stage] : "";
    if (grouped) return tq::grouped_stage_name(stage);
    if (stage >= 0 && stage < 3) return dec[stage];
    return "";
}

static tqfx4_status moe_ffn_impl(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x, float *out,
                                 int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes, void *stream,
                                 void *const *events) {
    const char *fn = "tqfx4_moe_ffn";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if ((s = check_moe_ptrs(ex, rt, fn))) return s;
    if (!x || !out || !sel_idx || !sel_w) return fail(TQFX4_EINVAL, "%s: NULL x, out or selection output", fn);
    if (!aligned(x, 16) || !aligned(out, 4) || !aligned(sel_idx, 4) || !aligned(sel_w, 4))
        return fail(TQFX4_EALIGN, "%s: x must be 16-byte aligned", fn);
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(ex, rt, nullptr, a, L))
        return fail(TQFX4_ESHAPE, "%s: too many row ranges for the counter area", fn);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    if (tq::gate_up_smem(a) > tq::max_smem_optin() || tq::down_smem(a) > tq::max_smem_optin())
        return fail(TQFX4_ESHAPE, "%s: top_k x inter too large for the decode kernels' shared memory", fn);
    tq::moe_decode_args(ex, rt, ws, a, L);
    // (debug build) the stacked experts: E x inter rows of gate and of up, E x hidden rows of down
    cudaError_t e = debug_validate(ex->gate, ex->n_experts * ex->inter, ex->hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(ex->up, ex->n_experts * ex->inter, ex->hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(ex->down, ex->n_experts * ex->hidden, ex->inter, ws, stream);
    if (e == cudaSuccess)
        e = tq::launch_moe_decode(a, x, out, sel_idx, sel_w, static_cast<cudaStream_t>(stream), events);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_moe_ffn(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x, float *out,
                           int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    return moe_ffn_impl(ex, rt, x, out, sel_idx, sel_w, ws, ws_bytes, stream, nullptr);
}

tqfx4_status tqfx4_moe_ffn_traced(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x, float *out,
                                  int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes, void *stream,
                                  void *const *events) {
    TQ_RANGE();
    return moe_ffn_impl(ex, rt, x, out, sel_idx, sel_w, ws, ws_bytes, stream, events);
}

// Staging of tqfx4_moe_ffn_host after the decode layout: x, out, the selection.
struct HostStaging {
    size_t x, out, sel, selw, total;
};
static HostStaging host_staging(const tqfx4_experts *ex, const tqfx4_router *rt) {
    HostStaging h;
    size_t off = tq::align256(tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, 1, false, true).total);
    h.x = off;
    off = tq::align256(off + 4 * static_cast<size_t>(ex->hidden));
    h.out = off;
    off = tq::align256(off + 4 * static_cast<size_t>(ex->hidden));
    h.sel = off;
    off = tq::align256(off + 4 * static_cast<size_t>(rt->top_k));
    h.selw = off;
    h.total = tq::align256(off + 4 * static_cast<size_t>(rt->top_k));
    return h;
}

size_t tqfx4_moe_ffn_host_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt) {
    if (check_moe_shapes(ex, rt, "tqfx4_moe_ffn_host_workspace_bytes")) return 0;
    return host_staging(ex, rt).total;
}

tqfx4_status tqfx4_moe_ffn_host(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x_host,
                                float *out_host, int32_t *sel_idx_host, float *sel_w_host, void *ws, size_t ws_bytes,
                                void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_moe_ffn_host";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if ((s = check_moe_ptrs(ex, rt, fn))) return s;
    if (!x_host || !out_host) return fail(TQFX4_EINVAL, "%s: NULL x or out", fn);
    const HostStaging h = host_staging(ex, rt);
    if ((s = check_ws(ws, ws_bytes, h.total, fn))) return s;
    uint8_t *base = static_cast<uint8_t *>(ws);
    float *xd = reinterpret_cast<float *>(base + h.x), *od = reinterpret_cast<float *>(base + h.out);
    int32_t *sd = reinterpret_cast<int32_t *>(base + h.sel);
    float *wd = reinterpret_cast<float *>(base + h.selw);
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t xb = 4 * static_cast<size_t>(ex->hidden), kb = 4 * static_cast<size_t>(rt->top_k);
    // Page-locked host buffers are used in place: x is read into the staging
    // by a small kernel and the layer writes out and the selection straight
    // into host memory, with no copy engine round trip. Pageable ones go
    // through the staging with cudaMemcpyAsync.
    const float *xm = static_cast<const float *>(mapped(x_host, 16));
    float *om = static_cast<float *>(mapped(out_host, 4));
    int32_t *sm = static_cast<int32_t *>(mapped(sel_idx_host, 4));
    float *wm = static_cast<float *>(mapped(sel_w_host, 4));
    cudaError_t e = xm ? tq::launch_copy_f32(xd, xm, ex->hidden, st)
                       : cudaMemcpyAsync(xd, x_host, xb, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    if ((s = moe_ffn_impl(ex, rt, xd, om ? om : od, sm ? sm : sd, wm ? wm : wd, ws, ws_bytes, stream, nullptr)))
        return s;
    if (!om) e = cudaMemcpyAsync(out_host, od, xb, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && sel_idx_host && !sm) e = cudaMemcpyAsync(sel_idx_host, sd, kb, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && sel_w_host && !wm) e = cudaMemcpyAsync(sel_w_host, wd, kb, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

size_t tqfx4_expert_ffn_workspace_bytes(int64_t hidden, int64_t inter) {
    if (hidden <= 0 || inter <= 0 || hidden % 256 || inter % 256 || hidden > TQFX4_MAX_K || inter > TQFX4_MAX_K)
        return 0;
    return tq::moe_layout(1, hidden, inter, 1, 1, false, true).total;
}

int tqfx4_expert_ffn_launches(int64_t hidden, int64_t inter) {
    if (tqfx4_expert_ffn_workspace_bytes(hidden, inter) == 0) return 0;
    const tqfx4_experts ex{nullptr, nullptr, nullptr, 1, hidden, inter};
    tqfx4_router rt{};
    rt.top_k = 1;
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(&ex, &rt, nullptr, a, L)) return 0;
    return tq::expert_ffn_one_launch(a) ? 1 : 2;
}

static tqfx4_status expert_ffn_impl(const void *gate, const void *up, const void *down, int64_t hidden,
                                    int64_t inter, const float *x, float *out, void *ws, size_t ws_bytes,
                                    void *stream, void *const *events) {
    const char *fn = "tqfx4_expert_ffn";
    const tqfx4_experts ex{gate, up, down, 1, hidden, inter};
    tqfx4_router rt{};
    rt.top_k = 1;
    tqfx4_status s = check_moe_shapes(&ex, &rt, fn);
    if (s) return s;
    if (!gate || !up || !down || !x || !out) return fail(TQFX4_EINVAL, "%s: NULL matrix, input or output", fn);
    if (!aligned(gate, 16) || !aligned(up, 16) || !aligned(down, 16) || !aligned(x, 16) || !aligned(out, 4))
        return fail(TQFX4_EALIGN, "%s: matrices and x must be 16-byte aligned", fn);
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(&ex, &rt, nullptr, a, L))
        return fail(TQFX4_ESHAPE, "%s: too many row ranges for the counter area", fn);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    if (tq::gate_up_smem(a) > tq::max_smem_optin() || tq::down_smem(a) > tq::max_smem_optin())
        return fail(TQFX4_ESHAPE, "%s: inter too large for the decode kernels' shared memory", fn);
    tq::moe_decode_args(&ex, &rt, ws, a, L);
    cudaError_t e = debug_validate(gate, inter, hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(up, inter, hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(down, hidden, inter, ws, stream);
    if (e == cudaSuccess) e = tq::launch_expert_ffn(a, x, out, static_cast<cudaStream_t>(stream), events);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_expert_ffn(const void *gate, const void *up, const void *down, int64_t hidden, int64_t inter,
                              const float *x, float *out, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    return expert_ffn_impl(gate, up, down, hidden, inter, x, out, ws, ws_bytes, stream, nullptr);
}

tqfx4_status tqfx4_expert_ffn_traced(const void *gate, const void *up, const void *down, int64_t hidden,
                                     int64_t inter, const float *x, float *out, void *ws, size_t ws_bytes,
                                     void *stream, void *const *events) {
    TQ_RANGE();
    return expert_ffn_impl(gate, up, down, hidden, inter, x, out, ws, ws_bytes, stream, events);
}

size_t tqfx4_expert_ffn_host_workspace_bytes(int64_t hidden, int64_t inter) {
    const size_t base = tqfx4_expert_ffn_workspace_bytes(hidden, inter);
    if (base == 0) return 0;
    return tq::align256(tq::align256(tq::align256(base) + 4 * static_cast<size_t>(hidden)) +
                        4 * static_cast<size_t>(hidden));
}

tqfx4_status tqfx4_expert_ffn_host(const void *gate, const void *up, const void *down, int64_t hidden,
                                   int64_t inter, const float *x_host, float *out_host, void *ws, size_t ws_bytes,
                                   void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_expert_ffn_host";
    const size_t base = tqfx4_expert_ffn_workspace_bytes(hidden, inter);
    if (base == 0) return fail(TQFX4_ESHAPE, "%s: hidden and inter must be positive multiples of 256", fn);
    const size_t need = tqfx4_expert_ffn_host_workspace_bytes(hidden, inter);
    if (!gate || !up || !down || !x_host || !out_host)
        return fail(TQFX4_EINVAL, "%s: NULL matrix, input or output", fn);
    tqfx4_status s = check_ws(ws, ws_bytes, need, fn);
    if (s) return s;
    uint8_t *b = static_cast<uint8_t *>(ws);
    const size_t xo = tq::align256(base), oo = tq::align256(xo + 4 * static_cast<size_t>(hidden));
    float *xd = reinterpret_cast<float *>(b + xo), *od = reinterpret_cast<float *>(b + oo);
    // page-locked buffers in place: a small kernel reads x into the staging
    // (once, not by every CTA of the FFN over the host link) and the kernel
    // that forms the down rows writes out straight into host memory
    const float *xm = static_cast<const float *>(mapped(x_host, 16));
    float *om = static_cast<float *>(mapped(out_host, 4));
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t hb = 4 * static_cast<size_t>(hidden);
    cudaError_t e = xm ? tq::launch_copy_f32(xd, xm, hidden, st) : cudaMemcpyAsync(xd, x_host, hb, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    if ((s = expert_ffn_impl(gate, up, down, hidden, inter, xd, om ? om : od, ws, ws_bytes, stream, nullptr)))
        return s;
    if (!om) e = cudaMemcpyAsync(out_host, od, hb, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_moe_route(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x, int32_t *sel_idx,
                             float *sel_w, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_moe_route";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (!rt->weight) return fail(TQFX4_EINVAL, "%s: NULL router weights", fn);
    if (!aligned(rt->weight, 16) || !aligned(rt->bias, 4))
        return fail(TQFX4_EALIGN, "%s: router weights must be 16-byte aligned", fn);
    if (!x || !sel_idx || !sel_w) return fail(TQFX4_EINVAL, "%s: NULL x or selection output", fn);
    if (!aligned(x, 16) || !aligned(sel_idx, 4) || !aligned(sel_w, 4))
        return fail(TQFX4_EALIGN, "%s: x must be 16-byte aligned", fn);
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(ex, rt, nullptr, a, L))
        return fail(TQFX4_ESHAPE, "%s: too many row ranges for the counter area", fn);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    tq::moe_decode_args(ex, rt, ws, a, L);
    cudaError_t e = tq::launch_moe_route(a, x, sel_idx, sel_w, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

static tqfx4_status moe_ffn_mxfp4_impl(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x,
                                       float *out, int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes,
                                       void *stream, void *const *events) {
    const char *fn = "tqfx4_moe_ffn_mxfp4";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (ex->hidden % 512 || ex->inter % 512)
        return fail(TQFX4_ESHAPE, "%s: hidden and inter must be multiples of 512", fn);
    if (!ex->gate || !ex->up || !ex->down || !rt->weight) return fail(TQFX4_EINVAL, "%s: NULL expert or router weights", fn);
    if (!x || !out || !sel_idx || !sel_w) return fail(TQFX4_EINVAL, "%s: NULL input or output", fn);
    if (!aligned(ex->gate, 16) || !aligned(ex->up, 16) || !aligned(ex->down, 16) || !aligned(rt->weight, 16) ||
        !aligned(rt->bias, 4) || !aligned(x, 16) || !aligned(out, 4) || !aligned(sel_idx, 4) || !aligned(sel_w, 4))
        return fail(TQFX4_EALIGN, "%s: expert blocks, router weights and x must be 16-byte aligned", fn);
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(ex, rt, nullptr, a, L))
        return fail(TQFX4_ESHAPE, "%s: too many row ranges for the counter area", fn);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    if (tq::mxfp4_gemv_smem(ex->hidden, 1) > tq::max_smem_optin() ||
        tq::mxfp4_gemv_smem(ex->inter, rt->top_k) > tq::max_smem_optin())
        return fail(TQFX4_ESHAPE, "%s: top_k x inter too large for the kernels' shared memory", fn);
    tq::moe_decode_args(ex, rt, ws, a, L);
    a.mb_gu = tq::mxfp4_bytes(ex->inter, ex->hidden);
    a.mb_d = tq::mxfp4_bytes(ex->hidden, ex->inter);
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaEvent_t const *ev = reinterpret_cast<cudaEvent_t const *>(events);
    cudaError_t e = ev ? tq::record_stage_event(ev[0], st) : cudaSuccess;
    if (e == cudaSuccess) e = tq::launch_moe_route(a, x, sel_idx, sel_w, st);
    if (e == cudaSuccess) e = tq::launch_moe_mxfp4_experts(a, out, st, ev ? ev + 1 : nullptr);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_moe_ffn_mxfp4(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x, float *out,
                                 int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    return moe_ffn_mxfp4_impl(ex, rt, x, out, sel_idx, sel_w, ws, ws_bytes, stream, nullptr);
}

tqfx4_status tqfx4_moe_ffn_mxfp4_traced(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x,
                                        float *out, int32_t *sel_idx, float *sel_w, void *ws, size_t ws_bytes,
                                        void *stream, void *const *events) {
    TQ_RANGE();
    return moe_ffn_mxfp4_impl(ex, rt, x, out, sel_idx, sel_w, ws, ws_bytes, stream, events);
}

tqfx4_status tqfx4_moe_experts(const tqfx4_experts *ex, const tqfx4_router *rt, const void *const *ptrs, float *out,
                               void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_moe_experts";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (!ptrs || !out) return fail(TQFX4_EINVAL, "%s: NULL pointer table or output", fn);
    if (!aligned(ptrs, 8) || !aligned(out, 4)) return fail(TQFX4_EALIGN, "%s: misaligned pointer table", fn);
    tq::MoeArgs a;
    tq::MoeLayout L;
    if (!tq::moe_decode_args(ex, rt, nullptr, a, L))
        return fail(TQFX4_ESHAPE, "%s: too many row ranges for the counter area", fn);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    if (tq::gate_up_smem(a) > tq::max_smem_optin() || tq::down_smem(a) > tq::max_smem_optin())
        return fail(TQFX4_ESHAPE, "%s: top_k x inter too large for the decode kernels' shared memory", fn);
    tq::moe_decode_args(ex, rt, ws, a, L);
    cudaError_t e = tq::launch_moe_experts(a, ptrs, out, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

static tqfx4_status moe_grouped_impl(const tqfx4_experts *ex, const tqfx4_router *rt, const float *X, int64_t T,
                                     float *OUT, int32_t *sel_idx, float *sel_w, int path, void *ws,
                                     size_t ws_bytes, void *stream, void *const *events) {
    const char *fn = "tqfx4_moe_grouped";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (T < 0) return fail(TQFX4_EINVAL, "%s: negative token count", fn);
    if (path < TQFX4_PATH_AUTO || path > TQFX4_PATH_PREFILL) return fail(TQFX4_EINVAL, "%s: unknown path %d", fn, path);
    if (ex->hidden % 512 || ex->inter % 512)
        return fail(TQFX4_ESHAPE, "%s: hidden and inter must be multiples of 512 for the grouped path", fn);
    if (T * rt->top_k > (int64_t(1) << 30)) return fail(TQFX4_ESHAPE, "%s: too many tokens", fn);
    if ((s = check_moe_ptrs(ex, rt, fn))) return s;
    if (T == 0) return ok();
    if (!X || !OUT || !sel_idx || !sel_w) return fail(TQFX4_EINVAL, "%s: NULL X, OUT or selection output", fn);
    if (!aligned(X, 16) || !aligned(OUT, 16) || !aligned(sel_idx, 4) || !aligned(sel_w, 4))
        return fail(TQFX4_EALIGN, "%s: X and OUT must be 16-byte aligned", fn);
    tq::GroupedArgs a;
    tq::MoeLayout L;
    tq::grouped_args(ex, rt, T, nullptr, a, L);
    if ((s = check_ws(ws, ws_bytes, L.total, fn))) return s;
    tq::grouped_args(ex, rt, T, ws, a, L);
    // The tensor-core contraction pays off once the chunks are mostly full.
    a.tc = path == TQFX4_PATH_PREFILL || (path == TQFX4_PATH_AUTO && T * rt->top_k >= tq::kTcMinPairs);
    cudaError_t e = debug_validate(ex->gate, ex->n_experts * ex->inter, ex->hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(ex->up, ex->n_experts * ex->inter, ex->hidden, ws, stream);
    if (e == cudaSuccess) e = debug_validate(ex->down, ex->n_experts * ex->hidden, ex->inter, ws, stream);
    if (e == cudaSuccess)
        e = tq::launch_moe_grouped(a, X, OUT, sel_idx, sel_w, static_cast<cudaStream_t>(stream), events);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_moe_grouped(const tqfx4_experts *ex, const tqfx4_router *rt, const float *X, int64_t T,
                               float *OUT, int32_t *sel_idx, float *sel_w, int path, void *ws, size_t ws_bytes,
                               void *stream) {
    TQ_RANGE();
    return moe_grouped_impl(ex, rt, X, T, OUT, sel_idx, sel_w, path, ws, ws_bytes, stream, nullptr);
}

// Staging of tqfx4_moe_grouped_host after the grouped layout: X, OUT, the selection.
struct GroupedStaging {
    size_t x, out, sel, selw, total;
};
static GroupedStaging grouped_staging(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t T) {
    GroupedStaging g;
    const size_t th = 4 * static_cast<size_t>(T) * ex->hidden, tk = 4 * static_cast<size_t>(T) * rt->top_k;
    size_t off = tq::align256(tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, T, true, true).total);
    g.x = off;
    off = tq::align256(off + th);
    g.out = off;
    off = tq::align256(off + th);
    g.sel = off;
    off = tq::align256(off + tk);
    g.selw = off;
    g.total = tq::align256(off + tk);
    return g;
}

size_t tqfx4_moe_grouped_host_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t tokens,
                                              int path) {
    (void)path;
    if (check_moe_shapes(ex, rt, "tqfx4_moe_grouped_host_workspace_bytes") || tokens < 1) return 0;
    return grouped_staging(ex, rt, tokens).total;
}

tqfx4_status tqfx4_moe_grouped_host(const tqfx4_experts *ex, const tqfx4_router *rt, const float *X_host,
                                    int64_t T, float *OUT_host, int32_t *sel_idx_host, float *sel_w_host, int path,
                                    void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    const char *fn = "tqfx4_moe_grouped_host";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (T < 0) return fail(TQFX4_EINVAL, "%s: negative token count", fn);
    if (T == 0) return ok();
    if ((s = check_moe_ptrs(ex, rt, fn))) return s;
    if (!X_host || !OUT_host) return fail(TQFX4_EINVAL, "%s: NULL X or OUT", fn);
    const GroupedStaging g = grouped_staging(ex, rt, T);
    if ((s = check_ws(ws, ws_bytes, g.total, fn))) return s;
    uint8_t *b = static_cast<uint8_t *>(ws);
    float *xd = reinterpret_cast<float *>(b + g.x), *od = reinterpret_cast<float *>(b + g.out);
    int32_t *sd = reinterpret_cast<int32_t *>(b + g.sel);
    float *wd = reinterpret_cast<float *>(b + g.selw);
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t th = 4 * static_cast<size_t>(T) * ex->hidden, tk = 4 * static_cast<size_t>(T) * rt->top_k;
    // page-locked buffers in place: a copy kernel reads X into the staging
    // (every router and gather CTA reads it), and the combine and the top-k
    // write OUT and the selection straight into host memory
    const float *xm = static_cast<const float *>(mapped(X_host, 16));
    float *om = static_cast<float *>(mapped(OUT_host, 16));
    int32_t *sm = static_cast<int32_t *>(mapped(sel_idx_host, 4));
    float *wm = static_cast<float *>(mapped(sel_w_host, 4));
    cudaError_t e = xm ? tq::launch_copy_f32(xd, xm, T * ex->hidden, st)
                       : cudaMemcpyAsync(xd, X_host, th, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    if ((s = moe_grouped_impl(ex, rt, xd, T, om ? om : od, sm ? sm : sd, wm ? wm : wd, path, ws, ws_bytes, stream,
                              nullptr)))
        return s;
    if (!om) e = cudaMemcpyAsync(OUT_host, od, th, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && sel_idx_host && !sm) e = cudaMemcpyAsync(sel_idx_host, sd, tk, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && sel_w_host && !wm) e = cudaMemcpyAsync(sel_w_host, wd, tk, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

tqfx4_status tqfx4_moe_grouped_traced(const tqfx4_experts *ex, const tqfx4_router *rt, const float *X, int64_t T,
                                      float *OUT, int32_t *sel_idx, float *sel_w, int path, void *ws,
                                      size_t ws_bytes, void *stream, void *const *events) {
    TQ_RANGE();
    return moe_grouped_impl(ex, rt, X, T, OUT, sel_idx, sel_w, path, ws, ws_bytes, stream, events);
}

tqfx4_status tqfx4_moe_workspace_views(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t tokens,
                                       int grouped, int path, tqfx4_moe_views *v) {
    (void)path;
    const char *fn = "tqfx4_moe_workspace_views";
    tqfx4_status s = check_moe_shapes(ex, rt, fn);
    if (s) return s;
    if (!v) return fail(TQFX4_EINVAL, "%s: NULL views", fn);
    const int64_t T = grouped ? tokens : 1;
    const tq::MoeLayout L = tq::moe_layout(ex->n_experts, ex->hidden, ex->inter, rt->top_k, T, grouped != 0, true);
    v->logits = L.logits;
    v->logits_lo = L.logits_lo;
    v->qx = L.qx;
    v->dx = L.dx;
    v->bx = L.bx;
    v->g = L.g;
    v->u = L.u;
    v->h = L.h;
    v->qh = L.qh;
    v->dh = L.dh;
    v->bh = L.bh;
    v->o = L.o;
    v->counts = L.counts;
    v->offsets = L.offsets;
    v->pair_token = L.pair_token;
    v->pair_slot = L.pair_slot;
    v->pair_of = L.pair_of;
    return ok();
}

tqfx4_status tqfx4_check(void *ws, void *stream) {
    TQ_RANGE();
    if (!ws) return fail(TQFX4_EINVAL, "tqfx4_check: workspace is NULL");
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: stream");
    int st[4] = {0, 0, 0, 0};
    e = cudaMemcpy(st, ws, sizeof(st), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: status read");
    if (st[0] == 0) return ok();
    e = cudaMemset(ws, 0, sizeof(st));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: status clear");
    static const char *kernels[] = {"?",      "pack",   "quantize", "gemv",     "router", "gate_up", "down",
                                    "topk",   "group",  "g_gateup", "g_down",   "combine", "prefill", "selftest"};
    const int nk = static_cast<int>(sizeof(kernels) / sizeof(kernels[0]));
    const char *kn = (st[1] >= 0 && st[1] < nk) ? kernels[st[1]] : "?";
    if (st[0] == TQFX4_EDATA || st[0] == TQFX4_ETIMEOUT)
        return fail(static_cast<tqfx4_status>(st[0]), "device error %d in kernel %s (unit %d)", st[0], kn, st[2]);
    return fail(TQFX4_ECUDA, "unknown device status %d in kernel %s", st[0], kn);
}

tqfx4_status tqfx4_selftest_wait_timeout(void *ws, size_t ws_bytes, void *stream) {
    TQ_RANGE();
    tqfx4_status s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, "tqfx4_selftest_wait_timeout");
    if (s) return s;
    cudaError_t e = tq::launch_selftest_timeout(static_cast<int *>(ws), static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_selftest_wait_timeout");
    return ok();
}

const char *tqfx4_last_error(void) { return g_err; }

const char *tqfx4_status_string(tqfx4_status s) {
    switch (s) {
        case TQFX4_OK: return "TQFX4_OK";
        case TQFX4_EINVAL: return "TQFX4_EINVAL";
        case TQFX4_ESHAPE: return "TQFX4_ESHAPE";
        case TQFX4_EALIGN: return "TQFX4_EALIGN";
        case TQFX4_EWORKSPACE: return "TQFX4_EWORKSPACE";
        case TQFX4_ECUDA: return "TQFX4_ECUDA";
        case TQFX4_ETIMEOUT: return "TQFX4_ETIMEOUT";
        case TQFX4_EDATA: return "TQFX4_EDATA";
    }
    return "TQFX4_UNKNOWN";
}

}  // extern "C"
