// C ABI of libtqfx4 (declared in include/tqfx4.h): argument checks on the
// host, then asynchronous launches on the caller's stream.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "tq_launch.h"
#include "tqfx4.h"

namespace {

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

extern "C" {

int64_t tqfx4_matrix_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || n % 4 || k % 256) return -1;
    return (n / 4) * (k / 256) * 520;
}

size_t tqfx4_basic_workspace_bytes(void) { return TQFX4_STATUS_BYTES; }

tqfx4_status tqfx4_pack(int src, const void *a, const int8_t *t2, const uint16_t *scales_f16, int64_t n,
                        int64_t k, void *blocks, void *ws, size_t ws_bytes, void *stream) {
    tqfx4_status s = check_nk(n, k, "tqfx4_pack");
    if (s) return s;
    if ((s = check_ws(ws, ws_bytes, TQFX4_STATUS_BYTES, "tqfx4_pack"))) return s;
    if (n == 0 || k == 0) return ok();
    if (!a || !blocks) return fail(TQFX4_EINVAL, "tqfx4_pack: NULL input or output");
    if (!aligned(blocks, 16)) return fail(TQFX4_EALIGN, "tqfx4_pack: blocks must be 16-byte aligned");
    if (src == TQFX4_SRC_F32_RTN) {
        if (t2 || scales_f16) return fail(TQFX4_EINVAL, "tqfx4_pack: t2/scales must be NULL for F32_RTN");
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
    cudaError_t e = tq::launch_gemv(blocks, n, k, q, da, bsum, y, block_sums, static_cast<int *>(ws),
                                    static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_gemv");
    return ok();
}

tqfx4_status tqfx4_check(void *ws, void *stream) {
    if (!ws) return fail(TQFX4_EINVAL, "tqfx4_check: workspace is NULL");
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: stream");
    int st[4] = {0, 0, 0, 0};
    e = cudaMemcpy(st, ws, sizeof(st), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: status read");
    if (st[0] == 0) return ok();
    e = cudaMemset(ws, 0, sizeof(st));
    if (e != cudaSuccess) return cuda_fail(e, "tqfx4_check: status clear");
    static const char *kernels[] = {"?",      "pack",   "quantize", "gemv",   "router",  "gate_up",
                                    "down",   "topk",   "group",    "g_gateup", "g_down", "combine",
                                    "prefill"};
    const char *kn = (st[1] >= 0 && st[1] < 13) ? kernels[st[1]] : "?";
    if (st[0] == TQFX4_EDATA || st[0] == TQFX4_ETIMEOUT)
        return fail(static_cast<tqfx4_status>(st[0]), "device error %d in kernel %s (unit %d)", st[0], kn, st[2]);
    return fail(TQFX4_ECUDA, "unknown device status %d in kernel %s", st[0], kn);
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
