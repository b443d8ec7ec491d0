// tqfx4_gemv: the integer dot pass of Tied Trit-Planes Sec. 2.2 on GB300.
//
// Data path: a matrix is one contiguous stream of 520-byte blocks. Each warp
// owns a private ring of shared-memory slots and streams "units" (whole row
// groups, about 32 blocks = 16.6 KB) into them with cp.async.bulk on an
// mbarrier, several units ahead of the one it computes. In a unit, lane i
// owns block i: it computes the four exact int32 block sums of the block's
// rows with dp4a (no cross-lane reduction), writes them to shared memory,
// and then one lane per row applies the fixed float schedule
// acc = acc + float(S) * (d * da) over the blocks in ascending order.
#include "tq_common.cuh"
#include "tq_launch.h"

namespace tq {

struct GemvGeom {
    int64_t n_rg;      // row groups in the matrix
    int nb;            // blocks per row group (K / 256)
    int rpu;           // row groups per unit
    int64_t units;     // ceil(n_rg / rpu)
    int slot_bytes;    // per slot, 16-byte multiple, including the alignment pad
    int stages;        // slots per warp
    int warps;         // warps per CTA
    int sbuf_stride;   // ints per row in the block-sum buffer (nb + 1)
};

__host__ __device__ inline int gemv_smem_act_bytes(int nb) {
    return ((nb * QS_STRIDE + 8 * nb + 127) / 128) * 128;
}

__host__ __device__ inline int gemv_sbuf_bytes(const GemvGeom &g) {
    return ((g.rpu * 4 * g.sbuf_stride * 4 + 15) / 16) * 16;
}

// Per-warp shared memory: slots, block-sum buffer, barriers; rounded up so
// that every warp's slots start 128-byte aligned.
__host__ __device__ inline int gemv_smem_warp_bytes(const GemvGeom &g) {
    return ((g.stages * g.slot_bytes + gemv_sbuf_bytes(g) + g.stages * 8 + 127) / 128) * 128;
}

__global__ void __launch_bounds__(256, 1) gemv_kernel(const uint8_t *__restrict__ blocks, GemvGeom g,
                                                      const int8_t *__restrict__ q,
                                                      const float *__restrict__ da,
                                                      const int32_t *__restrict__ bsum, float *__restrict__ y,
                                                      int32_t *__restrict__ s_out, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nb = g.nb;

    uint8_t *qs = smem;
    float *das = reinterpret_cast<float *>(smem + nb * QS_STRIDE);
    int *bss = reinterpret_cast<int *>(das + nb);
    uint8_t *wbase = smem + gemv_smem_act_bytes(nb) + warp * gemv_smem_warp_bytes(g);
    uint8_t *slots = wbase;
    int *sbuf = reinterpret_cast<int *>(wbase + g.stages * g.slot_bytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + g.stages * g.slot_bytes + gemv_sbuf_bytes(g));

    if (lane == 0)
        for (int s = 0; s < g.stages; ++s) mbar_init(&bars[s], 1);
    fence_barrier_init();
    load_act_smem(q, da, bsum, nb, qs, das, bss);
    __syncthreads();

    const int64_t total_warps = static_cast<int64_t>(gridDim.x) * g.warps;
    const int64_t gw = static_cast<int64_t>(blockIdx.x) * g.warps + warp;
    const int64_t unit_bytes = static_cast<int64_t>(g.rpu) * nb * BLOCK_BYTES;
    const int64_t matrix_bytes = g.n_rg * nb * BLOCK_BYTES;

    auto issue = [&](int64_t u, int slot) -> void {
        const int64_t off = u * unit_bytes;
        const int64_t len = imin64(unit_bytes, matrix_bytes - off);
        stage_range(lane, slots + slot * g.slot_bytes, blocks + off, static_cast<uint32_t>(len), &bars[slot]);
    };

    // prologue: fill the ring
    int64_t next = gw;
    for (int s = 0; s < g.stages; ++s) {
        if (next < g.units) issue(next, s);
        next += total_warps;
    }

    int it = 0;
    for (int64_t u = gw; u < g.units; u += total_warps, ++it) {
        const int slot = it % g.stages;
        const uint32_t parity = static_cast<uint32_t>((it / g.stages) & 1);
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[slot], parity))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(u));
            return;
        }
        __syncwarp();  // orders the head/tail pieces other lanes stored
        const uint8_t *data = slots + slot * g.slot_bytes +
                              (reinterpret_cast<uintptr_t>(blocks + u * unit_bytes) & 15u);
        const int64_t rg0 = u * g.rpu;
        const int rgs = static_cast<int>(imin64(g.rpu, g.n_rg - rg0));
        const int nblk = rgs * nb;
        for (int i = lane; i < nblk; i += 32) {
            const int rgl = i / nb;
            const int b = i - rgl * nb;
            const uint8_t *blk = data + i * BLOCK_BYTES;
            int S[4];
            block_dot(blk + CODE_OFS, qs + b * QS_STRIDE, bss[b], S);
#pragma unroll
            for (int r = 0; r < 4; ++r) sbuf[(rgl * 4 + r) * g.sbuf_stride + b] = S[r];
            if (s_out) {
#pragma unroll
                for (int r = 0; r < 4; ++r) s_out[((rg0 + rgl) * 4 + r) * nb + b] = S[r];
            }
        }
        __syncwarp();
        for (int t = lane; t < rgs * 4; t += 32) {
            const int rgl = t >> 2, r = t & 3;
            float acc = 0.0f;
            for (int b = 0; b < nb; ++b) {
                const float sc = __fmul_rn(block_scale(data + (rgl * nb + b) * BLOCK_BYTES, r), das[b]);
                acc = __fadd_rn(acc, __fmul_rn(static_cast<float>(sbuf[t * g.sbuf_stride + b]), sc));
            }
            y[(rg0 + rgl) * 4 + r] = acc;
        }
        __syncwarp();
        // refill this slot with the unit `stages` iterations ahead
        const int64_t nu = u + static_cast<int64_t>(g.stages) * total_warps;
        if (nu < g.units) {
            fence_proxy_async_smem();
            issue(nu, slot);
        }
    }
}

__global__ void zero_kernel(float *y, int64_t n) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i < n) y[i] = 0.0f;
}

static int g_num_sms = 0;

int num_sms() {
    if (g_num_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_num_sms <= 0) g_num_sms = 148;
    }
    return g_num_sms;
}

int max_smem_optin() {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    return v > 0 ? v : 232448;
}

static GemvGeom gemv_geom(int64_t n, int64_t k) {
    GemvGeom g{};
    g.n_rg = n / 4;
    g.nb = static_cast<int>(k / QK);
    g.rpu = g.nb >= 32 ? 1 : 32 / g.nb;
    g.units = (g.n_rg + g.rpu - 1) / g.rpu;
    g.slot_bytes = ((g.rpu * g.nb * BLOCK_BYTES + 16 + 15) / 16) * 16;
    g.sbuf_stride = g.nb + 1;
    const int budget = max_smem_optin() - 1024 - gemv_smem_act_bytes(g.nb);
    g.stages = 3;
    g.warps = 4;
    while (g.warps > 1 && g.warps * gemv_smem_warp_bytes(g) > budget) --g.warps;
    while (g.stages > 2 && g.warps * gemv_smem_warp_bytes(g) > budget) --g.stages;
    return g;
}

cudaError_t launch_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                        const int32_t *bsum, float *y, int32_t *block_sums, int *status, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (k == 0) {
        zero_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, st>>>(y, n);
        return cudaGetLastError();
    }
    const GemvGeom g = gemv_geom(n, k);
    const int smem = gemv_smem_act_bytes(g.nb) + g.warps * gemv_smem_warp_bytes(g);
    cudaError_t e = cudaFuncSetAttribute(gemv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int64_t want = (g.units + g.warps - 1) / g.warps;
    const int grid = static_cast<int>(imin64(want, num_sms()));
    gemv_kernel<<<grid, g.warps * 32, smem, st>>>(static_cast<const uint8_t *>(blocks), g, q, da, bsum, y,
                                                  block_sums, status);
    return cudaGetLastError();
}

}  // namespace tq
