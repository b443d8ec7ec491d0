// tqfx4_gemv: the integer dot pass of Tied Trit-Planes Sec. 2.2 on GB300.
//
// Data path: a matrix is one contiguous stream of 520-byte blocks. The grid
// splits it into one contiguous range of row groups per CTA; each warp of a
// CTA streams units of that range through its own shared-memory ring with
// cp.async.bulk (tq_stream.cuh) and applies the fixed float schedule
// acc = acc + float(S) * (d * da) over the blocks in ascending order.
#include "tq_launch.h"
#include "tq_stream.cuh"

namespace tq {

// One CTA streams a contiguous range of row groups; its warps split the range
// into units (see tq_stream.cuh).
struct GemvGeom {
    int64_t n_rg;     // row groups in the matrix
    int nb;           // blocks per row group (K / 256)
    int rpu;          // row groups per unit
    int slot_bytes;   // per slot, 16-byte multiple, including the alignment pad
    int stages;       // slots per warp
    int warps;        // warps per CTA
    int64_t rg_per_cta;
};

__host__ __device__ inline int gemv_act_bytes(int nb) { return ((nb * (QS_STRIDE + 8) + 127) / 128) * 128; }

__global__ void __launch_bounds__(256, 1) gemv_kernel(const uint8_t *__restrict__ blocks, GemvGeom g,
                                                      const int8_t *__restrict__ q,
                                                      const float *__restrict__ da,
                                                      const int32_t *__restrict__ bsum, float *__restrict__ y,
                                                      int32_t *__restrict__ s_out, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5;
    const int nb = g.nb;
    uint8_t *qs = smem;
    float *das = reinterpret_cast<float *>(smem + nb * QS_STRIDE);
    int *bss = reinterpret_cast<int *>(das + nb);
    const WarpRing ring = carve_ring(smem + gemv_act_bytes(nb) + warp * stream_warp_bytes(g.stages, g.slot_bytes,
                                                                                         g.rpu, nb),
                                     g.stages, g.slot_bytes, g.rpu, nb);
    ring_init(ring);
    fence_barrier_init();
    MatJob job;
    job.mat = blocks;
    job.rg_begin = static_cast<int64_t>(blockIdx.x) * g.rg_per_cta;
    job.rg_end = imin64(job.rg_begin + g.rg_per_cta, g.n_rg);
    job.y = y;
    job.s_out = s_out;
    job.qs = qs;
    job.das = das;
    job.bss = bss;
    job.nb = nb;
    if (job.rg_begin < job.rg_end) warp_stream_prefetch(ring, job, g.rpu, warp, g.warps);
    load_act_smem(q, da, bsum, nb, qs, das, bss);
    __syncthreads();
    if (job.rg_begin < job.rg_end) warp_stream_run(ring, job, g.rpu, warp, g.warps, status, K_GEMV);
}

__global__ void zero_kernel(float *y, int64_t n) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i < n) y[i] = 0.0f;
}

// Device attributes, cached per device (the only state the library keeps).
namespace {
constexpr int kMaxDevices = 64;
int g_sms[kMaxDevices];
int g_smem[kMaxDevices];

int current_device() {
    int dev = 0;
    cudaGetDevice(&dev);
    return (dev >= 0 && dev < kMaxDevices) ? dev : 0;
}
}  // namespace

int num_sms() {
    const int dev = current_device();
    if (g_sms[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        g_sms[dev] = v > 0 ? v : 148;
    }
    return g_sms[dev];
}

int max_smem_optin() {
    const int dev = current_device();
    if (g_smem[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
        g_smem[dev] = v > 0 ? v : 232448;
    }
    return g_smem[dev];
}

// Raise a kernel's dynamic shared-memory limit to the device maximum less its
// static shared memory, once per (kernel, device); `flags` is the kernel's
// own per-device flag array.
cudaError_t allow_max_smem(const void *kernel, unsigned char *flags) {
    const int dev = current_device();
    if (flags[dev]) return cudaSuccess;
    cudaFuncAttributes attr;
    cudaError_t e = cudaFuncGetAttributes(&attr, kernel);
    if (e != cudaSuccess) return e;
    const int dyn = max_smem_optin() - static_cast<int>(attr.sharedSizeBytes);
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) flags[dev] = 1;
    return e;
}

static GemvGeom gemv_geom(int64_t n, int64_t k) {
    GemvGeom g{};
    g.n_rg = n / 4;
    g.nb = static_cast<int>(k / QK);
    g.rpu = pow2_rows(32, g.nb);
    g.slot_bytes = stream_slot_bytes(g.rpu, g.nb);
    const int budget = max_smem_optin() - 1024 - gemv_act_bytes(g.nb);
    g.stages = 2;
    g.warps = 8;
    while (g.warps > 1 && g.warps * stream_warp_bytes(g.stages, g.slot_bytes, g.rpu, g.nb) > budget) --g.warps;
    const int64_t units = (g.n_rg + g.rpu - 1) / g.rpu;
    const int64_t ctas = imax64(1, imin64(num_sms(), (units + g.warps - 1) / g.warps));
    const int64_t upc = (units + ctas - 1) / ctas;  // units per CTA
    g.rg_per_cta = upc * g.rpu;
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
    const int smem = gemv_act_bytes(g.nb) + g.warps * stream_warp_bytes(g.stages, g.slot_bytes, g.rpu, g.nb);
    static unsigned char smem_set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(gemv_kernel), smem_set);
    if (e != cudaSuccess) return e;
    const int grid = static_cast<int>((g.n_rg + g.rg_per_cta - 1) / g.rg_per_cta);
    gemv_kernel<<<grid, g.warps * 32, smem, st>>>(static_cast<const uint8_t *>(blocks), g, q, da, bsum, y,
                                                  block_sums, status);
    return cudaGetLastError();
}

}  // namespace tq
