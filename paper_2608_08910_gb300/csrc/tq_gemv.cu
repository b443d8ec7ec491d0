// tqfx4_gemv: the integer dot pass of Tied Trit-Planes Sec. 2.2 on GB300.
//
// Data path: a matrix is one contiguous stream of 520-byte blocks, and the
// fixed float schedule acc = acc + float(S) * (d * da) runs over the blocks
// of a row in ascending order. For k a multiple of 512 the chunked pass
// below streams row groups in chunks of up to 16 blocks, two rows of a
// block per lane;
// otherwise (rows 8-byte aligned) the grid splits the matrix into one
// contiguous range of row groups per CTA and each warp streams units of it
// through the engine of tq_stream.cuh.
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
    grid_dependency_wait();  // the blocks, q, da and bsum may come from the previous kernel
    grid_dependents_launch();
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

// ---- the chunked pass (k a multiple of 512) ----------------------------
//
// A warp takes row groups (first, first + NW, ...) and streams each as
// chunks of up to 16 blocks (8320 bytes) through a three-slot ring of bulk
// copies. In a full chunk lane l takes rows 2 (l / 16), 2 (l / 16) + 1 of
// block l % 16: 128 code bytes a row (element j in the low nibble of byte j,
// element 128 + j in the high one), the two rows sharing the activation
// loads, with the activation laid out [16-byte word][block] in shared
// memory so that lanes on different blocks read different banks. Lanes 0..3 carry their row's sum from chunk to
// chunk; the float schedule is the one above.
constexpr int FX_SLOTS = 3, FX_WARPS = 8, FX_CHUNK = 16;

struct FxGeo {
    int64_t n;
    int L, C, Q;  // blocks per row group, per chunk (min(FX_CHUNK, L)), chunks per row group
};

__host__ __device__ inline int fx_act_bytes(int L) { return ((L * (QK + 8) + 127) / 128) * 128; }
__host__ __device__ inline int fx_warp_bytes(const FxGeo &g) {
    return FX_SLOTS * g.C * BLOCK_BYTES + 4 * ROWS * g.C + 32;
}

// Exact S of two rows of a block (codes: the first row's 128 bytes, the
// second row 128 bytes on): 32 code words a row against the activation
// words w (low nibbles) and 32 + w (high nibbles, kept at 16 u and divided
// out), S = sum u q - 4 bsum; the activation words are loaded once for both.
__device__ __forceinline__ void fx_row2_dot(const uint2 *codes, const uint4 *qv, int L, int bsum, int &S0,
                                            int &S1) {
    int lo[2] = {0, 0}, hi[2] = {0, 0};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const uint4 ql = qv[i * L], qh = qv[(8 + i) * L];  // activation words 4i..4i+3 and 32+4i..
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const uint2 c0 = codes[16 * r + 2 * i], c1 = codes[16 * r + 2 * i + 1];
            lo[r] = dp4a_us(c0.x & 0x0f0f0f0fu, ql.x, lo[r]);
            lo[r] = dp4a_us(c0.y & 0x0f0f0f0fu, ql.y, lo[r]);
            lo[r] = dp4a_us(c1.x & 0x0f0f0f0fu, ql.z, lo[r]);
            lo[r] = dp4a_us(c1.y & 0x0f0f0f0fu, ql.w, lo[r]);
            hi[r] = dp4a_us(c0.x & 0xf0f0f0f0u, qh.x, hi[r]);
            hi[r] = dp4a_us(c0.y & 0xf0f0f0f0u, qh.y, hi[r]);
            hi[r] = dp4a_us(c1.x & 0xf0f0f0f0u, qh.z, hi[r]);
            hi[r] = dp4a_us(c1.y & 0xf0f0f0f0u, qh.w, hi[r]);
        }
    }
    S0 = lo[0] + (hi[0] >> 4) - 4 * bsum;
    S1 = lo[1] + (hi[1] >> 4) - 4 * bsum;
}

// kFromX: the activation is the fp32 vector x, quantized per 256-block by
// each CTA into its shared memory with the quantizer of tqfx4_quantize_act
// (CTA 0 also writes q, da and bsum where given); otherwise it is the
// quantized vector (q, da, bsum).
template <bool kSums, bool kFromX>
__global__ void __launch_bounds__(FX_WARPS * 32) gemv_chunk_kernel(const uint8_t *__restrict__ blocks, FxGeo g,
                                                                   const int8_t *__restrict__ q,
                                                                   const float *__restrict__ da,
                                                                   const int32_t *__restrict__ bsum,
                                                                   float *__restrict__ y,
                                                                   int32_t *__restrict__ s_out, int *status,
                                                                   const float *__restrict__ x, int8_t *q_out,
                                                                   float *da_out, int32_t *bsum_out) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int L = g.L, C = g.C, Q = g.Q;
    uint4 *qv = reinterpret_cast<uint4 *>(smem);  // [16 words][L blocks]
    float *das = reinterpret_cast<float *>(smem + L * QK);
    int *bss = reinterpret_cast<int *>(smem + L * QK + 4 * L);
    uint8_t *wbase = smem + fx_act_bytes(L) + warp * fx_warp_bytes(g);
    const int slot = C * BLOCK_BYTES;
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + FX_SLOTS * slot);  // [4 rows][C]
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + FX_SLOTS * slot + 4 * ROWS * C);
    if (lane == 0)
        for (int i = 0; i < FX_SLOTS; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
    grid_dependency_wait();  // the blocks, q, da and bsum may come from the previous kernel
    grid_dependents_launch();

    const int64_t groups = g.n / ROWS;
    const int64_t NW = static_cast<int64_t>(gridDim.x) * FX_WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * FX_WARPS + warp;
    const int64_t units = first < groups ? (groups - first + NW - 1) / NW * Q : 0;
    const uint64_t policy = l2_policy_evict_first();
    auto chunk_blocks = [&](int qi) { return qi == Q - 1 ? L - qi * C : C; };
    int64_t rg_n = first;  // the next chunk to copy
    int qi_n = 0;
    auto issue_next = [&](int s) {
        if (lane == 0) {
            const uint32_t bytes = static_cast<uint32_t>(chunk_blocks(qi_n) * BLOCK_BYTES);
            mbar_arrive_expect_tx(&bars[s], bytes);
            bulk_g2s_hint(slots + s * slot, blocks + (rg_n * L + static_cast<int64_t>(qi_n) * C) * BLOCK_BYTES,
                          bytes, &bars[s], policy);
        }
        if (++qi_n == Q) {
            qi_n = 0;
            rg_n += NW;
        }
    };
    if (units > 0) issue_next(0);
    if (units > 1) issue_next(1);
    if constexpr (kFromX) {
        // one warp per 256-block while the first copies fly; lane l's eight
        // codes are bytes 8 l .. 8 l + 7 of the block: half l % 2 of word l / 2
        bool finite = true;
        for (int b = warp; b < L; b += FX_WARPS) {
            const float4 *src = reinterpret_cast<const float4 *>(x + b * QK + 8 * lane);
            const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
            const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            uint2 packed;
            float d;
            int sum;
            finite &= quant_block_warp(v, packed, d, sum);
            reinterpret_cast<uint2 *>(qv + (lane >> 1) * L + b)[lane & 1] = packed;
            if (lane == 0) {
                das[b] = d;
                bss[b] = sum;
            }
            if (blockIdx.x == 0 && q_out) {
                *reinterpret_cast<uint2 *>(q_out + b * QK + 8 * lane) = packed;
                if (lane == 0) {
                    da_out[b] = d;
                    bsum_out[b] = sum;
                }
            }
        }
        if (!finite && blockIdx.x == 0 && lane == 0) report(status, TQFX4_EDATA, K_QUANT, -1);
        __syncwarp();
    } else {
        for (int idx = threadIdx.x; idx < 16 * L; idx += blockDim.x) {
            const int b = idx % L, wd = idx / L;
            qv[idx] = __ldg(reinterpret_cast<const uint4 *>(q + b * QK + 16 * wd));
        }
        for (int i = threadIdx.x; i < L; i += blockDim.x) {
            das[i] = __ldg(da + i);
            bss[i] = __ldg(bsum + i);
        }
    }
    __syncthreads();

    float acc = 0.0f;  // lanes 0..3: the running sum of row `lane` of the current group
    int s = 0, ph = 0;
    int64_t rg = first;
    int qi = 0;
    for (int64_t u = 0; u < units; ++u) {
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[s], static_cast<uint32_t>(ph)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(u));
            break;
        }
        if (u + 2 < units) {  // the slot of the previous chunk takes the chunk two ahead
            fence_proxy_async_smem();
            issue_next(s == 0 ? FX_SLOTS - 1 : s - 1);
        }
        const int cb = chunk_blocks(qi);
        const uint8_t *tp = slots + s * slot;
        // rows 2 rp and 2 rp + 1 of block bl of the chunk
        auto pair = [&](int rp, int bl) {
            const int b = qi * C + bl;
            const uint8_t *blk = tp + bl * BLOCK_BYTES;
            int S[2];
            fx_row2_dot(reinterpret_cast<const uint2 *>(blk + CODE_OFS + 256 * rp), qv + b, L, bss[b], S[0], S[1]);
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const int r = 2 * rp + i;
                const float sc = __fmul_rn(block_scale(blk, r), das[b]);
                tb[r * C + bl] = __fmul_rn(static_cast<float>(S[i]), sc);
                if (kSums) s_out[(rg * ROWS + r) * L + b] = S[i];
            }
        };
        if (cb == FX_CHUNK) {
            pair(lane >> 4, lane & 15);
        } else {
            for (int p = lane; p < 2 * cb; p += 32) {
                const int rp = p / cb;
                pair(rp, p - rp * cb);
            }
        }
        __syncwarp();
        if (lane < ROWS) {
            if (qi == 0) acc = 0.0f;
            for (int bl = 0; bl < cb; ++bl) acc = __fadd_rn(acc, tb[lane * C + bl]);
            if (qi == Q - 1) y[rg * ROWS + lane] = acc;
        }
        __syncwarp();
        if (++qi == Q) {
            qi = 0;
            rg += NW;
        }
        if (++s == FX_SLOTS) {
            s = 0;
            ph ^= 1;
        }
    }
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
    if (k % 512 == 0) {  // the chunked pass (row groups start 16-byte aligned)
        FxGeo f{};
        f.n = n;
        f.L = static_cast<int>(k / QK);
        f.C = f.L < FX_CHUNK ? f.L : FX_CHUNK;
        f.Q = (f.L + f.C - 1) / f.C;
        const int smem = fx_act_bytes(f.L) + FX_WARPS * fx_warp_bytes(f);
        static unsigned char set[2][64];
        const bool sums = block_sums != nullptr;
        const void *fn = sums ? reinterpret_cast<const void *>(gemv_chunk_kernel<true, false>)
                              : reinterpret_cast<const void *>(gemv_chunk_kernel<false, false>);
        cudaError_t e = allow_max_smem(fn, set[sums ? 1 : 0]);
        if (e != cudaSuccess) return e;
        if (smem > max_smem_optin()) return cudaErrorInvalidValue;
        const int64_t groups = n / ROWS;
        const int64_t per_sm = max_smem_optin() / (smem + 1024);
        int64_t grid = (groups + FX_WARPS - 1) / FX_WARPS;
        const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
        if (grid > cap) grid = cap;
        const uint8_t *b = static_cast<const uint8_t *>(blocks);
        const dim3 gd(static_cast<unsigned>(grid)), bd(FX_WARPS * 32);
        const float *nx = nullptr;
        int8_t *nq = nullptr;
        float *nd = nullptr;
        int32_t *ns = nullptr;
        if (sums)
            return launch_dependent(gemv_chunk_kernel<true, false>, gd, bd, smem, st, b, f, q, da, bsum, y, block_sums,
                                    status, nx, nq, nd, ns);
        return launch_dependent(gemv_chunk_kernel<false, false>, gd, bd, smem, st, b, f, q, da, bsum, y,
                                static_cast<int32_t *>(nullptr), status, nx, nq, nd, ns);
    }
    const GemvGeom g = gemv_geom(n, k);
    const int smem = gemv_act_bytes(g.nb) + g.warps * stream_warp_bytes(g.stages, g.slot_bytes, g.rpu, g.nb);
    static unsigned char smem_set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(gemv_kernel), smem_set);
    if (e != cudaSuccess) return e;
    const int grid = static_cast<int>((g.n_rg + g.rg_per_cta - 1) / g.rg_per_cta);
    return launch_dependent(gemv_kernel, dim3(grid), dim3(g.warps * 32), smem, st, static_cast<const uint8_t *>(blocks),
                            g, q, da, bsum, y, block_sums, status);
}

// The chunked pass with the activation quantized inside (kFromX): k a
// multiple of 512 (the caller checks).
cudaError_t launch_gemv_x(const void *blocks, int64_t n, int64_t k, const float *x, int8_t *q, float *da,
                          int32_t *bsum, float *y, int *status, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    FxGeo f{};
    f.n = n;
    f.L = static_cast<int>(k / QK);
    f.C = f.L < FX_CHUNK ? f.L : FX_CHUNK;
    f.Q = (f.L + f.C - 1) / f.C;
    const int smem = fx_act_bytes(f.L) + FX_WARPS * fx_warp_bytes(f);
    static unsigned char set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(gemv_chunk_kernel<false, true>), set);
    if (e != cudaSuccess) return e;
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    const int64_t groups = n / ROWS;
    const int64_t per_sm = max_smem_optin() / (smem + 1024);
    int64_t grid = (groups + FX_WARPS - 1) / FX_WARPS;
    const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
    if (grid > cap) grid = cap;
    const int8_t *nq = nullptr;
    const float *nd = nullptr;
    const int32_t *ns = nullptr;
    return launch_dependent(gemv_chunk_kernel<false, true>, dim3(static_cast<unsigned>(grid)), dim3(FX_WARPS * 32),
                            smem, st, static_cast<const uint8_t *>(blocks), f, nq, nd, ns, y,
                            static_cast<int32_t *>(nullptr), status, x, q, da, bsum);
}

}  // namespace tq
