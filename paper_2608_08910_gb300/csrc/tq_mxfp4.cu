// tqfx4_gemv_mxfp4: the integer dot pass over MXFP4 blocks, the released
// expert bytes that the paper quantizes from (Sec. 2.1; Table 3's 4.25-bit
// format), served directly with no transcode.
//
// Block (OCP microscaling): 17 bytes per 32 elements, the e8m0 scale byte E
// (2^(E-127); E = 255 is NaN) then 16 bytes of e2m1 nibbles, element j < 16
// in the low nibble of byte 1 + j and element 16 + j in the high nibble;
// rows of k/32 blocks contiguous. The doubled e2m1 codes c in
// {0, 1, 2, 3, 4, 6, 8, 12} x sign make a block's sum S = sum c q an exact
// int32 (dp4a on the magnitudes, positive and negative lanes apart); the
// block's contribution is float(S) * (2^(E-128) * da) and a row adds them in
// ascending block order, the oracle's schedule.
//
// One warp per row, rows strided over the grid. Each warp streams its rows
// through a two-slot ring of bulk copies (a row is k/32 * 17 bytes, a
// multiple of 16 for k a multiple of 512); per row, lane l takes blocks l,
// l + 32, ... (17 bytes at an odd offset, read as aligned words and funnel
// shifts), writes the block products to shared memory, and one lane adds
// them in order. The activation (q, da) is staged once per CTA.
#include "tq_common.cuh"
#include "tq_launch.h"

namespace tq {

namespace {

constexpr int MX_K = 32, MX_BYTES = 17;
constexpr int MX_WARPS = 8;

struct MxGeo {
    int64_t n, k;
    int nb;         // blocks per row
    int row_bytes;  // nb * 17
    int slot;       // ring slot bytes: the row, padded for the last block's 5-word read
};

__host__ __device__ inline int mx_slot_bytes(int row_bytes) { return ((row_bytes + 16 + 15) / 16) * 16; }

__host__ inline int mx_smem(const MxGeo &g) {
    // activation (q and da), then per warp: two slots, block products, two barriers
    return static_cast<int>(((g.k + 4 * (g.k / QK) + 127) / 128) * 128) +
           MX_WARPS * (2 * g.slot + 4 * g.nb + 16);
}

// Magnitude codes (bytes, 0..7) to doubled e2m1 magnitudes, four at a time.
__device__ __forceinline__ uint32_t mx_mag(uint32_t codes) {
    const uint32_t t = codes | (codes >> 4);                      // byte 0: c0 | c1 << 4, byte 2: c2 | c3 << 4
    const uint32_t sel = (t & 0xffu) | ((t >> 8) & 0xff00u);      // four 4-bit selectors
    return __byte_perm(0x03020100u, 0x0C080604u, sel);            // 0,1,2,3 | 4,6,8,12
}

// S += sum of four signed doubled codes (nibbles in the bytes of `nib`) times q.
__device__ __forceinline__ int mx_dot4(uint32_t nib, uint32_t q, int S) {
    const uint32_t mag = mx_mag(nib & 0x07070707u);
    const uint32_t neg = ((nib >> 3) & 0x01010101u) * 0xffu;     // 0xff in the bytes of negative codes
    S = __dp4a(static_cast<int>(mag & ~neg), static_cast<int>(q), S);
    return S - __dp4a(static_cast<int>(mag & neg), static_cast<int>(q), 0);
}

__global__ void __launch_bounds__(MX_WARPS * 32) mxfp4_gemv_kernel(const uint8_t *__restrict__ blocks, MxGeo g,
                                                                   const int8_t *__restrict__ q,
                                                                   const float *__restrict__ da, float *__restrict__ y,
                                                                   int32_t *__restrict__ S_out, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t *qs = smem;
    float *das = reinterpret_cast<float *>(smem + g.k);
    uint8_t *wbase = smem + ((g.k + 4 * (g.k / QK) + 127) / 128) * 128 + warp * (2 * g.slot + 4 * g.nb + 16);
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + 2 * g.slot);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + 2 * g.slot + 4 * g.nb);
    if (lane == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
    }
    fence_barrier_init();
    for (int64_t i = threadIdx.x; i < g.k / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(qs)[i] = __ldg(reinterpret_cast<const uint4 *>(q) + i);
    for (int64_t i = threadIdx.x; i < g.k / QK; i += blockDim.x) das[i] = __ldg(da + i);
    __syncthreads();

    const int64_t NW = static_cast<int64_t>(gridDim.x) * MX_WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * MX_WARPS + warp;
    auto issue = [&](int64_t row, int s) {
        if (lane == 0) {
            mbar_arrive_expect_tx(&bars[s], static_cast<uint32_t>(g.row_bytes));
            bulk_g2s(slots + s * g.slot, blocks + row * g.row_bytes, static_cast<uint32_t>(g.row_bytes), &bars[s]);
        }
    };
    if (first < g.n) issue(first, 0);
    if (first + NW < g.n) issue(first + NW, 1);
    int it = 0;
    bool bad = false;
    for (int64_t row = first; row < g.n; row += NW, ++it) {
        const int s = it & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[s], static_cast<uint32_t>((it >> 1) & 1)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(row));
            break;
        }
        const uint8_t *rowp = slots + s * g.slot;
        const uint32_t *rw = reinterpret_cast<const uint32_t *>(rowp);
        for (int b = lane; b < g.nb; b += 32) {
            const int off = MX_BYTES * b;
            uint32_t w[6];
#pragma unroll
            for (int i = 0; i < 6; ++i) w[i] = rw[(off >> 2) + i];
            // realign: a[i] holds block bytes 4 i .. 4 i + 3
            const uint32_t sh = static_cast<uint32_t>(off & 3) * 8;
            uint32_t a[5];
#pragma unroll
            for (int i = 0; i < 5; ++i) a[i] = __funnelshift_r(w[i], w[i + 1], sh);
            const uint32_t E = a[0] & 0xffu;
            bad |= E == 255u;
            const uint32_t *qw = reinterpret_cast<const uint32_t *>(qs + b * MX_K);
            int S = 0;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t cw = __funnelshift_r(a[i], a[i + 1], 8);  // code bytes 1 + 4 i .. 4 + 4 i
                S = mx_dot4(cw & 0x0f0f0f0fu, qw[i], S);                 // elements 4 i .. 4 i + 3
                S = mx_dot4((cw >> 4) & 0x0f0f0f0fu, qw[4 + i], S);      // elements 16 + 4 i ..
            }
            if (S_out) S_out[row * g.nb + b] = S;
            // 2^(E-128) * da: exact (a power of two times da); E = 0 gives 2^-128
            const float sc = __fmul_rn(ldexpf(1.0f, static_cast<int>(E) - 128), das[(b * MX_K) / QK]);
            tb[b] = __fmul_rn(static_cast<float>(S), sc);
        }
        __syncwarp();
        // refill this slot with the row two steps ahead before the row sum
        if (row + 2 * NW < g.n) {
            fence_proxy_async_smem();
            issue(row + 2 * NW, s);
        }
        if (lane == 0) {
            float acc = 0.0f;
            for (int b = 0; b < g.nb; ++b) acc = __fadd_rn(acc, tb[b]);
            y[row] = acc;
        }
        __syncwarp();
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) report(status, TQFX4_EDATA, K_GEMV, -1);
}

}  // namespace

int64_t mxfp4_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || k % MX_K) return -1;
    return n * (k / MX_K) * MX_BYTES;
}

cudaError_t launch_mxfp4_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                              int32_t *block_sums, int *status, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    MxGeo g;
    g.n = n;
    g.k = k;
    g.nb = static_cast<int>(k / MX_K);
    g.row_bytes = g.nb * MX_BYTES;
    g.slot = mx_slot_bytes(g.row_bytes);
    const int smem = mx_smem(g);
    static unsigned char set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(mxfp4_gemv_kernel), set);
    if (e != cudaSuccess) return e;
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    const int64_t rows_per_cta = MX_WARPS * 2;  // two rows per warp in flight
    int64_t grid = (n + rows_per_cta - 1) / rows_per_cta;
    const int64_t cap = static_cast<int64_t>(num_sms()) * (max_smem_optin() / (smem + 1024 > 0 ? smem + 1024 : 1));
    if (grid > cap && cap > 0) grid = cap;
    mxfp4_gemv_kernel<<<static_cast<unsigned>(grid), MX_WARPS * 32, smem, st>>>(
        static_cast<const uint8_t *>(blocks), g, q, da, y, block_sums, status);
    return cudaGetLastError();
}

}  // namespace tq
