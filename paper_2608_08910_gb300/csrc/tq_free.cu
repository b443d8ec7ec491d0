// The free-scale two-plane format (Table 1's free-scale K=2 row, 4.125
// bits/weight): W = a1 t1 + a2 t2 per row and 256 columns with two
// independent f16 scales, the two trit planes stored apart because the pair
// does not fold. Blocks of 4 rows x 256 columns, 528 bytes, ordered
// [N/4 row groups][K/256 blocks]: bytes 0..7 a1 of rows 0..3, 8..15 a2,
// then per row r at 16 + 128 r the plane t1 (64 bytes) and the plane t2 (64
// bytes), element j in bits 2 (j % 4) of byte j / 4 as u = t + 1 (3 is
// invalid).
//
// tqfx4_pack_free: one warp per (row, 256-block), lane l packs elements
// 8l .. 8l + 7 of both planes.
//
// tqfx4_gemv_free: the two-plane dot pass. Exact sums S = sum t q per plane
// and block, then per block float(S1) * (a1 * da) + float(S2) * (a2 * da)
// added to the row's sum in block order (the oracle's schedule). A warp
// takes row groups (4 rows) and streams each as chunks of up to 8 blocks
// (4224 bytes) through a three-slot ring of bulk copies; in a chunk lane l
// takes the (row, block) pair l, and lanes 0..3 carry the row sums from
// chunk to chunk. A plane word
// holds 16 trits; its four 2-bit fields per byte are masked in place
// (x & (0x03030303 << 2i), no shift) so that the unsigned x signed dp4a
// sums 4^i u q into accumulator i; the four accumulators are shifted back
// exactly (each is a multiple of 4^i) and sum u q - sum q = sum t q. The
// activation is staged once per CTA with the four bytes of each dp4a word
// transposed to match the fields (elements 4b + i of a 16-element word).
#include "tq_common.cuh"
#include "tq_launch.h"

namespace tq {

namespace {

constexpr int FR_BLOCK = 528, FR_PLANE_OFS = 16, FR_ROW = 128;
constexpr int FR_SLOTS = 3;
constexpr int FR_WARPS = 8;
constexpr int FR_CHUNK = 8;  // blocks of a row group per copy: 4 rows x 8 blocks = one pair per lane

__global__ void __launch_bounds__(256) pack_free_kernel(const int8_t *__restrict__ t1, const int8_t *__restrict__ t2,
                                                        const uint16_t *__restrict__ a1,
                                                        const uint16_t *__restrict__ a2, int64_t n, int64_t k,
                                                        uint8_t *__restrict__ out, int *status) {
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t L = k / QK;
    if (w >= n * L) return;
    const int64_t row = w / L, b = w - row * L;
    const int r = static_cast<int>(row & 3);
    uint8_t *blk = out + ((row >> 2) * L + b) * FR_BLOCK;
    const int64_t src = row * k + b * QK + 8 * lane;
    bool bad = false;
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        const uint2 v = __ldg(reinterpret_cast<const uint2 *>((p ? t2 : t1) + src));
        const uint32_t words[2] = {v.x, v.y};
        uint32_t packed = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int t = static_cast<int8_t>((words[h] >> (8 * e)) & 0xffu);
                bad |= t < -1 || t > 1;
                packed |= static_cast<uint32_t>((t + 1) & 3) << (8 * h + 2 * e);
            }
        *reinterpret_cast<uint16_t *>(blk + FR_PLANE_OFS + FR_ROW * r + 64 * p + 2 * lane) =
            static_cast<uint16_t>(packed);
    }
    if (lane == 0) {
        reinterpret_cast<uint16_t *>(blk)[r] = a1[row * L + b];
        reinterpret_cast<uint16_t *>(blk + 8)[r] = a2[row * L + b];
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) report(status, TQFX4_EDATA, K_PACK, static_cast<int>(w));
}

__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

// sum u q over both planes of one (row, block): 16 words a plane, each
// with its transposed activation word group (loaded once for the two
// planes); acc[p][i] collects 4^i u q of plane p.
__device__ __forceinline__ void free_pair_sums(const uint4 *pw, const uint4 *qv, int L, int &U1, int &U2) {
    int acc[2][4] = {{0, 0, 0, 0}, {0, 0, 0, 0}};
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        const uint4 x4[2] = {pw[c], pw[4 + c]};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const uint4 qq = qv[(4 * c + e) * L];
#pragma unroll
            for (int p = 0; p < 2; ++p) {
                const uint32_t x = e == 0 ? x4[p].x : e == 1 ? x4[p].y : e == 2 ? x4[p].z : x4[p].w;
                acc[p][0] = dp4a_us(x & 0x03030303u, qq.x, acc[p][0]);
                acc[p][1] = dp4a_us(x & 0x0c0c0c0cu, qq.y, acc[p][1]);
                acc[p][2] = dp4a_us(x & 0x30303030u, qq.z, acc[p][2]);
                acc[p][3] = dp4a_us(x & 0xc0c0c0c0u, qq.w, acc[p][3]);
            }
        }
    }
    U1 = acc[0][0] + (acc[0][1] >> 2) + (acc[0][2] >> 4) + (acc[0][3] >> 6);
    U2 = acc[1][0] + (acc[1][1] >> 2) + (acc[1][2] >> 4) + (acc[1][3] >> 6);
}

__device__ __forceinline__ bool free_wait(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    return mbar_wait(bar, parity);
}

struct FreeGeo {
    int64_t n, k;
    int L;  // 256-blocks per row
    int C;  // blocks per chunk (one bulk copy): min(8, L)
    int Q;  // chunks per row group
};

__host__ __device__ inline int free_act_bytes(int L) { return ((L * (QK + 8) + 127) / 128) * 128; }
__host__ __device__ inline int free_warp_bytes(const FreeGeo &g) {
    return FR_SLOTS * g.C * FR_BLOCK + 4 * ROWS * g.C + 32;
}

// The fields of plane word w of a block: byte b of transposed word i is
// element 16 w + 4 b + i.
__device__ __forceinline__ uint4 free_transpose(uint4 v) {
    const uint32_t t01l = __byte_perm(v.x, v.y, 0x5140), t23l = __byte_perm(v.z, v.w, 0x5140);
    const uint32_t t01h = __byte_perm(v.x, v.y, 0x7362), t23h = __byte_perm(v.z, v.w, 0x7362);
    return make_uint4(__byte_perm(t01l, t23l, 0x5410), __byte_perm(t01l, t23l, 0x7632),
                      __byte_perm(t01h, t23h, 0x5410), __byte_perm(t01h, t23h, 0x7632));
}

template <bool kSums>
__global__ void __launch_bounds__(FR_WARPS * 32) gemv_free_kernel(const uint8_t *__restrict__ blocks, FreeGeo g,
                                                                  const int8_t *__restrict__ q,
                                                                  const float *__restrict__ da,
                                                                  const int32_t *__restrict__ bsum,
                                                                  float *__restrict__ y, int32_t *__restrict__ S1o,
                                                                  int32_t *__restrict__ S2o, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int L = g.L, C = g.C, Q = g.Q;
    uint4 *qv = reinterpret_cast<uint4 *>(smem);  // [16 words][L blocks]
    float *das = reinterpret_cast<float *>(smem + L * QK);
    int *bss = reinterpret_cast<int *>(smem + L * QK + 4 * L);
    uint8_t *wbase = smem + free_act_bytes(L) + warp * free_warp_bytes(g);
    uint8_t *slots = wbase;
    const int slot = C * FR_BLOCK;
    float *tb = reinterpret_cast<float *>(wbase + FR_SLOTS * slot);  // [4 rows][C]
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + FR_SLOTS * slot + 4 * ROWS * C);
    if (lane == 0)
        for (int i = 0; i < FR_SLOTS; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();

    // a warp's work: row groups first, first + NW, ..., each as Q chunks in
    // order; u numbers the warp's chunks
    const int64_t groups = g.n / ROWS;
    const int64_t NW = static_cast<int64_t>(gridDim.x) * FR_WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * FR_WARPS + warp;
    const int64_t my_groups = first < groups ? (groups - first + NW - 1) / NW : 0;
    const int64_t units = my_groups * Q;
    const uint64_t policy = l2_policy_evict_first();
    auto chunk_blocks = [&](int qi) { return qi == Q - 1 ? L - qi * C : C; };
    // the next chunk to copy (row group, chunk), advanced by every lane alike
    int64_t rg_n = first;
    int qi_n = 0;
    auto issue_next = [&](int s) {
        if (lane == 0) {
            const uint32_t bytes = static_cast<uint32_t>(chunk_blocks(qi_n) * FR_BLOCK);
            mbar_arrive_expect_tx(&bars[s], bytes);
            bulk_g2s_hint(slots + s * slot, blocks + (rg_n * L + static_cast<int64_t>(qi_n) * C) * FR_BLOCK, bytes,
                          &bars[s], policy);
        }
        if (++qi_n == Q) {
            qi_n = 0;
            rg_n += NW;
        }
    };
    if (units > 0) issue_next(0);
    if (units > 1) issue_next(1);
    for (int idx = threadIdx.x; idx < 16 * L; idx += blockDim.x) {
        const int b = idx % L, wd = idx / L;
        qv[idx] = free_transpose(__ldg(reinterpret_cast<const uint4 *>(q + b * QK + 16 * wd)));
    }
    for (int i = threadIdx.x; i < L; i += blockDim.x) {
        das[i] = __ldg(da + i);
        bss[i] = __ldg(bsum + i);
    }
    __syncthreads();

    float acc = 0.0f;  // lanes 0..3: the running sum of row `lane` of the current group
    int s = 0, ph = 0;
    int64_t rg = first;  // the current chunk (row group, chunk)
    int qi = 0;
    for (int64_t u = 0; u < units; ++u) {
        if (!__all_sync(0xffffffffu, free_wait(&bars[s], static_cast<uint32_t>(ph)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(u));
            break;
        }
        // the slot of the previous chunk (read before the last __syncwarp)
        // takes the chunk two ahead
        if (u + 2 < units) {
            fence_proxy_async_smem();
            issue_next(s == 0 ? FR_SLOTS - 1 : s - 1);
        }
        const int cb = chunk_blocks(qi);
        const uint8_t *tp = slots + s * slot;
        auto pair = [&](int r, int bl) {
            const int b = qi * C + bl;
            const uint8_t *blk = tp + bl * FR_BLOCK;
            const uint4 *pl = reinterpret_cast<const uint4 *>(blk + FR_PLANE_OFS + FR_ROW * r);
            int U1, U2;
            free_pair_sums(pl, qv + b, L, U1, U2);
            const int S1 = U1 - bss[b], S2 = U2 - bss[b];
            const float a1 = __half2float(reinterpret_cast<const __half *>(blk)[r]);
            const float a2 = __half2float(reinterpret_cast<const __half *>(blk + 8)[r]);
            const float p1 = __fmul_rn(static_cast<float>(S1), __fmul_rn(a1, das[b]));
            const float p2 = __fmul_rn(static_cast<float>(S2), __fmul_rn(a2, das[b]));
            tb[r * C + bl] = __fadd_rn(p1, p2);
            if (kSums) {
                const int64_t o = (rg * ROWS + r) * L + b;
                S1o[o] = S1;
                S2o[o] = S2;
            }
        };
        if (cb == FR_CHUNK) {
            pair(lane >> 3, lane & 7);  // a full chunk: one pair per lane
        } else {
            for (int p = lane; p < ROWS * cb; p += 32) {
                const int r = p / cb;
                pair(r, p - r * cb);
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
        if (++s == FR_SLOTS) {
            s = 0;
            ph ^= 1;
        }
    }
}

}  // namespace

int64_t free_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || n % ROWS || k % QK) return -1;
    return (n / ROWS) * (k / QK) * FR_BLOCK;
}

cudaError_t launch_pack_free(const int8_t *t1, const int8_t *t2, const uint16_t *a1, const uint16_t *a2, int64_t n,
                             int64_t k, void *out, int *status, cudaStream_t st) {
    const int64_t warps = n * (k / QK);
    if (warps == 0) return cudaSuccess;
    pack_free_kernel<<<static_cast<unsigned>((warps * 32 + 255) / 256), 256, 0, st>>>(
        t1, t2, a1, a2, n, k, static_cast<uint8_t *>(out), status);
    return cudaGetLastError();
}

int gemv_free_smem(int64_t k) {
    FreeGeo g{};
    g.L = static_cast<int>(k / QK);
    g.C = g.L < FR_CHUNK ? g.L : FR_CHUNK;
    return free_act_bytes(g.L) + FR_WARPS * free_warp_bytes(g);
}

cudaError_t launch_gemv_free(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                             const int32_t *bsum, float *y, int32_t *S1, int32_t *S2, int *status,
                             cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    FreeGeo g{};
    g.n = n;
    g.k = k;
    g.L = static_cast<int>(k / QK);
    g.C = g.L < FR_CHUNK ? g.L : FR_CHUNK;
    g.Q = (g.L + g.C - 1) / g.C;
    const int smem = gemv_free_smem(k);
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    static unsigned char set[2][64];
    const bool sums = S1 != nullptr;
    const void *fn = sums ? reinterpret_cast<const void *>(gemv_free_kernel<true>)
                          : reinterpret_cast<const void *>(gemv_free_kernel<false>);
    cudaError_t e = allow_max_smem(fn, set[sums ? 1 : 0]);
    if (e != cudaSuccess) return e;
    const int64_t groups = n / ROWS;
    int64_t grid = (groups + FR_WARPS - 1) / FR_WARPS;
    const int64_t per_sm = max_smem_optin() / (smem + 1024);
    const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
    if (grid > cap) grid = cap;
    const unsigned gr = static_cast<unsigned>(grid);
    const uint8_t *b = static_cast<const uint8_t *>(blocks);
    if (sums)
        gemv_free_kernel<true><<<gr, FR_WARPS * 32, smem, st>>>(b, g, q, da, bsum, y, S1, S2, status);
    else
        gemv_free_kernel<false><<<gr, FR_WARPS * 32, smem, st>>>(b, g, q, da, bsum, y, nullptr, nullptr, status);
    return cudaGetLastError();
}

}  // namespace tq
