// tqfx4_gemv_mxfp4: the integer dot pass over MXFP4 blocks, the released
// expert bytes that the paper quantizes from (Sec. 2.1; Table 3's 4.25-bit
// format), served directly with no transcode.
//
// Block (OCP microscaling): 17 bytes per 32 elements, the e8m0 scale byte E
// (2^(E-127); E = 255 is NaN) then 16 bytes of e2m1 nibbles, element j < 16
// in the low nibble of byte 1 + j and element 16 + j in the high nibble;
// rows of k/32 blocks contiguous. The doubled e2m1 codes c in
// {0, 1, 2, 3, 4, 6, 8, 12} x sign make a block's sum S = sum c q an exact
// int32, and its value t = float(S) * 2^(E-128) is exact too. Float schedule
// (the activation's scale unit): per 256-element group g, G = G + t over its
// eight blocks in order, then y = y + G * da[g] over the groups in order.
//
// Decode of a nibble without masks or branches: prmt picks byte m of the
// table {0, 1, 2, 3, 4, 6, 8, 12} for a selector nibble (s, m), and for s = 1
// replicates that byte's sign bit instead, which is 0 for every entry. So
// prmt(table, codes) is the positive codes' magnitudes with the negative
// codes zeroed, prmt(table, codes ^ 0x8888...) the negative codes'
// magnitudes, and S = dp4a(P, q) - dp4a(N, q). The four selector nibbles of
// a word pair a block's elements 4i, 16+4i, 4i+1, 17+4i; the activation is
// staged once per CTA in that interleaved order.
//
// Work split: a row is k/256 groups of 8 blocks (136 bytes each). A warp
// takes a tile of whole rows, R = 32/(k/256) of them (one row of up to 64
// groups for k > 8192), streams it through a two-slot ring of bulk copies,
// and lane l decodes groups l, l + 32 of the tile (its 136 bytes with
// compile-time offsets). Lane r then adds row r's group terms in order.
#include "tq_common.cuh"
#include "tq_launch.h"

namespace tq {

namespace {

constexpr int MX_K = 32, MX_BYTES = 17;
constexpr int MX_GB = (QK / MX_K) * MX_BYTES;  // 136 bytes per 256-element group
constexpr int MX_WARPS = 8;
constexpr uint32_t MX_T0 = 0x03020100u, MX_T1 = 0x0C080604u;  // doubled e2m1 magnitudes

struct MxGeo {
    int64_t n, k;
    int L;          // 256-element groups per row
    int R;          // rows per warp tile
    int J;          // groups per lane (2 when a row has more than 32)
    int row_bytes;  // L * 136
    int slot;       // ring slot bytes (a tile, a multiple of 16)
};

__host__ __device__ inline int mx_act_bytes(const MxGeo &g) {
    return static_cast<int>(((g.k + 4 * g.L + 127) / 128) * 128);
}
__host__ __device__ inline int mx_warp_bytes(const MxGeo &g) { return 2 * g.slot + 4 * 32 * g.J + 16; }

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// 2^(E-128) as binary32, E in 0..254 (E = 0 and 1 are subnormal).
__device__ __forceinline__ float mx_pow2(uint32_t E) {
    return __int_as_float(E >= 2u ? static_cast<int>((E - 1u) << 23) : static_cast<int>(0x00200000u << E));
}

// Bytes 4A + SH/8 .. of the group's 136 bytes as one word (compile-time).
template <int A, int SH>
__device__ __forceinline__ uint32_t mx_word(const uint32_t (&W)[35]) {
    if constexpr (SH == 0)
        return W[A];
    else
        return __funnelshift_r(W[A], W[A + 1], SH);
}

// Block J of the group: the exact S, and G += float(S) * 2^(E-128).
template <int J>
__device__ __forceinline__ void mx_block(const uint32_t (&W)[35], const uint4 q0, const uint4 q1, float &G, int &S,
                                         bool &bad) {
    constexpr int off = MX_BYTES * J;
    const uint32_t E = (W[off >> 2] >> ((off & 3) * 8)) & 0xffu;
    bad |= E == 255u;
    const uint32_t cw[4] = {mx_word<((off + 1) >> 2), (((off + 1) & 3) * 8)>(W),
                            mx_word<((off + 5) >> 2), (((off + 5) & 3) * 8)>(W),
                            mx_word<((off + 9) >> 2), (((off + 9) & 3) * 8)>(W),
                            mx_word<((off + 13) >> 2), (((off + 13) & 3) * 8)>(W)};
    const uint32_t qw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
    int sp = 0, sn = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t c = cw[i], ci = c ^ 0x88888888u;
        sp = __dp4a(static_cast<int>(prmt(MX_T0, MX_T1, c)), static_cast<int>(qw[2 * i]), sp);
        sp = __dp4a(static_cast<int>(prmt(MX_T0, MX_T1, c >> 16)), static_cast<int>(qw[2 * i + 1]), sp);
        sn = __dp4a(static_cast<int>(prmt(MX_T0, MX_T1, ci)), static_cast<int>(qw[2 * i]), sn);
        sn = __dp4a(static_cast<int>(prmt(MX_T0, MX_T1, ci >> 16)), static_cast<int>(qw[2 * i + 1]), sn);
    }
    S = sp - sn;
    G = __fadd_rn(G, __fmul_rn(static_cast<float>(S), mx_pow2(E)));
}

template <int J>
__device__ __forceinline__ void mx_blocks(const uint32_t (&W)[35], const uint4 *qv, int L, float &G, int32_t *S_g,
                                          bool &bad) {
    if constexpr (J < QK / MX_K) {
        int S;
        mx_block<J>(W, qv[(2 * J) * L], qv[(2 * J + 1) * L], G, S, bad);
        if (S_g) S_g[J] = S;
        mx_blocks<J + 1>(W, qv, L, G, S_g, bad);
    }
}

__global__ void __launch_bounds__(MX_WARPS * 32) mxfp4_gemv_kernel(const uint8_t *__restrict__ blocks, MxGeo g,
                                                                   const int8_t *__restrict__ q,
                                                                   const float *__restrict__ da, float *__restrict__ y,
                                                                   int32_t *__restrict__ S_out, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int L = g.L;
    uint4 *qv = reinterpret_cast<uint4 *>(smem);  // [8 blocks][2 halves][L groups]
    float *das = reinterpret_cast<float *>(smem + g.k);
    uint8_t *wbase = smem + mx_act_bytes(g) + warp * mx_warp_bytes(g);
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + 2 * g.slot);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + 2 * g.slot + 4 * 32 * g.J);
    if (lane == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
    }
    fence_barrier_init();
    // the activation, interleaved per 16-element half block: bytes
    // q[8h + e] and q[16 + 8h + e] alternate
    for (int idx = threadIdx.x; idx < 16 * L; idx += blockDim.x) {
        const int grp = idx % L, jh = idx / L;
        const int8_t *src = q + static_cast<int64_t>(grp) * QK + (jh >> 1) * MX_K + (jh & 1) * 8;
        const uint2 a = __ldg(reinterpret_cast<const uint2 *>(src));
        const uint2 b = __ldg(reinterpret_cast<const uint2 *>(src + 16));
        qv[idx] = make_uint4(__byte_perm(a.x, b.x, 0x5140), __byte_perm(a.x, b.x, 0x7362),
                             __byte_perm(a.y, b.y, 0x5140), __byte_perm(a.y, b.y, 0x7362));
    }
    for (int i = threadIdx.x; i < L; i += blockDim.x) das[i] = __ldg(da + i);
    __syncthreads();

    const int64_t tiles = (g.n + g.R - 1) / g.R;
    const int64_t NW = static_cast<int64_t>(gridDim.x) * MX_WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * MX_WARPS + warp;
    const uint64_t policy = l2_policy_evict_first();
    auto rows_of = [&](int64_t tile) {
        const int64_t left = g.n - tile * g.R;
        return static_cast<int>(left < g.R ? left : g.R);
    };
    auto issue = [&](int64_t tile, int s) {
        if (lane == 0) {
            const uint32_t bytes = static_cast<uint32_t>(rows_of(tile) * g.row_bytes);
            mbar_arrive_expect_tx(&bars[s], bytes);
            bulk_g2s_hint(slots + s * g.slot, blocks + tile * g.R * g.row_bytes, bytes, &bars[s], policy);
        }
    };
    if (first < tiles) issue(first, 0);
    if (first + NW < tiles) issue(first + NW, 1);
    const int nb = L * (QK / MX_K);
    int it = 0;
    bool bad = false;
    for (int64_t tile = first; tile < tiles; tile += NW, ++it) {
        const int s = it & 1;
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[s], static_cast<uint32_t>((it >> 1) & 1)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(tile));
            break;
        }
        const int rows = rows_of(tile);
        const uint8_t *tp = slots + s * g.slot;
        for (int jj = 0; jj < g.J; ++jj) {
            const int tg = lane + 32 * jj;  // group of the tile
            if (tg >= rows * L) continue;
            const int r = tg / L, grp = tg - r * L;
            uint32_t W[35];
            const uint2 *src = reinterpret_cast<const uint2 *>(tp + tg * MX_GB);
#pragma unroll
            for (int i = 0; i < MX_GB / 8; ++i) {
                const uint2 v = src[i];
                W[2 * i] = v.x;
                W[2 * i + 1] = v.y;
            }
            W[34] = 0u;
            float G = 0.0f;
            int32_t *S_g = S_out ? S_out + (tile * g.R + r) * nb + grp * (QK / MX_K) : nullptr;
            mx_blocks<0>(W, qv + grp, L, G, S_g, bad);
            tb[tg] = __fmul_rn(G, das[grp]);
        }
        __syncwarp();
        // refill this slot with the tile two steps ahead, then the row sums
        if (tile + 2 * NW < tiles) {
            fence_proxy_async_smem();
            issue(tile + 2 * NW, s);
        }
        if (lane < rows) {
            float acc = 0.0f;
            for (int i = 0; i < L; ++i) acc = __fadd_rn(acc, tb[lane * L + i]);
            y[tile * g.R + lane] = acc;
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
    g.L = static_cast<int>(k / QK);
    g.R = g.L <= 32 ? 32 / g.L : 1;
    g.J = (g.L + 31) / 32;
    g.row_bytes = g.L * MX_GB;
    g.slot = ((g.R * g.row_bytes + 15) / 16) * 16;
    const int smem = mx_act_bytes(g) + MX_WARPS * mx_warp_bytes(g);
    static unsigned char set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(mxfp4_gemv_kernel), set);
    if (e != cudaSuccess) return e;
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    const int64_t tiles = (n + g.R - 1) / g.R;
    int64_t grid = (tiles + 2 * MX_WARPS - 1) / (2 * MX_WARPS);  // two tiles per warp in flight
    const int64_t per_sm = max_smem_optin() / (smem + 1024);
    const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
    if (grid > cap) grid = cap;
    mxfp4_gemv_kernel<<<static_cast<unsigned>(grid), MX_WARPS * 32, smem, st>>>(
        static_cast<const uint8_t *>(blocks), g, q, da, y, block_sums, status);
    return cudaGetLastError();
}

}  // namespace tq
