// tqfx4_gemv_mxfp4: the integer dot pass over MXFP4 blocks, the released
// expert bytes of the expert-lossless arm (Sec. 2.3; Table 1 lists them at 4.25
// bits/weight), served directly with no transcode.
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
// P = prmt(table, codes) holds the positive codes' magnitudes (negative codes
// zeroed) and N = prmt(table, codes ^ 0x8888) the negative codes'. Per byte
// one of the two is 0 and both are at most 12, so P + 0x80808080 - N is,
// byte by byte, 128 + c with no carry or borrow between bytes; one unsigned
// x signed dp4a then gives sum (128 + c) q, and the block's accumulator
// starts at -128 * sum q (staged with the activation). The four selector
// nibbles of a word pair a block's elements 2i, 16+2i, 2i+1, 17+2i; the
// activation is staged once per CTA in that interleaved order.
//
// Work split: a row is k/256 groups of 8 blocks (136 bytes each). A warp
// takes a tile of whole rows, R = 32/(k/256) of them (one row of up to 64
// groups for k > 8192), streams it through a two-slot ring of bulk copies,
// and lane l decodes groups l, l + 32 of the tile (its 136 bytes with
// compile-time offsets). Lane r then adds row r's group terms in order.
// The ring has three slots: the copy two tiles ahead goes out before a
// tile is decoded.
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

// activation region: q interleaved (k bytes), -128 * sum q per block (8 L
// ints), da (L floats), then 2^(E-128) for E = 0..255
__host__ __device__ inline int mx_act_bytes(const MxGeo &g) {
    return static_cast<int>(((g.k + 36 * g.L + 127) / 128) * 128) + 1024;
}
constexpr int MX_SLOTS = 3;
__host__ __device__ inline int mx_warp_bytes(const MxGeo &g) { return MX_SLOTS * g.slot + 4 * 32 * g.J + 32; }

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// A word whose low 16 bits are bytes B and B + 1 of the group's 136 bytes
// (B compile-time): the register itself, or one prmt (a constant funnel
// shift costs more than that).
template <int B>
__device__ __forceinline__ uint32_t mx_pair(const uint32_t (&W)[35]) {
    constexpr int A = B >> 2, R = B & 3;
    if constexpr (R == 0)
        return W[A];
    else if constexpr (R == 3)
        return prmt(W[A], W[A + 1], 0x43);
    else
        return prmt(W[A], 0u, R | ((R + 1) << 4));
}

// dp4a of unsigned bytes a and signed bytes b.
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

// Block J of the group: the exact S, and G += float(S) * 2^(E-128) (the
// power of two from the CTA's table of the e8m0 values). S0 = -128 * sum q
// over the block.
template <int J>
__device__ __forceinline__ int mx_block(const uint32_t (&W)[35], const uint4 q0, const uint4 q1, int S0,
                                        const float *p2, float &G, uint32_t &emax) {
    constexpr int off = MX_BYTES * J;
    const uint32_t E = prmt(W[off >> 2], 0u, 0x4440u | (off & 3));
    emax = max(emax, E);
    // selector words: code bytes 1+2i, 2+2i of the block (elements 2i, 16+2i, 2i+1, 17+2i)
    const uint32_t cw[8] = {mx_pair<off + 1>(W), mx_pair<off + 3>(W), mx_pair<off + 5>(W), mx_pair<off + 7>(W),
                            mx_pair<off + 9>(W), mx_pair<off + 11>(W), mx_pair<off + 13>(W), mx_pair<off + 15>(W)};
    const uint32_t qw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
    int S = S0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const uint32_t P = prmt(MX_T0, MX_T1, cw[i]), N = prmt(MX_T0, MX_T1, cw[i] ^ 0x8888u);
        S = dp4a_us(P - N + 0x80808080u, qw[i], S);
    }
    G = __fadd_rn(G, __fmul_rn(static_cast<float>(S), p2[E]));
    return S;
}

template <bool kSums, int J>
__device__ __forceinline__ void mx_blocks(const uint32_t (&W)[35], const uint4 *qv, const int *qc, int L,
                                          const float *p2, float &G, int32_t *S_g, uint32_t &emax) {
    if constexpr (J < QK / MX_K) {
        const int S = mx_block<J>(W, qv[(2 * J) * L], qv[(2 * J + 1) * L], qc[J * L], p2, G, emax);
        if constexpr (kSums) S_g[J] = S;
        mx_blocks<kSums, J + 1>(W, qv, qc, L, p2, G, S_g, emax);
    }
}

// Bounded wait on a ring slot: a lane whose phase is not complete sleeps in
// the barrier unit (suspend-time hint) instead of re-polling, which would
// take issue slots from the warps that decode.
__device__ __forceinline__ uint32_t mx_try_wait_sleep(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
        : "memory");
    return ok;
}
__device__ __forceinline__ bool mx_wait(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (true) {
        if (mx_try_wait_sleep(bar, parity)) return true;
        if (clock64() - t0 > kWaitBudgetCycles) return false;
    }
}

template <bool kSums>
__global__ void __launch_bounds__(MX_WARPS * 32) mxfp4_gemv_kernel(const uint8_t *__restrict__ blocks, MxGeo g,
                                                                   const int8_t *__restrict__ q,
                                                                   const float *__restrict__ da, float *__restrict__ y,
                                                                   int32_t *__restrict__ S_out, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int L = g.L;
    uint4 *qv = reinterpret_cast<uint4 *>(smem);  // [8 blocks][2 halves][L groups]
    int *qc = reinterpret_cast<int *>(smem + g.k);  // [8 blocks][L groups]
    float *das = reinterpret_cast<float *>(smem + g.k + 32 * L);
    float *p2 = reinterpret_cast<float *>(smem + mx_act_bytes(g) - 1024);
    uint8_t *wbase = smem + mx_act_bytes(g) + warp * mx_warp_bytes(g);
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + MX_SLOTS * g.slot);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + MX_SLOTS * g.slot + 4 * 32 * g.J);
    if (lane == 0)
        for (int i = 0; i < MX_SLOTS; ++i) mbar_init(&bars[i], 1);
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
    for (int idx = threadIdx.x; idx < 8 * L; idx += blockDim.x) {
        const int grp = idx % L, j = idx / L;
        const uint4 *src = reinterpret_cast<const uint4 *>(q + static_cast<int64_t>(grp) * QK + j * MX_K);
        int sum = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const uint4 v = __ldg(src + h);
            sum = __dp4a(static_cast<int>(v.x), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.y), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.z), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.w), 0x01010101, sum);
        }
        qc[idx] = -128 * sum;
    }
    for (int i = threadIdx.x; i < L; i += blockDim.x) das[i] = __ldg(da + i);
    // 2^(E-128) for E = 0..254 (0 and 1 subnormal); E = 255 is flagged, its entry unused
    for (int E = threadIdx.x; E < 256; E += blockDim.x)
        p2[E] = __int_as_float(E >= 2 ? (E - 1) << 23 : 0x00200000 << E);
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
    // this lane's groups of a tile: row gr[jj] (R when the lane has none), group gg[jj] of the row
    int gr[2], gg[2];
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) {
        const int tg = lane + 32 * jj;
        gr[jj] = (jj < g.J && tg < g.R * L) ? tg / L : g.R;
        gg[jj] = tg % L;
    }
    uint32_t emax = 0;
    int s = 0, ph = 0;  // slot of this tile, and the parity of its barrier
    for (int64_t tile = first; tile < tiles; tile += NW) {
        if (!__all_sync(0xffffffffu, mx_wait(&bars[s], static_cast<uint32_t>(ph)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, static_cast<int>(tile));
            break;
        }
        // the slot that held the previous tile (read by every lane before
        // the last __syncwarp) takes the tile two steps ahead
        const int s2 = s == 0 ? MX_SLOTS - 1 : s - 1;
        if (tile + 2 * NW < tiles) {
            fence_proxy_async_smem();
            issue(tile + 2 * NW, s2);
        }
        const int rows = rows_of(tile);
        const uint8_t *tp = slots + s * g.slot;
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
            if (gr[jj] >= rows) continue;  // also jj >= J
            const int tg = lane + 32 * jj;  // group of the tile
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
            int32_t *S_g = kSums ? S_out + (tile * g.R + gr[jj]) * nb + gg[jj] * (QK / MX_K) : nullptr;
            mx_blocks<kSums, 0>(W, qv + gg[jj], qc + gg[jj], L, p2, G, S_g, emax);
            tb[tg] = __fmul_rn(G, das[gg[jj]]);
        }
        __syncwarp();
        if (lane < rows) {
            const float2 *t2 = reinterpret_cast<const float2 *>(tb + lane * L);
            float acc = 0.0f;
#pragma unroll 4
            for (int i = 0; i < L / 2; ++i) {
                const float2 v = t2[i];
                acc = __fadd_rn(__fadd_rn(acc, v.x), v.y);
            }
            y[tile * g.R + lane] = acc;
        }
        __syncwarp();
        if (++s == MX_SLOTS) {
            s = 0;
            ph ^= 1;
        }
    }
    if (__any_sync(0xffffffffu, emax == 255u) && lane == 0) report(status, TQFX4_EDATA, K_GEMV, -1);
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
    const void *fn = block_sums ? reinterpret_cast<const void *>(mxfp4_gemv_kernel<true>)
                                : reinterpret_cast<const void *>(mxfp4_gemv_kernel<false>);
    cudaError_t e = allow_max_smem(fn, block_sums ? set : set + 32);
    if (e != cudaSuccess) return e;
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    const int64_t tiles = (n + g.R - 1) / g.R;
    int64_t grid = (tiles + 2 * MX_WARPS - 1) / (2 * MX_WARPS);  // at least two tiles per warp
    const int64_t per_sm = max_smem_optin() / (smem + 1024);
    const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
    if (grid > cap) grid = cap;
    if (block_sums)
        mxfp4_gemv_kernel<true><<<static_cast<unsigned>(grid), MX_WARPS * 32, smem, st>>>(
            static_cast<const uint8_t *>(blocks), g, q, da, y, block_sums, status);
    else
        mxfp4_gemv_kernel<false><<<static_cast<unsigned>(grid), MX_WARPS * 32, smem, st>>>(
            static_cast<const uint8_t *>(blocks), g, q, da, y, nullptr, status);
    return cudaGetLastError();
}

}  // namespace tq
