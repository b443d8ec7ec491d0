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
#include "tq_moe_common.cuh"

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

// activation region: per activation q interleaved (k bytes), -128 * sum q
// per block (8 L ints) and da (L floats); then 2^(E-128) for E = 0..255
__host__ __device__ inline int mx_act_unit(const MxGeo &g) { return static_cast<int>(((g.k + 36 * g.L + 15) / 16) * 16); }
__host__ __device__ inline int mx_act_bytes(const MxGeo &g, int acts) {
    return ((acts * mx_act_unit(g) + 127) / 128) * 128 + 1024;
}

// The matrices of one launch, all n x k: matrix m (of n_mat <= 2K) is
// base[m / K] + sel[m % K] * mat_bytes (sel null: base[m / K]), takes
// activation m % K when acts > 1 (else the only one), and writes y[m / K] +
// (m % K) * n. One matrix: K = 1, n_mat = 1 (block sums only then).
struct MxJob {
    const uint8_t *base[2];
    int64_t mat_bytes;
    const int32_t *sel;
    int K, n_mat, acts;
    const int8_t *q;  // [acts][k]
    const float *da;  // [acts][k / 256]
    float *y[2];
    int32_t *S;  // nullable block sums [n_mat * n][k / 32]
    // per-matrix mode: CTA c serves matrix c % K only, and builds its
    // activation as the int8 quantization of h = silu(g_j) * u_j from these
    // ([K][k] fp32 each) instead of reading q and da
    const float *g, *u;
};

// Kernel modes: one matrix; several matrices sharing the CTAs; several
// matrices with the CTAs split among them (activation from g and u).
enum { MX_ONE = 0, MX_SHARED = 1, MX_PER_MAT = 2 };
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

// Stages activation `a` (q [k] int8, da [k/256]) into the interleaved layout.
__device__ __forceinline__ void mx_stage_act(uint8_t *dst, const MxGeo &g, const int8_t *q, const float *da) {
    const int L = g.L;
    for (int r = threadIdx.x; r < 16 * L; r += blockDim.x) {
        const int grp = r % L, jh = r / L;
        const int8_t *src = q + grp * QK + (jh >> 1) * MX_K + (jh & 1) * 8;
        const uint2 x0 = __ldg(reinterpret_cast<const uint2 *>(src));
        const uint2 x1 = __ldg(reinterpret_cast<const uint2 *>(src + 16));
        reinterpret_cast<uint4 *>(dst)[r] =
            make_uint4(__byte_perm(x0.x, x1.x, 0x5140), __byte_perm(x0.x, x1.x, 0x7362),
                       __byte_perm(x0.y, x1.y, 0x5140), __byte_perm(x0.y, x1.y, 0x7362));
    }
    for (int r = threadIdx.x; r < 8 * L; r += blockDim.x) {
        const int grp = r % L, j = r / L;
        const uint4 *src = reinterpret_cast<const uint4 *>(q + grp * QK + j * MX_K);
        int sum = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const uint4 v = __ldg(src + h);
            sum = __dp4a(static_cast<int>(v.x), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.y), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.z), 0x01010101, sum);
            sum = __dp4a(static_cast<int>(v.w), 0x01010101, sum);
        }
        reinterpret_cast<int *>(dst + g.k)[r] = -128 * sum;
    }
    for (int r = threadIdx.x; r < L; r += blockDim.x) reinterpret_cast<float *>(dst + g.k + 32 * L)[r] = __ldg(da + r);
}

// Builds the activation from h = silu(g) * u (k elements, fp32): one warp
// per 256-element block, the decode path's SwiGLU and quantizer, written
// straight into the interleaved layout. Returns false if h is not finite.
__device__ __forceinline__ bool mx_stage_swiglu(uint8_t *dst, const MxGeo &g, const float *gv, const float *uv) {
    const int L = g.L, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    bool ok = true;
    for (int b = warp; b < L; b += MX_WARPS) {
        const int o = b * QK + 8 * lane;
        const float4 g0 = __ldcg(reinterpret_cast<const float4 *>(gv + o));
        const float4 g1 = __ldcg(reinterpret_cast<const float4 *>(gv + o) + 1);
        const float4 u0 = __ldcg(reinterpret_cast<const float4 *>(uv + o));
        const float4 u1 = __ldcg(reinterpret_cast<const float4 *>(uv + o) + 1);
        const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
        const float uu[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
        float hv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) hv[i] = tq_swiglu(gg[i], uu[i]);
        uint2 pk;
        float d;
        int bsum;
        ok &= quant_block_warp(hv, pk, d, bsum);
        // lane holds elements 8 (lane % 4) .. + 7 of 32-block lane / 4: the
        // half-block words pair lanes l and l + 2 (elements e and 16 + e)
        const uint2 hi = make_uint2(__shfl_down_sync(0xffffffffu, pk.x, 2), __shfl_down_sync(0xffffffffu, pk.y, 2));
        const int jb = lane >> 2, part = lane & 3;
        if (part < 2)
            reinterpret_cast<uint4 *>(dst)[(2 * jb + part) * L + b] =
                make_uint4(__byte_perm(pk.x, hi.x, 0x5140), __byte_perm(pk.x, hi.x, 0x7362),
                           __byte_perm(pk.y, hi.y, 0x5140), __byte_perm(pk.y, hi.y, 0x7362));
        int sum = __dp4a(static_cast<int>(pk.x), 0x01010101, __dp4a(static_cast<int>(pk.y), 0x01010101, 0));
        sum += __shfl_xor_sync(0xffffffffu, sum, 1);
        sum += __shfl_xor_sync(0xffffffffu, sum, 2);
        if (part == 0) reinterpret_cast<int *>(dst + g.k)[jb * L + b] = -128 * sum;
        if (lane == 0) reinterpret_cast<float *>(dst + g.k + 32 * L)[b] = d;
    }
    return ok;
}

template <bool kSums, int kMode>
__global__ void __launch_bounds__(MX_WARPS * 32) mxfp4_gemv_kernel(MxGeo g, MxJob job, int *status) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int L = g.L, AU = mx_act_unit(g);
    const int acts = kMode == MX_SHARED ? job.acts : 1;
    const int act_bytes = mx_act_bytes(g, acts);
    float *p2 = reinterpret_cast<float *>(smem + act_bytes - 1024);
    uint8_t *wbase = smem + act_bytes + warp * mx_warp_bytes(g);
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + MX_SLOTS * g.slot);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + MX_SLOTS * g.slot + 4 * 32 * g.J);
    if (lane == 0)
        for (int i = 0; i < MX_SLOTS; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
    // 2^(E-128) for E = 0..254 (0 and 1 subnormal); E = 255 is flagged, its entry unused
    for (int E = threadIdx.x; E < 256; E += blockDim.x)
        p2[E] = __int_as_float(E >= 2 ? (E - 1) << 23 : 0x00200000 << E);
    // everything below may read the previous kernel's results
    grid_dependency_wait();

    const int tpm = static_cast<int>((g.n + g.R - 1) / g.R);  // tiles per matrix
    // the CTA's matrix (per-matrix mode) and the tiles its warps take
    const int cta_m = kMode == MX_PER_MAT ? static_cast<int>(blockIdx.x) % job.K : 0;
    const int cta_p = kMode == MX_PER_MAT ? static_cast<int>(blockIdx.x) / job.K : static_cast<int>(blockIdx.x);
    const int n_cta = kMode == MX_PER_MAT ? static_cast<int>(gridDim.x) / job.K : static_cast<int>(gridDim.x);
    const int tiles = kMode == MX_SHARED ? tpm * job.n_mat : tpm;
    const int NW = n_cta * MX_WARPS;
    const int first = cta_p * MX_WARPS + warp;
    const uint64_t policy = l2_policy_evict_first();
    auto locate = [&](int tile, int &m, int &t) {
        m = kMode == MX_SHARED ? tile / tpm : cta_m;
        t = tile - (kMode == MX_SHARED ? m * tpm : 0);
    };
    auto rows_of = [&](int t) {
        const int64_t left = g.n - static_cast<int64_t>(t) * g.R;
        return static_cast<int>(left < g.R ? left : g.R);
    };
    auto issue = [&](int tile, int s) {
        if (lane == 0) {
            int m, t;
            locate(tile, m, t);
            const uint8_t *mat = job.base[0];
            if (kMode != MX_ONE)
                mat = (m >= job.K ? job.base[1] : job.base[0]) + (job.sel ? job.sel[m % job.K] : 0) * job.mat_bytes;
            const uint32_t bytes = static_cast<uint32_t>(rows_of(t) * g.row_bytes);
            mbar_arrive_expect_tx(&bars[s], bytes);
            bulk_g2s_hint(slots + s * g.slot, mat + static_cast<int64_t>(t) * g.R * g.row_bytes, bytes, &bars[s],
                          policy);
        }
    };
    // the first weight tiles go out before the activation is staged
    if (first < tiles) issue(first, 0);
    if (first + NW < tiles) issue(first + NW, 1);
    if (kMode == MX_PER_MAT) {
        if (!mx_stage_swiglu(smem, g, job.g + static_cast<int64_t>(cta_m) * g.k,
                             job.u + static_cast<int64_t>(cta_m) * g.k) &&
            lane == 0)
            report(status, TQFX4_EDATA, K_DOWN, cta_m);
    } else {
        for (int a = 0; a < acts; ++a)
            mx_stage_act(smem + a * AU, g, job.q + static_cast<int64_t>(a) * g.k, job.da + static_cast<int64_t>(a) * L);
    }
    __syncthreads();
    grid_dependents_launch();

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
    for (int tile = first; tile < tiles; tile += NW) {
        if (!__all_sync(0xffffffffu, mx_wait(&bars[s], static_cast<uint32_t>(ph)))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, K_GEMV, tile);
            break;
        }
        // the slot that held the previous tile (read by every lane before
        // the last __syncwarp) takes the tile two steps ahead
        const int s2 = s == 0 ? MX_SLOTS - 1 : s - 1;
        if (tile + 2 * NW < tiles) {
            fence_proxy_async_smem();
            issue(tile + 2 * NW, s2);
        }
        int m, t;
        locate(tile, m, t);
        const int jm = kMode == MX_ONE ? 0 : m % job.K;
        const uint8_t *act = smem + (kMode == MX_SHARED && acts > 1 ? jm : 0) * AU;
        const uint4 *qv = reinterpret_cast<const uint4 *>(act);
        const int *qc = reinterpret_cast<const int *>(act + g.k);
        const float *das = reinterpret_cast<const float *>(act + g.k + 32 * L);
        const int rows = rows_of(t);
        const int64_t row0 = static_cast<int64_t>(m) * g.n + static_cast<int64_t>(t) * g.R;
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
            int32_t *S_g = kSums ? job.S + (row0 + gr[jj]) * nb + gg[jj] * (QK / MX_K) : nullptr;
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
            float *yb = kMode == MX_SHARED && m >= job.K ? job.y[1] : job.y[0];
            yb[static_cast<int64_t>(jm) * g.n + static_cast<int64_t>(t) * g.R + lane] = acc;
        }
        __syncwarp();
        if (++s == MX_SLOTS) {
            s = 0;
            ph ^= 1;
        }
    }
    if (__any_sync(0xffffffffu, emax == 255u) && lane == 0) report(status, TQFX4_EDATA, K_GEMV, -1);
}

// out[n] = sum over j in rank order of w_j * o_j[n] (binary32, no fused multiply-add).
__global__ void __launch_bounds__(256) mx_combine_kernel(const float *__restrict__ o, const float *__restrict__ w,
                                                         int K, int H, float *__restrict__ out) {
    grid_dependency_wait();  // o of the down projections
    const int n = blockIdx.x * blockDim.x + threadIdx.x;
    if (n >= H) return;
    float acc = 0.0f;
    for (int j = 0; j < K; ++j) acc = __fadd_rn(acc, __fmul_rn(__ldg(w + j), __ldg(o + static_cast<int64_t>(j) * H + n)));
    out[n] = acc;
}

}  // namespace

int64_t mxfp4_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || k % MX_K) return -1;
    return n * (k / MX_K) * MX_BYTES;
}

static MxGeo mx_geo(int64_t n, int64_t k) {
    MxGeo g;
    g.n = n;
    g.k = k;
    g.L = static_cast<int>(k / QK);
    g.R = g.L <= 32 ? 32 / g.L : 1;
    g.J = (g.L + 31) / 32;
    g.row_bytes = g.L * MX_GB;
    g.slot = ((g.R * g.row_bytes + 15) / 16) * 16;
    return g;
}

int mxfp4_gemv_smem(int64_t k, int acts) {
    const MxGeo g = mx_geo(1, k);
    return mx_act_bytes(g, acts) + MX_WARPS * mx_warp_bytes(g);
}

// One launch of the kernel in `mode`; `pdl`: as a programmatic dependent of
// the previous kernel in the stream. Per-matrix mode: `ctas_per_mat` CTAs
// per matrix.
static cudaError_t launch_job(const MxGeo &g, const MxJob &job, int mode, bool pdl, int *status, cudaStream_t st) {
    const int smem = mx_act_bytes(g, mode == MX_SHARED ? job.acts : 1) + MX_WARPS * mx_warp_bytes(g);
    static unsigned char set[4][64];
    const bool sums = job.S != nullptr;
    const int v = mode == MX_ONE ? (sums ? 1 : 0) : mode + 1;
    const void *fns[4] = {reinterpret_cast<const void *>(mxfp4_gemv_kernel<false, MX_ONE>),
                          reinterpret_cast<const void *>(mxfp4_gemv_kernel<true, MX_ONE>),
                          reinterpret_cast<const void *>(mxfp4_gemv_kernel<false, MX_SHARED>),
                          reinterpret_cast<const void *>(mxfp4_gemv_kernel<false, MX_PER_MAT>)};
    cudaError_t e = allow_max_smem(fns[v], set[v]);
    if (e != cudaSuccess) return e;
    if (smem > max_smem_optin()) return cudaErrorInvalidValue;
    const int64_t tpm = (g.n + g.R - 1) / g.R;
    const int64_t per_sm = max_smem_optin() / (smem + 1024);
    const int64_t cap = static_cast<int64_t>(num_sms()) * (per_sm > 0 ? per_sm : 1);
    int64_t grid;
    if (mode == MX_PER_MAT) {
        // the CTAs that fit, split evenly among the matrices (at least two tiles per warp)
        int64_t per = cap / job.K;
        const int64_t need = (tpm + 2 * MX_WARPS - 1) / (2 * MX_WARPS);
        if (per > need) per = need;
        if (per < 1) per = 1;
        grid = per * job.K;
    } else {
        grid = (tpm * (mode == MX_SHARED ? job.n_mat : 1) + 2 * MX_WARPS - 1) / (2 * MX_WARPS);
        if (grid > cap) grid = cap;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(MX_WARPS * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    MxGeo ga = g;
    MxJob ja = job;
    void *args[] = {&ga, &ja, &status};
    return cudaLaunchKernelExC(&cfg, fns[v], args);
}

cudaError_t launch_mxfp4_gemv(const void *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                              int32_t *block_sums, int *status, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    MxJob job{};
    job.base[0] = job.base[1] = static_cast<const uint8_t *>(blocks);
    job.K = job.n_mat = job.acts = 1;
    job.q = q;
    job.da = da;
    job.y[0] = job.y[1] = y;
    job.S = block_sums;
    return launch_job(mx_geo(n, k), job, MX_ONE, false, status, st);
}

// ev (nullable): events recorded before gate/up, down (SwiGLU and the
// quantization of h run in its prologue) and combine, and after combine.
cudaError_t launch_moe_mxfp4_experts(const MoeArgs &a, float *out, cudaStream_t st, const cudaEvent_t *ev) {
    const int K = a.top_k;
    if (ev) record_stage_event(ev[0], st);
    // gate and up of the selected experts: 2K matrices of I x H, one activation
    MxJob gu{};
    gu.base[0] = a.gate;
    gu.base[1] = a.up;
    gu.mat_bytes = a.mb_gu;
    gu.sel = a.sel;
    gu.K = K;
    gu.n_mat = 2 * K;
    gu.acts = 1;
    gu.q = a.qx;
    gu.da = a.dx;
    gu.y[0] = a.g;
    gu.y[1] = a.u;
    cudaError_t e = launch_job(mx_geo(a.I, a.H), gu, MX_SHARED, ev == nullptr, a.status, st);
    if (e != cudaSuccess) return e;
    if (ev) record_stage_event(ev[1], st);
    // down: K matrices of H x I, the CTAs split among the experts, each
    // forming its expert's activation from g and u
    MxJob dn{};
    dn.base[0] = dn.base[1] = a.down;
    dn.mat_bytes = a.mb_d;
    dn.sel = a.sel;
    dn.K = K;
    dn.n_mat = K;
    dn.acts = 1;
    dn.g = a.g;
    dn.u = a.u;
    dn.y[0] = dn.y[1] = a.o;
    if ((e = launch_job(mx_geo(a.H, a.I), dn, MX_PER_MAT, ev == nullptr, a.status, st)) != cudaSuccess) return e;
    if (ev) record_stage_event(ev[2], st);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((a.H + 255) / 256);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = ev ? 0 : 1;
    const float *o = a.o, *w = a.selw;
    int Kk = K, H = a.H;
    void *args[] = {&o, &w, &Kk, &H, &out};
    e = cudaLaunchKernelExC(&cfg, reinterpret_cast<const void *>(mx_combine_kernel), args);
    if (ev) record_stage_event(ev[3], st);
    return e;
}

}  // namespace tq
