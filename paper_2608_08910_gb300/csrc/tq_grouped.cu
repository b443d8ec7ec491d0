// tqfx4_moe_grouped: T tokens through the routed-expert MoE layer, grouped
// by expert so each touched expert's weights are read once for all its
// tokens (batched decode and prefill).
//
// Stages (one launch each):
//   router   logits of every (token, expert) by the compensated dot product
//   topk     per token: top-k selection and softmax weights
//   group    counts per expert, exclusive scan, stable gather of the
//            (token, slot) pairs (expert, then ascending token), and the
//            work list of <= 64-pair chunks per expert
//   quant_x  int8 quantization of the T hidden states
//   gate_up  grouped GEMM of the gate and up projections over the chunks
//   swiglu   h = silu(g) u per pair and its int8 quantization
//   down     grouped GEMM of the down projection
//   combine  out[t] = sum_j w[t][j] o[pair(t, j)] in rank order
//
// The grouped GEMM computes, per 256-element block, the exact integer block
// sums U = sum u q of 128 weight rows x 64 pairs with warp-level int8 MMAs
// (mma.sync m16n8k32, s8 x s8 -> s32; the nibbles u = c + 4 are the A
// operand, S = U - 4 bsum), then applies the fixed float schedule
// y = y + float(S) * (d * da) block by block, so its outputs are the
// oracle's, bit for bit. One producer warp streams each stage (two blocks of
// 32 row groups plus the chunk's activation rows) with cp.async.bulk; eight
// consumer warps each own 16 weight rows.
#include "tq_launch.h"
#include "tq_moe_common.cuh"

namespace tq {



// ---------------------------------------------------------------- router

constexpr int RB_TOK = 16;  // tokens per CTA (4 per warp)

__global__ void __launch_bounds__(128) router_batch_kernel(GroupedArgs a) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int e = blockIdx.x;
    const float *w = a.wr + static_cast<int64_t>(e) * a.H;
    for (int i = 0; i < RB_TOK / 4; ++i) {
        const int t = blockIdx.y * RB_TOK + warp * (RB_TOK / 4) + i;
        if (t >= a.T) break;
        float hi, lo;
        router_logit_warp(w, a.X + static_cast<int64_t>(t) * a.H, a.H, hi, lo);
        if (lane == 0) {
            if (a.bias) ff_add(hi, lo, __ldg(a.bias + e), 0.0f, hi, lo);
            a.logits[static_cast<int64_t>(t) * a.E + e] = hi;
            a.logits_lo[static_cast<int64_t>(t) * a.E + e] = lo;
        }
    }
}

// ---------------------------------------------------------------- top-k

__global__ void __launch_bounds__(128) topk_batch_kernel(GroupedArgs a) {
    __shared__ TopkScratch s;
    const int t = blockIdx.x, lane = threadIdx.x & 31;
    const int k = a.top_k;
    const float *lh = a.logits + static_cast<int64_t>(t) * a.E;
    const float *ll = a.logits_lo + static_cast<int64_t>(t) * a.E;
    int *sel = a.sel + static_cast<int64_t>(t) * k;
    __shared__ float w[TQFX4_MAX_TOP_K];
    topk_block(lh, ll, a.E, k, sel, s);
    if (threadIdx.x >= 32) return;
    softmax_ff_warp(lh, ll, s.res, k, w);
    if (lane < k) {
        a.selw[static_cast<int64_t>(t) * k + lane] = w[lane];
        a.sel_out[static_cast<int64_t>(t) * k + lane] = s.res[lane];
        a.selw_out[static_cast<int64_t>(t) * k + lane] = w[lane];
    }
}

// ---------------------------------------------------------------- group

// Inclusive scan of one value per thread over a block of 1024 threads.
__device__ __forceinline__ int block_scan_1024(int v, int *warp_tot) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += n;
    }
    if (lane == 31) warp_tot[warp] = v;
    __syncthreads();
    if (warp == 0) {
        int w = warp_tot[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += n;
        }
        warp_tot[lane] = w;
    }
    __syncthreads();
    const int r = v + (warp > 0 ? warp_tot[warp - 1] : 0);
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(1024) group_kernel(GroupedArgs a) {
    __shared__ int cnt[TQFX4_MAX_EXPERTS], off[TQFX4_MAX_EXPERTS + 1], run[TQFX4_MAX_EXPERTS];
    __shared__ int warp_tot[32];
    const int tid = threadIdx.x, lane = tid & 31;
    const int E = a.E, P = a.P, k = a.top_k;
    if (tid < E) {
        cnt[tid] = 0;
        run[tid] = 0;
    }
    __syncthreads();
    for (int p = tid; p < P; p += blockDim.x) atomicAdd(&cnt[__ldcg(a.sel + p)], 1);
    __syncthreads();
    const int c = tid < E ? cnt[tid] : 0;
    const int incl = block_scan_1024(c, warp_tot);
    if (tid < E) {
        off[tid + 1] = incl;
        a.counts[tid] = c;
        a.offsets[tid + 1] = incl;
    }
    if (tid == 0) {
        off[0] = 0;
        a.offsets[0] = 0;
    }
    // chunk list: ceil(count / GG_TOK) chunks per expert
    const int nc = (c + GG_TOK - 1) / GG_TOK;
    const int cincl = block_scan_1024(nc, warp_tot);
    if (tid < E) {
        const int base = cincl - nc;
        for (int i = 0; i < nc; ++i) {
            a.chunk_expert[base + i] = tid;
            a.chunk_begin[base + i] = incl - c + i * GG_TOK;
            a.chunk_len[base + i] = min(GG_TOK, c - i * GG_TOK);
        }
    }
    if (tid == blockDim.x - 1) *a.n_chunks = cincl;
    __syncthreads();
    // stable placement by one warp: pairs visited in (token, slot) order
    if (tid < 32) {
        const unsigned lt = (1u << lane) - 1u;
        for (int base = 0; base < P; base += 32) {
            const int p = base + lane;
            const bool valid = p < P;
            const int e = valid ? __ldcg(a.sel + p) : -1 - lane;
            const unsigned peers = __match_any_sync(0xffffffffu, e);
            const int rank = __popc(peers & lt);
            const int leader = __ffs(peers) - 1;
            int b = 0;
            if (valid && lane == leader) {
                b = run[e];
                run[e] = b + __popc(peers);
            }
            b = __shfl_sync(0xffffffffu, b, leader);
            if (valid) {
                const int pos = off[e] + b + rank;
                a.pair_token[pos] = p / k;
                a.pair_slot[pos] = p - (p / k) * k;
                a.pair_of[p] = pos;
            }
            __syncwarp();
        }
    }
}

// ---------------------------------------------------------------- grouped GEMM

constexpr int GG_CW = 8;                       // consumer warps, 16 weight rows each
constexpr int GG_RG = GG_CW * 16 / 4;          // 32 row groups per tile
constexpr int GG_KB = 2;                       // 256-blocks per stage
constexpr int GG_STAGES = 3;
constexpr int GG_WROW = GG_KB * BLOCK_BYTES;   // 1040 bytes per row group per stage
constexpr int GG_TSTRIDE = GG_KB * QK + 32;    // 544: activation row stride in shared memory
constexpr int GG_W_BYTES = GG_RG * GG_WROW;    // 33280
constexpr int GG_T_BYTES = GG_TOK * GG_TSTRIDE;  // 34816
constexpr int GG_S_BYTES = GG_TOK * GG_KB * 8;   // da and bsum
constexpr int GG_STAGE_BYTES = GG_W_BYTES + GG_T_BYTES + GG_S_BYTES;
constexpr int GG_SMEM = GG_STAGES * GG_STAGE_BYTES + 2 * GG_STAGES * 8;

struct GemmJob {
    const uint8_t *mat0;  // expert 0's matrix; expert e at mat0 + e * mb
    int64_t mb;
    int N, nb;            // rows and 256-blocks per row of one expert matrix
    const int8_t *act;    // activation rows (K = 256 nb bytes each)
    const float *act_da;  // [rows][nb]
    const int *act_bs;
    int by_token;         // activation row of pair p: pair_token[p] (1) or p (0)
    float *Y;             // [P][N]
};

__device__ __forceinline__ uint32_t nib(uint32_t w, int hi) {
    return hi ? ((w >> 4) & 0x0f0f0f0fu) : (w & 0x0f0f0f0fu);
}

__device__ __forceinline__ void mma_s8(int (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                       uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__global__ void __launch_bounds__((GG_CW + 1) * 32, 1) grouped_gemm_kernel(GroupedArgs a, GemmJob j0, GemmJob j1,
                                                                           int njobs) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + GG_STAGES * GG_STAGE_BYTES);
    uint64_t *empty = full + GG_STAGES;
    if (threadIdx.x == 0) {
        for (int s = 0; s < GG_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], GG_CW);
        }
    }
    fence_barrier_init();
    __syncthreads();
    const int n_chunks = __ldcg(a.n_chunks);
    int64_t it = 0;  // stage counter, identical in every warp
    const int64_t tiles0 = (j0.N / 4 + GG_RG - 1) / GG_RG;
    const int64_t tiles1 = njobs > 1 ? (j1.N / 4 + GG_RG - 1) / GG_RG : 0;
    const int64_t items = static_cast<int64_t>(n_chunks) * (tiles0 + tiles1);
    for (int64_t w = blockIdx.x; w < items; w += gridDim.x) {
        const int64_t per_chunk = tiles0 + tiles1;
        const int chunk = static_cast<int>(w / per_chunk);
        int64_t tl = w - chunk * per_chunk;
        const bool second = tl >= tiles0;
        if (second) tl -= tiles0;
        const GemmJob &J = second ? j1 : j0;
        const int e = __ldcg(a.chunk_expert + chunk);
        const int pb = __ldcg(a.chunk_begin + chunk);
        const int m = __ldcg(a.chunk_len + chunk);
        const int n_rg = J.N / 4;
        const int rg0 = static_cast<int>(tl) * GG_RG;
        const int rgs = min(GG_RG, n_rg - rg0);
        const uint8_t *mat = J.mat0 + static_cast<int64_t>(e) * J.mb;
        const int64_t stripe = static_cast<int64_t>(J.nb) * BLOCK_BYTES;
        const int K = J.nb * QK;
        const int n_st = J.nb / GG_KB;
        if (warp == GG_CW) {
            // ---- producer ----
            for (int kc = 0; kc < n_st; ++kc, ++it) {
                const int slot = static_cast<int>(it % GG_STAGES);
                const uint32_t par = static_cast<uint32_t>(((it / GG_STAGES) & 1) ^ 1);
                if (!__all_sync(0xffffffffu, mbar_wait(&empty[slot], par))) {
                    if (lane == 0) report(a.status, TQFX4_ETIMEOUT, K_GGATEUP, static_cast<int>(w));
                    return;
                }
                uint8_t *st = smem + slot * GG_STAGE_BYTES;
                float *sda = reinterpret_cast<float *>(st + GG_W_BYTES + GG_T_BYTES);
                int *sbs = reinterpret_cast<int *>(sda + GG_TOK * GG_KB);
                for (int i = lane; i < m * GG_KB; i += 32) {
                    const int ti = i / GG_KB, bl = i - ti * GG_KB;
                    const int p = pb + ti;
                    const int64_t r = J.by_token ? __ldcg(a.pair_token + p) : p;
                    sda[ti * GG_KB + bl] = __ldcg(J.act_da + r * J.nb + kc * GG_KB + bl);
                    sbs[ti * GG_KB + bl] = __ldcg(J.act_bs + r * J.nb + kc * GG_KB + bl);
                }
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive_expect_tx(&full[slot],
                                          static_cast<uint32_t>(rgs * GG_WROW + m * GG_KB * QK));
                    for (int r = 0; r < rgs; ++r)
                        bulk_g2s(st + r * GG_WROW, mat + (rg0 + r) * stripe + kc * GG_WROW, GG_WROW, &full[slot]);
                    for (int ti = 0; ti < m; ++ti) {
                        const int p = pb + ti;
                        const int64_t row = J.by_token ? __ldcg(a.pair_token + p) : p;
                        bulk_g2s(st + GG_W_BYTES + ti * GG_TSTRIDE, J.act + row * K + kc * GG_KB * QK, GG_KB * QK,
                                 &full[slot]);
                    }
                }
                __syncwarp();
            }
        } else {
            // ---- consumers: warp owns rows 16 warp .. 16 warp + 15 of the tile ----
            const int g = lane >> 2, tig = lane & 3;
            const int row_a = warp * 16 + g, row_b = row_a + 8;  // rows within the tile
            const int rga = row_a >> 2, rgb = row_b >> 2, r4 = g & 3;
            const bool va = rga < rgs, vb = rgb < rgs;
            const int ntiles = (m + 7) >> 3;
            float y[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                for (int q = 0; q < 4; ++q) y[nt][q] = 0.0f;
            for (int kc = 0; kc < n_st; ++kc, ++it) {
                const int slot = static_cast<int>(it % GG_STAGES);
                const uint32_t par = static_cast<uint32_t>((it / GG_STAGES) & 1);
                if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], par))) {
                    if (lane == 0) report(a.status, TQFX4_ETIMEOUT, K_GGATEUP, static_cast<int>(w));
                    return;
                }
                const uint8_t *st = smem + slot * GG_STAGE_BYTES;
                const uint8_t *stt = st + GG_W_BYTES;
                const float *sda = reinterpret_cast<const float *>(st + GG_W_BYTES + GG_T_BYTES);
                const int *sbs = reinterpret_cast<const int *>(sda + GG_TOK * GG_KB);
#pragma unroll 1
                for (int bl = 0; bl < GG_KB; ++bl) {
                    // this thread's 32 code bytes of rows a and b in this block
                    uint32_t wa[8], wb[8];
                    const uint8_t *ba = st + rga * GG_WROW + bl * BLOCK_BYTES + CODE_OFS + ROW_BYTES * r4;
                    const uint8_t *bb = st + rgb * GG_WROW + bl * BLOCK_BYTES + CODE_OFS + ROW_BYTES * r4;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int o = (q < 2 ? 16 * tig + 8 * q : 64 + 16 * tig + 8 * (q - 2));
                        uint2 v = va ? *reinterpret_cast<const uint2 *>(ba + o) : make_uint2(0u, 0u);
                        wa[2 * q] = v.x;
                        wa[2 * q + 1] = v.y;
                        v = vb ? *reinterpret_cast<const uint2 *>(bb + o) : make_uint2(0u, 0u);
                        wb[2 * q] = v.x;
                        wb[2 * q + 1] = v.y;
                    }
                    int acc[8][4];
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                        for (int q = 0; q < 4; ++q) acc[nt][q] = 0;
#pragma unroll
                    for (int s = 0; s < 8; ++s) {
                        const int q = s & 3, hh = s >> 2;
                        const int koff = (q < 2 ? 16 * tig + 8 * q : 64 + 16 * tig + 8 * (q - 2)) + 128 * hh;
                        const uint32_t a0 = nib(wa[2 * q], hh), a2 = nib(wa[2 * q + 1], hh);
                        const uint32_t a1 = nib(wb[2 * q], hh), a3 = nib(wb[2 * q + 1], hh);
#pragma unroll
                        for (int nt = 0; nt < 8; ++nt) {
                            if (nt < ntiles) {
                                const uint2 bw = *reinterpret_cast<const uint2 *>(
                                    stt + (nt * 8 + g) * GG_TSTRIDE + bl * QK + koff);
                                mma_s8(acc[nt], a0, a1, a2, a3, bw.x, bw.y);
                            }
                        }
                    }
                    // fixed float schedule for this block
                    const float dwa = va ? block_scale(st + rga * GG_WROW + bl * BLOCK_BYTES, r4) : 0.0f;
                    const float dwb = vb ? block_scale(st + rgb * GG_WROW + bl * BLOCK_BYTES, r4) : 0.0f;
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt) {
                        if (nt < ntiles) {
                            const int t0 = nt * 8 + 2 * tig, t1 = t0 + 1;
                            const float da0 = sda[t0 * GG_KB + bl], da1 = sda[t1 * GG_KB + bl];
                            const int bs0 = sbs[t0 * GG_KB + bl], bs1 = sbs[t1 * GG_KB + bl];
                            y[nt][0] = __fadd_rn(y[nt][0], __fmul_rn(static_cast<float>(acc[nt][0] - 4 * bs0),
                                                                     __fmul_rn(dwa, da0)));
                            y[nt][1] = __fadd_rn(y[nt][1], __fmul_rn(static_cast<float>(acc[nt][1] - 4 * bs1),
                                                                     __fmul_rn(dwa, da1)));
                            y[nt][2] = __fadd_rn(y[nt][2], __fmul_rn(static_cast<float>(acc[nt][2] - 4 * bs0),
                                                                     __fmul_rn(dwb, da0)));
                            y[nt][3] = __fadd_rn(y[nt][3], __fmul_rn(static_cast<float>(acc[nt][3] - 4 * bs1),
                                                                     __fmul_rn(dwb, da1)));
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[slot]);
            }
            // write the outputs of valid rows and pairs
            const int gra = rg0 * 4 + row_a, grb = rg0 * 4 + row_b;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                const int t0 = nt * 8 + 2 * tig, t1 = t0 + 1;
                if (va && t0 < m) J.Y[static_cast<int64_t>(pb + t0) * J.N + gra] = y[nt][0];
                if (va && t1 < m) J.Y[static_cast<int64_t>(pb + t1) * J.N + gra] = y[nt][1];
                if (vb && t0 < m) J.Y[static_cast<int64_t>(pb + t0) * J.N + grb] = y[nt][2];
                if (vb && t1 < m) J.Y[static_cast<int64_t>(pb + t1) * J.N + grb] = y[nt][3];
            }
        }
    }
}

// ---------------------------------------------------------------- SwiGLU + requant

__global__ void __launch_bounds__(256) swiglu_quant_kernel(GroupedArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t unit = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (unit >= static_cast<int64_t>(a.P) * a.nbi) return;
    const int64_t p = unit / a.nbi;
    const int b = static_cast<int>(unit - p * a.nbi);
    const int64_t o = p * a.I + b * QK + 8 * lane;
    const float4 g0 = __ldcg(reinterpret_cast<const float4 *>(a.g + o));
    const float4 g1 = __ldcg(reinterpret_cast<const float4 *>(a.g + o) + 1);
    const float4 u0 = __ldcg(reinterpret_cast<const float4 *>(a.u + o));
    const float4 u1 = __ldcg(reinterpret_cast<const float4 *>(a.u + o) + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    const float uu[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
    float hv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) hv[i] = tq_swiglu(gg[i], uu[i]);
    uint2 packed;
    float d;
    int sum;
    const bool ok = quant_block_warp(hv, packed, d, sum);
    *reinterpret_cast<uint2 *>(a.qh + o) = packed;
    if (a.keep_h) {
        reinterpret_cast<float4 *>(a.h + o)[0] = make_float4(hv[0], hv[1], hv[2], hv[3]);
        reinterpret_cast<float4 *>(a.h + o)[1] = make_float4(hv[4], hv[5], hv[6], hv[7]);
    }
    if (lane == 0) {
        a.dh[unit] = d;
        a.bh[unit] = sum;
        if (!ok) report(a.status, TQFX4_EDATA, K_GDOWN, static_cast<int>(unit));
    }
}

// ---------------------------------------------------------------- combine

__global__ void __launch_bounds__(256) combine_kernel(GroupedArgs a) {
    const int t = blockIdx.x;
    const int k = a.top_k;
    __shared__ int pos[TQFX4_MAX_TOP_K];
    __shared__ float w[TQFX4_MAX_TOP_K];
    if (threadIdx.x < k) {
        pos[threadIdx.x] = __ldcg(a.pair_of + static_cast<int64_t>(t) * k + threadIdx.x);
        w[threadIdx.x] = __ldcg(a.selw + static_cast<int64_t>(t) * k + threadIdx.x);
    }
    __syncthreads();
    for (int n = threadIdx.x * 4; n < a.H; n += blockDim.x * 4) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int j = 0; j < k; ++j) {
            const float4 v = __ldcg(reinterpret_cast<const float4 *>(a.o + static_cast<int64_t>(pos[j]) * a.H + n));
            acc.x = __fadd_rn(acc.x, __fmul_rn(w[j], v.x));
            acc.y = __fadd_rn(acc.y, __fmul_rn(w[j], v.y));
            acc.z = __fadd_rn(acc.z, __fmul_rn(w[j], v.z));
            acc.w = __fadd_rn(acc.w, __fmul_rn(w[j], v.w));
        }
        *reinterpret_cast<float4 *>(a.OUT + static_cast<int64_t>(t) * a.H + n) = acc;
    }
}

// ---------------------------------------------------------------- host side

bool grouped_args(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t T, void *ws, GroupedArgs &a,
                  MoeLayout &L) {
    a = GroupedArgs{};
    a.E = static_cast<int>(ex->n_experts);
    a.H = static_cast<int>(ex->hidden);
    a.I = static_cast<int>(ex->inter);
    a.top_k = rt->top_k;
    a.T = static_cast<int>(T);
    a.P = a.T * a.top_k;
    a.nbh = a.H / QK;
    a.nbi = a.I / QK;
    a.mb_gu = static_cast<int64_t>(a.I / 4) * a.nbh * BLOCK_BYTES;
    a.mb_d = static_cast<int64_t>(a.H / 4) * a.nbi * BLOCK_BYTES;
    a.gate = static_cast<const uint8_t *>(ex->gate);
    a.up = static_cast<const uint8_t *>(ex->up);
    a.down = static_cast<const uint8_t *>(ex->down);
    a.wr = rt->weight;
    a.bias = rt->bias;
    a.keep_h = 1;
    L = moe_layout(a.E, a.H, a.I, a.top_k, T, true, true);
    uint8_t *base = static_cast<uint8_t *>(ws);
    if (base) {
        a.status = reinterpret_cast<int *>(base);
        a.logits = reinterpret_cast<float *>(base + L.logits);
        a.logits_lo = reinterpret_cast<float *>(base + L.logits_lo);
        a.sel = reinterpret_cast<int *>(base + L.sel);
        a.selw = reinterpret_cast<float *>(base + L.selw);
        a.qx = reinterpret_cast<int8_t *>(base + L.qx);
        a.dx = reinterpret_cast<float *>(base + L.dx);
        a.bx = reinterpret_cast<int *>(base + L.bx);
        a.g = reinterpret_cast<float *>(base + L.g);
        a.u = reinterpret_cast<float *>(base + L.u);
        a.h = reinterpret_cast<float *>(base + L.h);
        a.qh = reinterpret_cast<int8_t *>(base + L.qh);
        a.dh = reinterpret_cast<float *>(base + L.dh);
        a.bh = reinterpret_cast<int *>(base + L.bh);
        a.o = reinterpret_cast<float *>(base + L.o);
        a.counts = reinterpret_cast<int *>(base + L.counts);
        a.offsets = reinterpret_cast<int *>(base + L.offsets);
        a.pair_token = reinterpret_cast<int *>(base + L.pair_token);
        a.pair_slot = reinterpret_cast<int *>(base + L.pair_slot);
        a.pair_of = reinterpret_cast<int *>(base + L.pair_of);
        a.chunk_expert = reinterpret_cast<int *>(base + L.chunk_expert);
        a.chunk_begin = reinterpret_cast<int *>(base + L.chunk_begin);
        a.chunk_len = reinterpret_cast<int *>(base + L.chunk_len);
        a.n_chunks = reinterpret_cast<int *>(base + L.n_chunks);
    }
    return true;
}

int grouped_stage_count() { return 8; }

const char *grouped_stage_name(int s) {
    static const char *names[] = {"router", "topk", "group", "quant_x", "gate_up", "swiglu", "down", "combine"};
    return (s >= 0 && s < 8) ? names[s] : "";
}

cudaError_t launch_moe_grouped(const GroupedArgs &a0, const float *X, float *OUT, int32_t *sel_idx, float *sel_w,
                               cudaStream_t st, void *const *events) {
    GroupedArgs a = a0;
    a.X = X;
    a.OUT = OUT;
    a.sel_out = sel_idx;
    a.selw_out = sel_w;
    static unsigned char set_gg[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(grouped_gemm_kernel), set_gg);
    if (e != cudaSuccess) return e;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (events) cudaStreamIsCapturing(st, &cap);
    auto rec = [&](int i) {
        if (events && events[i])
            cudaEventRecordWithFlags(static_cast<cudaEvent_t>(events[i]), st,
                                     cap == cudaStreamCaptureStatusActive ? cudaEventRecordExternal
                                                                          : cudaEventRecordDefault);
    };
    const int sms = num_sms();
    rec(0);
    router_batch_kernel<<<dim3(a.E, (a.T + RB_TOK - 1) / RB_TOK), 128, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(1);
    topk_batch_kernel<<<a.T, 128, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(2);
    group_kernel<<<1, 1024, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(3);
    if ((e = launch_quantize(a.X, a.T, a.H, a.qx, a.dx, a.bx, a.status, st)) != cudaSuccess) return e;
    rec(4);
    GemmJob jg{a.gate, a.mb_gu, a.I, a.nbh, a.qx, a.dx, a.bx, 1, a.g};
    GemmJob ju{a.up, a.mb_gu, a.I, a.nbh, a.qx, a.dx, a.bx, 1, a.u};
    grouped_gemm_kernel<<<sms, (GG_CW + 1) * 32, GG_SMEM, st>>>(a, jg, ju, 2);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(5);
    const int64_t units = static_cast<int64_t>(a.P) * a.nbi;
    swiglu_quant_kernel<<<static_cast<unsigned>((units * 32 + 255) / 256), 256, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(6);
    GemmJob jd{a.down, a.mb_d, a.H, a.nbi, a.qh, a.dh, a.bh, 0, a.o};
    grouped_gemm_kernel<<<sms, (GG_CW + 1) * 32, GG_SMEM, st>>>(a, jd, jd, 1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(7);
    combine_kernel<<<a.T, 256, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(8);
    return cudaSuccess;
}

}  // namespace tq
