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
//   quant_x  int8 quantization of the T hidden states, then a gather of
//            each pair's token row into pair order
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
// oracle's, bit for bit. A producer warp streams each stage with TMA tensor
// copies (one box of weight blocks, four swizzled boxes of pair-ordered
// activations); four consumer warps each own 8 row groups (32 rows).
#include <cuda.h>
#include <cudaTypedefs.h>

#include "tq_launch.h"
#include "tq_moe_common.cuh"

namespace tq {



// ---------------------------------------------------------------- router

constexpr int RB_TOK = 4;  // tokens per CTA, one per warp (each logit is a latency-bound 16 KB dot product)
// Batches from which the router screens with an fp32 GEMM first.
constexpr int kScreenMinTokens = 256;

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

// Screened router for large batches. An fp32 GEMM gives every logit
// approximately, with a rigorous error bound; only the experts that can
// still reach a token's top k get the compensated (Dot2) logit of
// router_logit_warp, the same value the exact path computes. Every other
// expert keeps its approximation, which lies strictly below k exactly
// evaluated candidates, so the top-k selection and the softmax weights are
// those of the exact path.
//
// Bound: the H products of a logit are summed in kScreenSplit slices, each
// in ascending order with fused multiply-adds by one thread, and the slice
// sums are then added in slice order: every product passes through at most
// H / kScreenSplit + kScreenSplit - 1 <= H roundings, so
// |fl(g) - g| <= gamma_H * sum_h |x_h w_h| <= gamma_H * ||x|| * ||w||
// (Higham, Accuracy and Stability of Numerical Algorithms, section 3.1;
// Cauchy-Schwarz), gamma_H = H u / (1 - H u), u = 2^-24. The bias add and
// the bound arithmetic add a few units of roundoff relative to |logit|; the
// bound below covers them with margin.
constexpr int RG_T = 128, RG_E = 128, RG_BK = 8;

__global__ void __launch_bounds__(256) router_norm_kernel(GroupedArgs a) {
    const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (w >= a.T + a.E) return;
    const float *v = w < a.T ? a.X + static_cast<int64_t>(w) * a.H : a.wr + static_cast<int64_t>(w - a.T) * a.H;
    float s = 0.0f;
    for (int i = lane; i < a.H / 4; i += 32) {
        const float4 q = __ldg(reinterpret_cast<const float4 *>(v) + i);
        s = fmaf(q.x, q.x, fmaf(q.y, q.y, fmaf(q.z, q.z, fmaf(q.w, q.w, s))));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) a.rnorm[w] = sqrtf(s);
}

// part[s][t][e] = fl(sum over slice s of x[t][h] w[e][h]), h ascending, one
// thread per output; tiles of 128 tokens x 128 experts, 8 x 8 outputs per
// thread (rows 4 ty .. + 3 and 64 + 4 ty .. + 3, columns likewise with tx),
// k-steps of 8 staged through shared memory, grid z = slice.
__global__ void __launch_bounds__(256, 2) router_gemm_kernel(GroupedArgs a) {
    __shared__ __align__(16) float xs[2][RG_BK][RG_T + 4];
    __shared__ __align__(16) float wsm[2][RG_BK][RG_E + 4];
    const int e0 = blockIdx.x * RG_E, t0 = blockIdx.y * RG_T;
    const int hs = a.H / kScreenSplit, h0 = blockIdx.z * hs;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;
    // staging: thread i loads 4 consecutive k of row i / 2 of each tile
    const int sr = threadIdx.x >> 1, sc = 4 * (threadIdx.x & 1);
    const float *xrow = t0 + sr < a.T ? a.X + static_cast<int64_t>(t0 + sr) * a.H : nullptr;
    const float *wrow = e0 + sr < a.E ? a.wr + static_cast<int64_t>(e0 + sr) * a.H : nullptr;
    float4 xr, wr;
    auto fetch = [&](int k0) {
        xr = xrow ? __ldg(reinterpret_cast<const float4 *>(xrow + k0 + sc)) : make_float4(0.f, 0.f, 0.f, 0.f);
        wr = wrow ? __ldg(reinterpret_cast<const float4 *>(wrow + k0 + sc)) : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    auto stash = [&](int buf) {
        xs[buf][sc][sr] = xr.x, xs[buf][sc + 1][sr] = xr.y, xs[buf][sc + 2][sr] = xr.z, xs[buf][sc + 3][sr] = xr.w;
        wsm[buf][sc][sr] = wr.x, wsm[buf][sc + 1][sr] = wr.y, wsm[buf][sc + 2][sr] = wr.z, wsm[buf][sc + 3][sr] = wr.w;
    };
    fetch(h0);
    stash(0);
    __syncthreads();
    const int nk = hs / RG_BK;
    for (int it = 0; it < nk; ++it) {
        const int buf = it & 1;
        if (it + 1 < nk) fetch(h0 + (it + 1) * RG_BK);
#pragma unroll
        for (int k = 0; k < RG_BK; ++k) {
            const float4 x0 = *reinterpret_cast<const float4 *>(&xs[buf][k][4 * ty]);
            const float4 x1 = *reinterpret_cast<const float4 *>(&xs[buf][k][64 + 4 * ty]);
            const float4 w0 = *reinterpret_cast<const float4 *>(&wsm[buf][k][4 * tx]);
            const float4 w1 = *reinterpret_cast<const float4 *>(&wsm[buf][k][64 + 4 * tx]);
            const float xx[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
            const float ww[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = __fmaf_rn(xx[i], ww[j], acc[i][j]);
        }
        if (it + 1 < nk) stash(buf ^ 1);
        __syncthreads();
    }
    float *part = a.rpart + static_cast<int64_t>(blockIdx.z) * a.T * a.E;
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int t = t0 + (i < 4 ? 4 * ty + i : 60 + 4 * ty + i);
            const int e = e0 + (j < 4 ? 4 * tx + j : 60 + 4 * tx + j);
            if (t < a.T && e < a.E) part[static_cast<int64_t>(t) * a.E + e] = acc[i][j];
        }
}

// One CTA per token: the slice sums and the bounds, the k-th largest lower
// bound (warp 0), then the list of candidates (the experts whose upper bound
// reaches it), whose compensated logits router_cand_kernel forms.
constexpr int RF_WARPS = 4;

__global__ void __launch_bounds__(RF_WARPS * 32) router_refine_kernel(GroupedArgs a) {
    extern __shared__ float lower[];  // [E]
    __shared__ int n_cand;
    __shared__ float kth_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x;
    float *lg = a.logits + static_cast<int64_t>(t) * a.E;
    float *ll = a.logits_lo + static_cast<int64_t>(t) * a.E;
    const int64_t TE = static_cast<int64_t>(a.T) * a.E;
    // gamma_H ||x|| with 1% margin for gamma's denominator and the norms' own roundoff
    const float cx = 1.01f * static_cast<float>(a.H) * 5.9604645e-8f * __ldcg(a.rnorm + t);
    auto bound = [&](int e, float v) { return cx * __ldcg(a.rnorm + a.T + e) + 4.0e-7f * fabsf(v); };
    if (threadIdx.x == 0) n_cand = 0;
    for (int e = threadIdx.x; e < a.E; e += blockDim.x) {
        const float *p = a.rpart + static_cast<int64_t>(t) * a.E + e;
        float v = __ldcg(p);
#pragma unroll
        for (int s = 1; s < kScreenSplit; ++s) v = __fadd_rn(v, __ldcg(p + s * TE));
        if (a.bias) v = __fadd_rn(v, __ldg(a.bias + e));
        lg[e] = v;
        ll[e] = 0.0f;
        lower[e] = v - bound(e, v);
    }
    __syncthreads();
    if (warp == 0) {
        // k-th largest lower bound: k rounds of a warp maximum, taking one entry per round
        float kth = 0.0f;
        for (int r = 0; r < a.top_k; ++r) {
            float best = -INFINITY;
            int bi = 0x7fffffff;
            for (int e = lane; e < a.E; e += 32) {
                const float v = lower[e];
                if (v > best || (v == best && e < bi)) best = v, bi = e;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ob = __shfl_xor_sync(0xffffffffu, best, o);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                if (ob > best || (ob == best && oi < bi)) best = ob, bi = oi;
            }
            kth = best;
            __syncwarp();
            if (lane == 0) lower[bi] = -INFINITY;
            __syncwarp();
        }
        if (lane == 0) kth_s = kth;
    }
    __syncthreads();
    const float kth = kth_s;
    int *cand = a.rcand + static_cast<int64_t>(t) * a.E;
    for (int e = threadIdx.x; e < a.E; e += blockDim.x) {
        const float v = lg[e];
        if (v + bound(e, v) >= kth) cand[atomicAdd(&n_cand, 1)] = e;
    }
    __syncthreads();
    if (threadIdx.x == 0) a.rcount[t] = n_cand;
}

// The candidates' compensated logits, one warp per (token, candidate): CTA
// (t, y) takes candidates y * RC_WARPS + w, then every RC_Y * RC_WARPS-th,
// so the work is spread over the whole grid whatever each token's count.
constexpr int RC_WARPS = 8, RC_Y = 2;

__global__ void __launch_bounds__(RC_WARPS * 32) router_cand_kernel(GroupedArgs a) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x;
    const int n = __ldcg(a.rcount + t);
    const int *cand = a.rcand + static_cast<int64_t>(t) * a.E;
    const float *x = a.X + static_cast<int64_t>(t) * a.H;
    float *lg = a.logits + static_cast<int64_t>(t) * a.E;
    float *ll = a.logits_lo + static_cast<int64_t>(t) * a.E;
    for (int i = blockIdx.y * RC_WARPS + warp; i < n; i += RC_Y * RC_WARPS) {
        const int c = __ldcg(cand + i);
        float hi, lo;
        router_logit_warp(a.wr + static_cast<int64_t>(c) * a.H, x, a.H, hi, lo);
        if (lane == 0) {
            if (a.bias) ff_add(hi, lo, __ldg(a.bias + c), 0.0f, hi, lo);
            lg[c] = hi;
            ll[c] = lo;
        }
    }
}

// ---------------------------------------------------------------- top-k

// One warp per token: the top-k selection and its softmax weights.
__global__ void __launch_bounds__(128) topk_batch_kernel(GroupedArgs a) {
    __shared__ int sel_s[4][TQFX4_MAX_TOP_K];
    __shared__ float w_s[4][TQFX4_MAX_TOP_K];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x * 4 + warp;
    if (t >= a.T) return;
    const int k = a.top_k;
    const float *lh = a.logits + static_cast<int64_t>(t) * a.E;
    const float *ll = a.logits_lo + static_cast<int64_t>(t) * a.E;
    topk_warp(lh, ll, a.E, k, sel_s[warp]);
    softmax_ff_warp(lh, ll, sel_s[warp], k, w_s[warp]);
    __syncwarp();
    if (lane < k) {
        const int64_t o = static_cast<int64_t>(t) * k + lane;
        a.sel[o] = sel_s[warp][lane];
        a.sel_out[o] = sel_s[warp][lane];
        a.selw[o] = w_s[warp][lane];
        a.selw_out[o] = w_s[warp][lane];
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

// The lanes whose expert equals this lane's (valid lanes only; an invalid
// lane's mask holds the invalid lanes): one ballot per bit of the expert
// index and one for validity. Deterministic, and far cheaper than
// __match_any_sync with many distinct values in the warp.
template <int BITS>
__device__ __forceinline__ unsigned expert_peers_t(int e, bool valid) {
    unsigned m = __ballot_sync(0xffffffffu, valid);
    if (!valid) m = ~m;
#pragma unroll
    for (int b = 0; b < BITS; ++b) {
        const bool set = (e >> b) & 1;
        const unsigned bal = __ballot_sync(0xffffffffu, set);
        m &= set ? bal : ~bal;
    }
    return m;
}
__device__ __forceinline__ unsigned expert_peers(int e, bool valid, int bits) {
    return bits <= 8 ? expert_peers_t<8>(e, valid) : expert_peers_t<10>(e, valid);
}

// Work lists of at least this many pairs leave the scattered (token, slot)
// stores to scatter_pairs_kernel; smaller ones take them in the grouping kernel.
constexpr int kScatterMinPairs = 4096;

__global__ void __launch_bounds__(1024) group_kernel(GroupedArgs a) {
    // counts, offsets, the chunk list and the stable (token, slot) order of
    // the pairs inside each expert's range. W warps take consecutive ranges
    // of the pairs; each counts its hits per expert (the experts' totals are
    // the sums over warps), the counts are turned into per-warp start
    // positions (expert offset + hits of the earlier ranges), and each warp
    // places its pairs in order, ranking equal experts by lane.
    constexpr int HIST = 8192;  // per-warp counts: warps x experts
    __shared__ int hist[HIST];
    __shared__ int warp_tot[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int E = a.E, P = a.P, k = a.top_k, CH = a.chunk;
    const int W = min(32, HIST / E);
    const int ebits = E > 256 ? 10 : 8;  // bits of an expert index (at most TQFX4_MAX_EXPERTS = 1024)
    const int R = (P + W - 1) / W;
    const unsigned lt = (1u << lane) - 1u;
    // the selections are read 8 rounds of 32 at a time (all loads in flight
    // before the first use), then processed round by round in order
    constexpr int GB = 8;
    for (int i = tid; i < W * E; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    if (warp < W) {
        const int p0 = warp * R, p1 = min(P, p0 + R);
        for (int base0 = p0; base0 < p1; base0 += 32 * GB) {
            int ev[GB];
#pragma unroll
            for (int u = 0; u < GB; ++u) {
                const int p = base0 + 32 * u + lane;
                ev[u] = p < p1 ? __ldcg(a.sel + p) : -1 - lane;
            }
#pragma unroll
            for (int u = 0; u < GB; ++u) {
                if (base0 + 32 * u >= p1) break;
                const int e = ev[u];
                const bool valid = base0 + 32 * u + lane < p1;
                const unsigned peers = expert_peers(e, valid, ebits);
                if (valid && lane == __ffs(peers) - 1) hist[warp * E + e] += __popc(peers);
            }
        }
    }
    __syncthreads();
    int c = 0;
    if (tid < E)
        for (int w = 0; w < W; ++w) c += hist[w * E + tid];
    const int incl = block_scan_1024(c, warp_tot);
    if (tid < E) {
        a.counts[tid] = c;
        a.offsets[tid + 1] = incl;
    }
    if (tid == 0) a.offsets[0] = 0;
    // chunk list: ceil(count / CH) chunks per expert
    const int nc = (c + CH - 1) / CH;
    const int cincl = block_scan_1024(nc, warp_tot);
    if (tid < E) {
        const int base = cincl - nc;
        for (int i = 0; i < nc; ++i) {
            a.chunk_expert[base + i] = tid;
            a.chunk_begin[base + i] = incl - c + i * CH;
            a.chunk_len[base + i] = min(CH, c - i * CH);
        }
    }
    if (tid == blockDim.x - 1) *a.n_chunks = cincl;
    // The tensor-core launches' share of the list: the chunks of more than
    // small_max pairs, in chunk order, so that those launches deal their items
    // out over these alone (the small-group pass takes the others). An entry
    // carries the chunk's fields too: one load per item.
    int ntc = 0;
    for (int i = 0; i < nc; ++i) ntc += min(CH, c - i * CH) > a.small_max;
    const int tincl = block_scan_1024(ntc, warp_tot);
    if (tid < E) {
        const int base = cincl - nc;
        int pos = tincl - ntc;
        for (int i = 0; i < nc; ++i) {
            const int len = min(CH, c - i * CH);
            if (len > a.small_max) a.tc_list[pos++] = make_int4(base + i, tid, incl - c + i * CH, len);
        }
    }
    if (tid == blockDim.x - 1) *a.n_tc = tincl;
    // per-warp start positions
    if (tid < E) {
        int run = incl - c;
        for (int w = 0; w < W; ++w) {
            const int h = hist[w * E + tid];
            hist[w * E + tid] = run;
            run += h;
        }
    }
    __syncthreads();
    const bool inline_scatter = P < kScatterMinPairs;
    if (warp < W) {
        const int p0 = warp * R, p1 = min(P, p0 + R);
        for (int base0 = p0; base0 < p1; base0 += 32 * GB) {
            int ev[GB];
#pragma unroll
            for (int u = 0; u < GB; ++u) {
                const int p = base0 + 32 * u + lane;
                ev[u] = p < p1 ? __ldcg(a.sel + p) : -1 - lane;
            }
#pragma unroll
            for (int u = 0; u < GB; ++u) {
                if (base0 + 32 * u >= p1) break;
                const int p = base0 + 32 * u + lane;
                const bool valid = p < p1;
                const int e = ev[u];
                const unsigned peers = expert_peers(e, valid, ebits);
                const int leader = __ffs(peers) - 1;
                int b = 0;
                if (valid && lane == leader) {
                    b = hist[warp * E + e];
                    hist[warp * E + e] = b + __popc(peers);
                }
                b = __shfl_sync(0xffffffffu, b, leader);
                if (valid) {
                    const int pos = b + __popc(peers & lt);
                    a.pair_of[p] = pos;
                    if (inline_scatter) {
                        a.pair_token[pos] = p / k;
                        a.pair_slot[pos] = p - (p / k) * k;
                    }
                }
            }
        }
    }
}

// The inverse of pair_of (each pair's token and slot at its place in expert
// order): scattered stores, spread over many CTAs rather than the grouping
// kernel's one.
__global__ void __launch_bounds__(256) scatter_pairs_kernel(GroupedArgs a) {
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= a.P) return;
    const int pos = __ldcg(a.pair_of + p);
    const int t = p / a.top_k;
    a.pair_token[pos] = t;
    a.pair_slot[pos] = p - t * a.top_k;
}

// ---------------------------------------------------------------- grouped GEMM

// Tile: 128 weight rows (32 row groups) x one chunk of <= 64 pairs. Four
// consumer warps own 8 row groups (32 rows) each and all 64 pairs; a fifth
// warp produces. A stage is two 256-blocks: the 32 row groups' blocks (one
// 2-D tensor copy, 1040 bytes per row group) and the chunk's 512 activation
// bytes per pair (four 2-D tensor copies of one 128-byte line x 64 pairs,
// 128-byte swizzled so that ldmatrix reads are conflict-free).
constexpr int GG_CW = 4;
constexpr int GG_RG = GG_CW * 8;               // 32 row groups per tile
constexpr int GG_KB = 2;                       // 256-blocks per stage
constexpr int GG_STAGES = 3;
constexpr int GG_WROW = GG_KB * BLOCK_BYTES;   // 1040 bytes per row group per stage
constexpr int GG_W_BYTES = 33 * 1024;          // 32 x 1040 = 33280, padded to 1 KB
constexpr int GG_LINE_BYTES = GG_TOK * 128;    // one 128-byte line of 64 pairs
constexpr int GG_T_BYTES = 4 * GG_LINE_BYTES;  // 32768
constexpr int GG_S_BYTES = 2048;               // da and bsum boxes: 64 pairs x 4 blocks each
constexpr int GG_STAGE_BYTES = GG_W_BYTES + GG_T_BYTES + GG_S_BYTES;
constexpr int GG_SMEM = GG_STAGES * GG_STAGE_BYTES + 1024 + 2 * GG_STAGES * 8;

struct GemmJob {
    int64_t mb;  // bytes of one expert matrix
    int N, nb;   // rows and 256-blocks per row of one expert matrix
    float *Y;    // [P][N]
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

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int c0, int c1, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// One stage (GG_KB blocks) of a consumer warp for NT token tiles of 8.
template <int NT>
__device__ __forceinline__ void gg_stage(const uint8_t *st, uint32_t stt, const float *sda, const int *sbs, int cofs,
                                         int rgl, bool vr, int lane, float (&y)[2][8][4]) {
    const int tig = lane & 3;
#pragma unroll 1
    for (int bl = 0; bl < GG_KB; ++bl) {
                    // this thread's code words of the 4 rows of its row group in this block
                    const uint8_t *blk = st + rgl * GG_WROW + bl * BLOCK_BYTES;
                    uint32_t W[4][8];
#pragma unroll
                    for (int r = 0; r < 4; ++r)
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            W[r][j] = *reinterpret_cast<const uint32_t *>(blk + CODE_OFS + ROW_BYTES * r + 4 * tig +
                                                                           16 * j);
                    int acc[2][8][4];
#pragma unroll
                    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                            for (int q = 0; q < 4; ++q) acc[mt][nt][q] = 0;
#pragma unroll
                    for (int s = 0; s < 8; ++s) {
                        const int q = s & 3, hh = s >> 2;
                        const int E0 = bl * QK + 32 * s;  // first element of this k-step in the stage
                        const int L = E0 >> 7, c0 = (E0 & 127) >> 4;
                        uint32_t bf[8][2];
#pragma unroll
                        for (int np = 0; np < 4; ++np) {
                            if (2 * np < NT) {
                                const int mi = lane >> 3;  // matrix supplied by this lane's address
                                const int t = (2 * np + (mi >> 1)) * 8 + (lane & 7);
                                const int c = c0 + (mi & 1);
                                const uint32_t addr = stt + L * GG_LINE_BYTES + t * 128 + ((c ^ (t & 7)) << 4);
                                ldmatrix_x4(addr, bf[2 * np][0], bf[2 * np][1], bf[2 * np + 1][0],
                                            bf[2 * np + 1][1]);
                            }
                        }
#pragma unroll
                        for (int mt = 0; mt < 2; ++mt) {
                            const uint32_t a0 = nib(W[2 * mt][2 * q], hh), a2 = nib(W[2 * mt][2 * q + 1], hh);
                            const uint32_t a1 = nib(W[2 * mt + 1][2 * q], hh), a3 = nib(W[2 * mt + 1][2 * q + 1], hh);
#pragma unroll
                            for (int nt = 0; nt < 8; ++nt)
                                if (nt < NT) mma_s8(acc[mt][nt], a0, a1, a2, a3, bf[nt][0], bf[nt][1]);
                        }
                    }
                    // fixed float schedule for this block
                    float dw[4];
#pragma unroll
                    for (int r = 0; r < 4; ++r) dw[r] = vr ? block_scale(blk, r) : 0.0f;
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt) {
                        if (nt < NT) {
                            const int t0 = nt * 8 + 2 * tig, t1 = t0 + 1;
                            const float da0 = sda[t0 * 4 + cofs + bl], da1 = sda[t1 * 4 + cofs + bl];
                            const int bs0 = sbs[t0 * 4 + cofs + bl], bs1 = sbs[t1 * 4 + cofs + bl];
#pragma unroll
                            for (int mt = 0; mt < 2; ++mt) {
                                const float dlo = dw[2 * mt], dhi = dw[2 * mt + 1];
                                y[mt][nt][0] = __fadd_rn(y[mt][nt][0], __fmul_rn(static_cast<float>(acc[mt][nt][0] - 4 * bs0),
                                                                                 __fmul_rn(dlo, da0)));
                                y[mt][nt][1] = __fadd_rn(y[mt][nt][1], __fmul_rn(static_cast<float>(acc[mt][nt][1] - 4 * bs1),
                                                                                 __fmul_rn(dlo, da1)));
                                y[mt][nt][2] = __fadd_rn(y[mt][nt][2], __fmul_rn(static_cast<float>(acc[mt][nt][2] - 4 * bs0),
                                                                                 __fmul_rn(dhi, da0)));
                                y[mt][nt][3] = __fadd_rn(y[mt][nt][3], __fmul_rn(static_cast<float>(acc[mt][nt][3] - 4 * bs1),
                                                                                 __fmul_rn(dhi, da1)));
                            }
                        }
                    }
                }
}

__global__ void __launch_bounds__((GG_CW + 1) * 32, 1)
    grouped_gemm_kernel(GroupedArgs a, GemmJob j0, GemmJob j1, int njobs, const __grid_constant__ CUtensorMap w0,
                        const __grid_constant__ CUtensorMap w1, const __grid_constant__ CUtensorMap xmap,
                        const __grid_constant__ CUtensorMap damap, const __grid_constant__ CUtensorMap bsmap) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
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
    const int64_t per_chunk = tiles0 + tiles1;
    const int64_t items = static_cast<int64_t>(n_chunks) * per_chunk;
    // the chunk descriptor of the next item is loaded one item ahead
    auto chunk_of = [&](int64_t w) { return static_cast<int>(w / per_chunk); };
    int ce = 0, cb = 0, cl = 0;
    if (blockIdx.x < items) {
        const int c = chunk_of(blockIdx.x);
        ce = __ldcg(a.chunk_expert + c);
        cb = __ldcg(a.chunk_begin + c);
        cl = __ldcg(a.chunk_len + c);
    }
    for (int64_t w = blockIdx.x; w < items; w += gridDim.x) {
        const int chunk = chunk_of(w);
        int64_t tl = w - chunk * per_chunk;
        const bool second = tl >= tiles0;
        if (second) tl -= tiles0;
        const GemmJob &J = second ? j1 : j0;
        const CUtensorMap *wmap = second ? &w1 : &w0;
        const int e = ce, pb = cb, m = cl;
        if (w + gridDim.x < items) {
            const int c = chunk_of(w + gridDim.x);
            ce = __ldcg(a.chunk_expert + c);
            cb = __ldcg(a.chunk_begin + c);
            cl = __ldcg(a.chunk_len + c);
        }
        const int n_rg = J.N / 4;
        const int rg0 = static_cast<int>(tl) * GG_RG;
        const int n_st = J.nb / GG_KB;
        if (warp == GG_CW) {
            // ---- producer ----
            for (int kc = 0; kc < n_st; ++kc, ++it) {
                const int slot = static_cast<int>(it % GG_STAGES);
                const uint32_t par = static_cast<uint32_t>(((it / GG_STAGES) & 1) ^ 1);
#ifdef TQ_INSTRUMENT
                const long long tw0 = clock64();
#endif
                if (!__all_sync(0xffffffffu, mbar_wait(&empty[slot], par))) {
                    if (lane == 0) report(a.status, TQFX4_ETIMEOUT, K_GGATEUP, static_cast<int>(w));
                    return;
                }
                TQ_ADD(3, 0, clock64() - tw0);
                uint8_t *st = smem + slot * GG_STAGE_BYTES;
#ifdef TQ_INSTRUMENT
                const long long ti0 = clock64();
#endif
                if (lane == 0) {
                    mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(GG_RG * GG_WROW + GG_T_BYTES + GG_S_BYTES));
                    // weights: rows e * n_rg + rg0 .. + 31 of the stacked matrix, bytes kc * 1040 ..
                    tma_load_2d(st, wmap, kc * (GG_WROW / 8), e * n_rg + rg0, &full[slot]);
                    // activations: four 128-byte lines of 64 pair rows starting at pb
                    for (int L = 0; L < 4; ++L)
                        tma_load_2d(st + GG_W_BYTES + L * GG_LINE_BYTES, &xmap, (kc * GG_KB * QK + L * 128) / 8, pb,
                                    &full[slot]);
                    // scales and block sums of blocks 4 (kc / 2) .. + 3 of the 64 pairs
                    tma_load_2d(st + GG_W_BYTES + GG_T_BYTES, &damap, 4 * (kc >> 1), pb, &full[slot]);
                    tma_load_2d(st + GG_W_BYTES + GG_T_BYTES + 1024, &bsmap, 4 * (kc >> 1), pb, &full[slot]);
                }
                TQ_ADD(3, 1, clock64() - ti0);
                TQ_ADD(3, 2, 1);
                __syncwarp();
            }
        } else {
            // ---- consumers: warp owns row groups rg0 + 8 warp + (lane >> 2) ----
            const int g = lane >> 2, tig = lane & 3;
            const int rgl = warp * 8 + g;  // row group within the tile
            const bool vr = rg0 + rgl < n_rg;
            const int ntiles = (m + 7) >> 3;
            float y[2][8][4];
#pragma unroll
            for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                    for (int q = 0; q < 4; ++q) y[mt][nt][q] = 0.0f;
            for (int kc = 0; kc < n_st; ++kc, ++it) {
                const int slot = static_cast<int>(it % GG_STAGES);
                const uint32_t par = static_cast<uint32_t>((it / GG_STAGES) & 1);
#ifdef TQ_INSTRUMENT
                const long long tf0 = clock64();
#endif
                if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], par))) {
                    if (lane == 0) report(a.status, TQFX4_ETIMEOUT, K_GGATEUP, static_cast<int>(w));
                    return;
                }
#ifdef TQ_INSTRUMENT
                const long long tc0 = clock64();
                if (warp == 0) TQ_ADD(3, 3, tc0 - tf0);
#endif
                const uint8_t *st = smem + slot * GG_STAGE_BYTES;
                const uint32_t stt = smem_u32(st + GG_W_BYTES);
                const float *sda = reinterpret_cast<const float *>(st + GG_W_BYTES + GG_T_BYTES);
                const int *sbs = reinterpret_cast<const int *>(st + GG_W_BYTES + GG_T_BYTES + 1024);
                const int cofs = (kc & 1) * GG_KB;  // this stage's blocks inside the 4-block scale box
                switch (ntiles) {
                    case 1: gg_stage<1>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 2: gg_stage<2>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 3: gg_stage<3>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 4: gg_stage<4>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 5: gg_stage<5>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 6: gg_stage<6>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    case 7: gg_stage<7>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                    default: gg_stage<8>(st, stt, sda, sbs, cofs, rgl, vr, lane, y); break;
                }
                __syncwarp();
#ifdef TQ_INSTRUMENT
                if (warp == 0) TQ_ADD(3, 4, clock64() - tc0);
#endif
                if (lane == 0) mbar_arrive(&empty[slot]);
            }
            if (vr) {
                const int64_t row0 = static_cast<int64_t>(rg0 + rgl) * 4;
#pragma unroll
                for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt) {
                        const int t0 = nt * 8 + 2 * tig, t1 = t0 + 1;
                        if (t0 < m) {
                            J.Y[static_cast<int64_t>(pb + t0) * J.N + row0 + 2 * mt] = y[mt][nt][0];
                            J.Y[static_cast<int64_t>(pb + t0) * J.N + row0 + 2 * mt + 1] = y[mt][nt][2];
                        }
                        if (t1 < m) {
                            J.Y[static_cast<int64_t>(pb + t1) * J.N + row0 + 2 * mt] = y[mt][nt][1];
                            J.Y[static_cast<int64_t>(pb + t1) * J.N + row0 + 2 * mt + 1] = y[mt][nt][3];
                        }
                    }
            }
        }
    }
}

// Gather the quantized hidden state of each pair's token into pair order.
__global__ void __launch_bounds__(256) gather_rows_kernel(GroupedArgs a) {
    const int64_t pos = blockIdx.x;
    int64_t t = __ldcg(a.pair_token + pos);
    if (!TQ_DEBUG_CHECK(t >= 0 && t < a.T, a.status, K_GROUP, static_cast<int>(pos))) t = 0;
    const uint4 *src = reinterpret_cast<const uint4 *>(a.qx + t * a.H);
    uint4 *dst = reinterpret_cast<uint4 *>(a.xg + pos * a.H);
    for (int i = threadIdx.x; i < a.H / 16; i += blockDim.x) dst[i] = __ldcg(src + i);
    for (int b = threadIdx.x; b < a.nbhp; b += blockDim.x) {
        a.dxg[pos * a.nbhp + b] = b < a.nbh ? __ldcg(a.dx + t * a.nbh + b) : 0.0f;
        a.bxg[pos * a.nbhp + b] = b < a.nbh ? __ldcg(a.bx + t * a.nbh + b) : 0;
    }
}

// Tensor-core path: per chunk, its pairs' quantized hidden states as the two
// e4m3 planes, and per block the pairs' scales da and -4 bsum (as float) in
// the chunk-aligned layout the contraction stages with one bulk copy.
// The e4m3 planes of the tokens' quantized x, once per token (in token order;
// the gather below copies them into pair order): one thread per 8 bytes.
__global__ void __launch_bounds__(256) planes_tok_kernel(GroupedArgs a) {
    const int64_t n8 = static_cast<int64_t>(a.T) * a.H / 8;
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n8) return;
    uint2 hi, lo;
    q_planes8(__ldcg(reinterpret_cast<const uint2 *>(a.qx) + i), hi, lo);
    reinterpret_cast<uint2 *>(a.xqt)[i] = hi;
    reinterpret_cast<uint2 *>(a.xqt + static_cast<int64_t>(a.T) * a.H)[i] = lo;
}

// CTA (c, y) handles pair columns 16 y .. 16 y + 15 of chunk c (chunks hold
// 1..TC_CHUNK pairs, so a chunk is spread over several CTAs): copies the pairs'
// plane rows from token order and writes the chunk's scale columns.
constexpr int GT_PAIRS = 16;
static_assert(TC_CHUNK % GT_PAIRS == 0, "whole CTAs per chunk");

__global__ void __launch_bounds__(256) gather_tc_kernel(GroupedArgs a) {
    const int c = blockIdx.x;
    if (c >= __ldcg(a.n_chunks)) return;
    const int pb = __ldcg(a.chunk_begin + c), m = __ldcg(a.chunk_len + c);
    const int n0 = blockIdx.y * GT_PAIRS;
    const int64_t plane = static_cast<int64_t>(a.P) * a.H, tplane = static_cast<int64_t>(a.T) * a.H;
    const int lane = threadIdx.x & 31, n16 = a.H / 16;
    for (int n = n0 + (threadIdx.x >> 5); n < m && n < n0 + GT_PAIRS; n += blockDim.x >> 5) {
        const int64_t pos = pb + n;
        int64_t t = __ldcg(a.pair_token + pos);
        if (!TQ_DEBUG_CHECK(t >= 0 && t < a.T, a.status, K_GROUP, static_cast<int>(pos))) t = 0;
#pragma unroll
        for (int pl = 0; pl < 2; ++pl) {
            const uint4 *src = reinterpret_cast<const uint4 *>(a.xqt + pl * tplane + t * a.H);
            uint4 *dst = reinterpret_cast<uint4 *>(a.xq + pl * plane + pos * a.H);
            for (int i = lane; i < n16; i += 32) dst[i] = __ldcg(src + i);
        }
        if (lane == 0) a.pair_hs[pos] = c * a.nbi * 2 * TC_CHUNK + n;
    }
    for (int i = threadIdx.x; i < a.nbh * GT_PAIRS; i += blockDim.x) {
        const int b = i / GT_PAIRS, n = n0 + (i - b * GT_PAIRS);
        float d = 0.0f, nb4 = 0.0f;
        if (n < m) {
            const int64_t t = __ldcg(a.pair_token + pb + n);
            d = __ldcg(a.dx + t * a.nbh + b);
            nb4 = static_cast<float>(-4 * __ldcg(a.bx + t * a.nbh + b));
        }
        float *o = a.xs + (static_cast<int64_t>(c) * a.nbh + b) * 2 * TC_CHUNK;
        o[n] = d;
        o[TC_CHUNK + n] = nb4;
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
    // the pair's scale slot, loaded with g and u (used at the end)
    const int hsb = (a.tc && lane == 0) ? __ldcg(a.pair_hs + p) : 0;
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
    if (a.tc) {
        uint2 hi, lo;
        q_planes8(packed, hi, lo);
        *reinterpret_cast<uint2 *>(a.hq + o) = hi;
        *reinterpret_cast<uint2 *>(a.hq + static_cast<int64_t>(a.P) * a.I + o) = lo;
        if (lane == 0) {
            float *hs = a.hs + hsb + static_cast<int64_t>(b) * 2 * TC_CHUNK;
            hs[0] = d;
            hs[TC_CHUNK] = static_cast<float>(-4 * sum);
        }
    }
    if (a.keep_h) {
        reinterpret_cast<float4 *>(a.h + o)[0] = make_float4(hv[0], hv[1], hv[2], hv[3]);
        reinterpret_cast<float4 *>(a.h + o)[1] = make_float4(hv[4], hv[5], hv[6], hv[7]);
    }
    if (lane == 0) {
        a.dh[unit] = d;
        a.bh[unit] = sum;
        a.dhp[p * a.nbip + b] = d;
        a.bhp[p * a.nbip + b] = sum;
        if (b == a.nbi - 1)
            for (int i = a.nbi; i < a.nbip; ++i) {
                a.dhp[p * a.nbip + i] = 0.0f;
                a.bhp[p * a.nbip + i] = 0;
            }
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
        int p = __ldcg(a.pair_of + static_cast<int64_t>(t) * k + threadIdx.x);
        if (!TQ_DEBUG_CHECK(p >= 0 && p < a.P, a.status, K_COMBINE, t)) p = 0;
        pos[threadIdx.x] = p;
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

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t encoder() {
    if (g_encode) return cudaSuccess;
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// The stacked matrices of one projection as a 2-D tensor of 8-byte elements:
// one row per row group (E * n_rg rows, stride nb * 520 bytes), boxes of
// GG_KB blocks (130 elements) x GG_RG row groups.
cudaError_t weight_map(CUtensorMap *m, const void *base, int64_t E, int64_t n_rg, int nb) {
    cudaError_t e = encoder();
    if (e != cudaSuccess) return e;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(nb) * BLOCK_BYTES / 8, static_cast<cuuint64_t>(E * n_rg)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(nb) * BLOCK_BYTES};
    const cuuint32_t box[2] = {GG_WROW / 8, GG_RG};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_UINT64, 2, const_cast<void *>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Activation rows [rows][K] int8 as 8-byte elements; boxes of one 128-byte
// line x GG_TOK rows, 128-byte swizzled.
cudaError_t act_map(CUtensorMap *m, const void *base, int64_t rows, int64_t K) {
    cudaError_t e = encoder();
    if (e != cudaSuccess) return e;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K / 8), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K)};
    const cuuint32_t box[2] = {16, GG_TOK};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_UINT64, 2, const_cast<void *>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Per-pair block scales (fp32) or block sums (int32) [rows][nbp] with nbp a
// multiple of 4; boxes of 4 blocks x GG_TOK rows.
cudaError_t scale_map(CUtensorMap *m, const void *base, int64_t rows, int nbp, bool is_float) {
    cudaError_t e = encoder();
    if (e != cudaSuccess) return e;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(nbp), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(nbp) * 4};
    const cuuint32_t box[2] = {4, GG_TOK};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(m, is_float ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_INT32, 2,
                          const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

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
    a.nbhp = (a.nbh + 3) / 4 * 4;
    a.nbip = (a.nbi + 3) / 4 * 4;
    L = moe_layout(a.E, a.H, a.I, a.top_k, T, true, true);
    a.max_chunks = static_cast<int>(L.max_chunks);
    a.chunk = GG_TOK;
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
        a.xg = reinterpret_cast<int8_t *>(base + L.xg);
        a.dxg = reinterpret_cast<float *>(base + L.dxg);
        a.bxg = reinterpret_cast<int *>(base + L.bxg);
        a.dhp = reinterpret_cast<float *>(base + L.dhp);
        a.bhp = reinterpret_cast<int *>(base + L.bhp);
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
        a.tc_list = reinterpret_cast<int4 *>(base + L.tc_list);
        a.n_tc = reinterpret_cast<int *>(base + L.n_tc);
        a.xq = base + L.xq;
        a.xqt = base + L.xqt;
        a.hq = base + L.hq;
        a.pair_hs = reinterpret_cast<int *>(base + L.pair_hs);
        a.xs = reinterpret_cast<float *>(base + L.xs);
        a.hs = reinterpret_cast<float *>(base + L.hs);
        a.rnorm = reinterpret_cast<float *>(base + L.rnorm);
        a.rpart = reinterpret_cast<float *>(base + L.rpart);
        a.rcand = reinterpret_cast<int *>(base + L.rcand);
        a.rcount = reinterpret_cast<int *>(base + L.rcount);
    }
    return true;
}

int grouped_stage_count() { return 8; }

const char *grouped_stage_name(int s) {
    static const char *names[] = {"router", "topk", "group", "quant_gather", "gate_up", "swiglu", "down",
                                  "combine"};
    return (s >= 0 && s < 8) ? names[s] : "";
}

cudaError_t launch_moe_grouped(const GroupedArgs &a0, const float *X, float *OUT, int32_t *sel_idx, float *sel_w,
                               cudaStream_t st, void *const *events) {
    GroupedArgs a = a0;
    a.chunk = a.tc ? TC_CHUNK : GG_TOK;
    a.small_max = a.tc ? small_groups_max(a) : 0;
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
    if (a.T >= kScreenMinTokens) {
        router_norm_kernel<<<(a.T + a.E + 7) / 8, 256, 0, st>>>(a);
        router_gemm_kernel<<<dim3((a.E + RG_E - 1) / RG_E, (a.T + RG_T - 1) / RG_T, kScreenSplit), 256, 0, st>>>(a);
        router_refine_kernel<<<a.T, RF_WARPS * 32, a.E * sizeof(float), st>>>(a);
        router_cand_kernel<<<dim3(a.T, RC_Y), RC_WARPS * 32, 0, st>>>(a);
    } else {
        router_batch_kernel<<<dim3(a.E, (a.T + RB_TOK - 1) / RB_TOK), 128, 0, st>>>(a);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(1);
    topk_batch_kernel<<<(a.T + 3) / 4, 128, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(2);
    group_kernel<<<1, 1024, 0, st>>>(a);
    if (a.P >= kScatterMinPairs) scatter_pairs_kernel<<<(a.P + 255) / 256, 256, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(3);
    if ((e = launch_quantize(a.X, a.T, a.H, a.qx, a.dx, a.bx, a.status, st)) != cudaSuccess) return e;
    if (a.tc) {
        const int64_t n8 = static_cast<int64_t>(a.T) * a.H / 8;
        planes_tok_kernel<<<static_cast<unsigned>((n8 + 255) / 256), 256, 0, st>>>(a);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (a.tc)
        gather_tc_kernel<<<dim3(static_cast<unsigned>(a.max_chunks), TC_CHUNK / GT_PAIRS), 256, 0, st>>>(a);
    else
        gather_rows_kernel<<<a.P, 256, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(4);
    const int64_t units = static_cast<int64_t>(a.P) * a.nbi;
    if (a.tc) {
        if ((e = launch_tc_gemm(a, false, st)) != cudaSuccess) return e;
        if (a.small_max && (e = launch_small_groups(a, false, st)) != cudaSuccess) return e;
        rec(5);
        swiglu_quant_kernel<<<static_cast<unsigned>((units * 32 + 255) / 256), 256, 0, st>>>(a);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        rec(6);
        if ((e = launch_tc_gemm(a, true, st)) != cudaSuccess) return e;
        if (a.small_max && (e = launch_small_groups(a, true, st)) != cudaSuccess) return e;
    } else {
        CUtensorMap mg, mu, md, mx, mh, sdx, sbx, sdh, sbh;
        if ((e = scale_map(&sdx, a.dxg, a.P, a.nbhp, true)) != cudaSuccess) return e;
        if ((e = scale_map(&sbx, a.bxg, a.P, a.nbhp, false)) != cudaSuccess) return e;
        if ((e = scale_map(&sdh, a.dhp, a.P, a.nbip, true)) != cudaSuccess) return e;
        if ((e = scale_map(&sbh, a.bhp, a.P, a.nbip, false)) != cudaSuccess) return e;
        if ((e = weight_map(&mg, a.gate, a.E, a.I / 4, a.nbh)) != cudaSuccess) return e;
        if ((e = weight_map(&mu, a.up, a.E, a.I / 4, a.nbh)) != cudaSuccess) return e;
        if ((e = weight_map(&md, a.down, a.E, a.H / 4, a.nbi)) != cudaSuccess) return e;
        if ((e = act_map(&mx, a.xg, a.P, a.H)) != cudaSuccess) return e;
        if ((e = act_map(&mh, a.qh, a.P, a.I)) != cudaSuccess) return e;
        GemmJob jg{a.mb_gu, a.I, a.nbh, a.g};
        GemmJob ju{a.mb_gu, a.I, a.nbh, a.u};
        grouped_gemm_kernel<<<sms, (GG_CW + 1) * 32, GG_SMEM, st>>>(a, jg, ju, 2, mg, mu, mx, sdx, sbx);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        rec(5);
        swiglu_quant_kernel<<<static_cast<unsigned>((units * 32 + 255) / 256), 256, 0, st>>>(a);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        rec(6);
        GemmJob jd{a.mb_d, a.H, a.nbi, a.o};
        grouped_gemm_kernel<<<sms, (GG_CW + 1) * 32, GG_SMEM, st>>>(a, jd, jd, 1, md, md, mh, sdh, sbh);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    rec(7);
    combine_kernel<<<a.T, 256, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(8);
    return cudaSuccess;
}

}  // namespace tq
