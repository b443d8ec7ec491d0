// Pieces shared by the MoE decode and grouped kernels: workspace layout,
// top-k selection, and two-range bulk staging.
#pragma once

#include "tq_common.cuh"

namespace tq {

// ---- workspace layout (byte offsets from the workspace base) -------------------

struct MoeLayout {
    size_t ctr;      // int32 counters, zeroed by the first kernel of every call
    size_t n_ctr;
    size_t logits;   // fp32 [T][E]
    size_t logits_lo; // fp32 [T][E]: logit = logits + logits_lo (double-binary32)
    size_t sel;      // int32 [T][top_k]
    size_t selw;     // fp32 [T][top_k]
    size_t qx, dx, bx;
    size_t g, u, h;  // fp32 [P][I]
    size_t qh, dh, bh;
    size_t o;        // fp32 [P][H]
    size_t counts, offsets, pair_token, pair_slot, pair_of;
    size_t xg;  // int8 [P][H] (grouped only)
    size_t dxg, bxg, dhp, bhp;  // [P][round4(nb)] (grouped only)
    size_t chunk_expert, chunk_begin, chunk_len, n_chunks;  // grouped GEMM work list
    size_t tc_list, n_tc;  // int4 [max_chunks] (chunk, expert, begin, pairs) of the tensor-core launches' chunks, and their count (grouped only)
    size_t xq, hq;    // e4m3 activation planes [2][P][H], [2][P][I] for the tensor-core contraction (grouped only)
    size_t xqt;       // the same planes of x in token order [2][T][H] (grouped only)
    size_t pair_hs, xs, hs;  // tensor-core work list helpers (grouped only)
    size_t rnorm;     // fp32 [T + E]: Euclidean norms of the hidden states and router rows (grouped only)
    size_t rpart;     // fp32 [kScreenSplit][T][E]: partial router logits of the screening GEMM (grouped only)
    size_t rcand, rcount;  // int [T][E], [T]: each token's screened-in experts and their count (grouped only)
    int64_t max_chunks;
    size_t total;
};

// Tokens (pairs) per chunk of the grouped GEMM.
constexpr int GG_TOK = 64;
// Pairs from which the automatic path choice takes the tensor-core
// contraction: it measured faster than the integer-MMA one at every batch
// from 4 tokens (top-8) up, so the automatic choice always takes it.
constexpr int64_t kTcMinPairs = 1;
// Slices of the hidden dimension the router's screening GEMM sums separately.
constexpr int kScreenSplit = 8;
// Pairs per chunk on the tensor-core path: both activation planes of a
// chunk side by side make the MMA's N = 2 x 96 = 192.
constexpr int TC_CHUNK = 96;

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

inline MoeLayout moe_layout(int64_t E, int64_t H, int64_t I, int64_t top_k, int64_t T, bool grouped,
                            bool keep_gu) {
    MoeLayout L{};
    const int64_t P = T * top_k;
    const int64_t nbh = H / QK, nbi = I / QK;
    size_t off = TQFX4_STATUS_BYTES;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align256(off + bytes);
        return at;
    };
    L.n_ctr = static_cast<size_t>(P * nbi + (H / 4) * (grouped ? T : 1) + E + 1024);
    L.ctr = take(4 * L.n_ctr);
    L.logits = take(4 * static_cast<size_t>(T * E));
    L.logits_lo = take(4 * static_cast<size_t>(T * E));
    L.sel = take(4 * static_cast<size_t>(P));
    L.selw = take(4 * static_cast<size_t>(P));
    L.qx = take(static_cast<size_t>(T * H));
    L.dx = take(4 * static_cast<size_t>(T * nbh));
    L.bx = take(4 * static_cast<size_t>(T * nbh));
    if (keep_gu) {
        L.g = take(4 * static_cast<size_t>(P * I));
        L.u = take(4 * static_cast<size_t>(P * I));
    } else {
        L.g = L.u = SIZE_MAX;
    }
    L.h = take(4 * static_cast<size_t>(P * I));
    L.qh = take(static_cast<size_t>(P * I));
    L.dh = take(4 * static_cast<size_t>(P * nbi));
    L.bh = take(4 * static_cast<size_t>(P * nbi));
    L.o = take(4 * static_cast<size_t>(P * H));
    if (grouped) {
        L.counts = take(4 * static_cast<size_t>(E));
        L.offsets = take(4 * static_cast<size_t>(E + 1));
        L.pair_token = take(4 * static_cast<size_t>(P));
        L.pair_slot = take(4 * static_cast<size_t>(P));
        L.pair_of = take(4 * static_cast<size_t>(P));
        L.xg = take(static_cast<size_t>(P * H));
        const int64_t nbhp = (nbh + 3) / 4 * 4, nbip = (nbi + 3) / 4 * 4;
        L.dxg = take(4 * static_cast<size_t>(P * nbhp));
        L.bxg = take(4 * static_cast<size_t>(P * nbhp));
        L.dhp = take(4 * static_cast<size_t>(P * nbip));
        L.bhp = take(4 * static_cast<size_t>(P * nbip));
        // every chunk holds at least one pair, and an expert adds at most one partial chunk
        L.max_chunks = (P < P / GG_TOK + E ? P : P / GG_TOK + E) + 1;
        L.chunk_expert = take(4 * static_cast<size_t>(L.max_chunks));
        L.chunk_begin = take(4 * static_cast<size_t>(L.max_chunks));
        L.chunk_len = take(4 * static_cast<size_t>(L.max_chunks));
        L.n_chunks = take(4);
        L.tc_list = take(16 * static_cast<size_t>(L.max_chunks));
        L.n_tc = take(4);
        L.xq = take(2 * static_cast<size_t>(P * H));
        L.hq = take(2 * static_cast<size_t>(P * I));
        L.xqt = take(2 * static_cast<size_t>(T * H));
        L.pair_hs = take(4 * static_cast<size_t>(P));
        L.rnorm = take(4 * static_cast<size_t>(T + E));
        L.rpart = take(4 * static_cast<size_t>(kScreenSplit) * T * E);
        L.rcand = take(4 * static_cast<size_t>(T) * E);
        L.rcount = take(4 * static_cast<size_t>(T));
        L.xs = take(static_cast<size_t>(L.max_chunks) * nbh * 2 * TC_CHUNK * 4);
        L.hs = take(static_cast<size_t>(L.max_chunks) * nbi * 2 * TC_CHUNK * 4);
    } else {
        L.counts = L.offsets = L.pair_token = L.pair_slot = L.pair_of = L.xg = SIZE_MAX;
        L.dxg = L.bxg = L.dhp = L.bhp = SIZE_MAX;
        L.chunk_expert = L.chunk_begin = L.chunk_len = L.n_chunks = SIZE_MAX;
        L.tc_list = L.n_tc = SIZE_MAX;
        L.xq = L.hq = L.xqt = L.pair_hs = L.xs = L.hs = L.rnorm = L.rpart = SIZE_MAX;
        L.rcand = L.rcount = SIZE_MAX;
        L.max_chunks = 0;
    }
    L.total = off;
    return L;
}

// ---- kernel arguments of the decode path ----

struct MoeArgs {
    const uint8_t *gate, *up, *down;
    int64_t mb_gu, mb_d;  // bytes of one expert's gate (= up) and down matrix
    const float *wr, *bias;
    const float *x;
    float *out;
    int32_t *sel_out;
    float *selw_out;
    int E, H, I, top_k, nbh, nbi;
    // workspace views
    int *status, *ctr;
    int n_ctr;
    float *logits, *logits_lo;
    int *sel;
    float *selw;
    int8_t *qx;
    float *dx;
    int *bx;
    float *g, *u, *h;
    int8_t *qh;
    float *dh;
    int *bh;
    float *o;
    // gate/up geometry: top_k x parts_gu CTAs; static_gu units per CTA before the shared counter
    int rpu_gu, slot_gu, stages_gu, warps_gu, parts_gu, static_gu;
    // down geometry: top_k x parts_d CTAs, each a range of row groups
    int rpu_d, slot_d, stages_d, warps_d, parts_d;
    // the selected experts' blocks given by the caller (device array of
    // 3 x top_k pointers: gate, then up, then down, in rank order), or null
    // for the stacked layout (base + expert * matrix bytes)
    const uint8_t *const *ptrs;
    int route_only;  // the router also forms the routing weights, and no expert kernels follow
    // one expert's FFN without a router (tqfx4_expert_ffn): the expert is
    // expert 0 of the stacked matrices, its weight 1; gate/up quantizes x
    // itself and down resets gate/up's unit counter for the next call
    int single;
};

// Arguments of the grouped (T-token) kernels.
struct GroupedArgs {
    int E, H, I, top_k, T, P, nbh, nbi;
    const uint8_t *gate, *up, *down;
    int64_t mb_gu, mb_d;
    const float *wr, *bias;
    const float *X;
    float *OUT;
    int32_t *sel_out;
    float *selw_out;
    int *status;
    float *logits, *logits_lo;
    int *sel;
    float *selw;
    int8_t *qx;
    float *dx;
    int *bx;
    int8_t *xg;  // [P][H] quantized hidden state of each pair, in pair order
    float *dxg, *dhp;  // [P][nbp] scales in pair order, rows padded to a multiple of 4 blocks
    int *bxg, *bhp;
    int nbhp, nbip;
    float *g, *u, *h;
    int8_t *qh;
    float *dh;
    int *bh;
    float *o;
    int *counts, *offsets, *pair_token, *pair_slot, *pair_of;
    int *chunk_expert, *chunk_begin, *chunk_len, *n_chunks;
    int4 *tc_list;        // chunks of more than small_max pairs, in chunk order: (chunk, expert, first pair, pairs)
    int *n_tc;            // their count
    int keep_h;
    int tc;               // contraction on tcgen05 tensor cores
    int chunk;            // pairs per chunk of the work list (GG_TOK, or TC_CHUNK on tensor cores)
    int max_chunks;       // capacity of the work list
    int small_max;        // chunks of at most this many pairs take the streaming
                          // small-group pass instead of the tensor cores (0: none)
    uint8_t *xq, *hq;     // [2][P][H], [2][P][I]: e4m3 planes 16 h and l of q = 16 h + l (tensor-core path)
    uint8_t *xqt;         // [2][T][H]: the planes of the tokens' x, in token order (tensor-core path)
    int *pair_hs;         // [P] each pair's block-0 scale slot in hs: chunk * nbi * 2 TC_CHUNK + place (tensor-core path)
    float *xs, *hs;       // [chunks][nb][2][TC_CHUNK]: per chunk and block, the pairs' scales da,
                          // then -4 bsum as float (tensor-core path)
    float *rnorm;         // [T + E] norms for the screened router
    float *rpart;         // [kScreenSplit][T][E] partial logits of the screening GEMM
    int *rcand, *rcount;  // [T][E], [T]: the experts each token's compensated logits are formed for
};

// Shared-memory bytes of one quantized activation vector of nb blocks
// (codes at QS_STRIDE, then scales and block sums), 128-byte rounded.
__host__ __device__ inline int act_bytes(int nb) { return ((nb * (QS_STRIDE + 8) + 127) / 128) * 128; }

// ---- router ----------------------------------------------------------------------

// Error-free transformations (Knuth's TwoSum, and the fused-multiply-add
// product error), used to evaluate router logits to twice binary32 precision
// with the "Dot2" compensated dot product of Ogita, Rump and Oishi (2005).
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// (hi, lo) + (hi, lo) in double-binary32 arithmetic: TwoSum of the high
// parts, the low parts added into the error, then renormalized with
// Fast2Sum. Relative error of order 2^-44 of the operands' magnitude.
__device__ __forceinline__ void ff_add(float ah, float al, float bh, float bl, float &sh, float &sl) {
    float s, e;
    two_sum(ah, bh, s, e);
    e = __fadd_rn(e, __fadd_rn(al, bl));
    sh = __fadd_rn(s, e);
    sl = __fsub_rn(e, __fsub_rn(sh, s));
}

// One router logit, sum_k w[k] x[k], by a block of 128 threads (H a
// multiple of 256; w and x 16-byte aligned). Each thread runs Dot2 over its
// float4s (all loads issued up front) with four independent (sum, error)
// pairs; partial results are combined as double-binary32 pairs across the
// warp (binary64 arithmetic is slow on this part). Returns the warp's
// partial as (hi, lo) in every lane; the caller adds the four warps' pairs
// in a fixed order. The result is within a few units of 2^-44 of the exact
// dot product relative to sum |w x|, so top-k decisions and softmax weights
// match an fp64 reference.
__device__ __forceinline__ void router_logit_block(const float *w, const float *x, int H, float &hi, float &lo) {
    const float4 *w4 = reinterpret_cast<const float4 *>(w);
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    float s[4] = {0.f, 0.f, 0.f, 0.f}, c[4] = {0.f, 0.f, 0.f, 0.f};
    const int n4 = H >> 2;
    // the router is read by every call: keep it in L2 ahead of the streamed experts
    const uint64_t pol = l2_policy_evict_last();
#pragma unroll 8
    for (int i = threadIdx.x; i < n4; i += 128) {
        const float4 wv = ldg_f4_hint(w4 + i, pol), xv = __ldg(x4 + i);
        const float ww[4] = {wv.x, wv.y, wv.z, wv.w}, xx[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float p = __fmul_rn(ww[q], xx[q]);
            const float pe = __fmaf_rn(ww[q], xx[q], -p);
            float t, te;
            two_sum(s[q], p, t, te);
            s[q] = t;
            c[q] = __fadd_rn(c[q], __fadd_rn(te, pe));
        }
    }
    float h01, l01, h23, l23;
    ff_add(s[0], c[0], s[1], c[1], h01, l01);
    ff_add(s[2], c[2], s[3], c[3], h23, l23);
    ff_add(h01, l01, h23, l23, hi, lo);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xffffffffu, hi, o), ol = __shfl_xor_sync(0xffffffffu, lo, o);
        ff_add(hi, lo, oh, ol, hi, lo);
    }
}

// One router logit by one warp (H a multiple of 128): Dot2 over the lane's
// float4s with four (sum, error) pairs, then double-binary32 sums across the
// warp. Every lane receives (hi, lo).
__device__ __forceinline__ void router_logit_warp(const float *w, const float *x, int H, float &hi, float &lo) {
    const int lane = threadIdx.x & 31;
    const float4 *w4 = reinterpret_cast<const float4 *>(w);
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    float s[4] = {0.f, 0.f, 0.f, 0.f}, c[4] = {0.f, 0.f, 0.f, 0.f};
    const int n4 = H >> 2;
#pragma unroll 4
    for (int i = lane; i < n4; i += 32) {
        const float4 wv = __ldg(w4 + i), xv = __ldg(x4 + i);
        const float ww[4] = {wv.x, wv.y, wv.z, wv.w}, xx[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float p = __fmul_rn(ww[q], xx[q]);
            const float pe = __fmaf_rn(ww[q], xx[q], -p);
            float t, te;
            two_sum(s[q], p, t, te);
            s[q] = t;
            c[q] = __fadd_rn(c[q], __fadd_rn(te, pe));
        }
    }
    float h01, l01, h23, l23;
    ff_add(s[0], c[0], s[1], c[1], h01, l01);
    ff_add(s[2], c[2], s[3], c[3], h23, l23);
    ff_add(h01, l01, h23, l23, hi, lo);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xffffffffu, hi, o), ol = __shfl_xor_sync(0xffffffffu, lo, o);
        ff_add(hi, lo, oh, ol, hi, lo);
    }
}

// Total order on binary32 values as unsigned keys (-0 folded into +0).
__device__ __forceinline__ uint32_t order_key(float f) {
    const uint32_t u = __float_as_uint(f + 0.0f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Sort key of expert e with logit (hi, lo), a normalized double-binary32
// pair: the hi key, then the top 22 bits of the lo key (the pair's order is
// the order of the exact values; 22 bits of lo resolve differences down to
// about 2^-37 of the logit, below the accuracy of its evaluation), then the
// lower expert index first. Distinct for distinct experts.
__device__ __forceinline__ unsigned long long topk_key(float hi, float lo, int e) {
    return (static_cast<unsigned long long>(order_key(hi)) << 32) |
           (static_cast<unsigned long long>(order_key(lo) >> 10) << 10) |
           static_cast<unsigned long long>(1023 - e);
}

// Top-k of E <= 32 * KPL logits (double-binary32 pairs, read through L2) by
// one warp, descending by key, ties to the lower index. Lane l holds the keys
// of experts l, l + 32, ... as (high, low) 32-bit words, sorted in
// descending order in registers by a bitonic network; each of the k rounds
// takes the largest head with two warp reductions (the high words, then the
// low words of the lanes whose head has that high word), and the owning lane
// shifts its list. Keys are distinct (their low bits are the expert index),
// so exactly one lane owns the maximum. Writes the selection, in rank order,
// to res. All lanes of the warp must call.
template <int KPL>
__device__ __forceinline__ void topk_warp_kpl(const float *lhi, const float *llo, int E, int k, int *res) {
    const int lane = threadIdx.x & 31;
    uint32_t kh[KPL], kl[KPL];  // (0, 0) is below every key
    float h[KPL], l[KPL];
#pragma unroll
    for (int i = 0; i < KPL; ++i) {  // all loads in flight before the first use
        const int e = lane + 32 * i;
        h[i] = e < E ? __ldcg(lhi + e) : 0.0f;
        l[i] = e < E ? __ldcg(llo + e) : 0.0f;
    }
#pragma unroll
    for (int i = 0; i < KPL; ++i) {
        const int e = lane + 32 * i;
        const unsigned long long key = e < E ? topk_key(h[i], l[i], e) : 0ull;
        kh[i] = static_cast<uint32_t>(key >> 32);
        kl[i] = static_cast<uint32_t>(key);
    }
    // bitonic sort, descending
#pragma unroll
    for (int size = 2; size <= KPL; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
#pragma unroll
            for (int i = 0; i < KPL; ++i) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool desc = (i & size) == 0;
                    const bool gt = kh[i] > kh[j] || (kh[i] == kh[j] && kl[i] > kl[j]);
                    if (gt != desc) {
                        const uint32_t th = kh[i], tl = kl[i];
                        kh[i] = kh[j], kl[i] = kl[j];
                        kh[j] = th, kl[j] = tl;
                    }
                }
            }
        }
    }
    for (int r = 0; r < k; ++r) {
        const uint32_t mh = __reduce_max_sync(0xffffffffu, kh[0]);
        const uint32_t ml = __reduce_max_sync(0xffffffffu, kh[0] == mh ? kl[0] : 0u);
        if (kh[0] == mh && kl[0] == ml) {
#pragma unroll
            for (int i = 0; i + 1 < KPL; ++i) kh[i] = kh[i + 1], kl[i] = kl[i + 1];
            kh[KPL - 1] = kl[KPL - 1] = 0u;
        }
        if (lane == 0) res[r] = 1023 - static_cast<int>(ml & 1023u);
    }
    __syncwarp();
}

// topk_warp_kpl with the register capacity chosen for E (<= 1024).
__device__ __forceinline__ void topk_warp(const float *lhi, const float *llo, int E, int k, int *res) {
    if (E <= 256)
        topk_warp_kpl<8>(lhi, llo, E, k, res);
    else if (E <= 512)
        topk_warp_kpl<16>(lhi, llo, E, k, res);
    else
        topk_warp_kpl<32>(lhi, llo, E, k, res);
}

// ---- double-binary32 softmax ----------------------------------------------------

__device__ __forceinline__ void fast_two_sum(float a, float b, float &s, float &e) {
    s = __fadd_rn(a, b);
    e = __fsub_rn(b, __fsub_rn(s, a));
}

// (ah, al) * (bh, bl), normalized.
__device__ __forceinline__ void ff_mul(float ah, float al, float bh, float bl, float &ph, float &pl) {
    const float p = __fmul_rn(ah, bh);
    float e = __fmaf_rn(ah, bh, -p);
    e = __fadd_rn(e, __fadd_rn(__fmul_rn(ah, bl), __fmul_rn(al, bh)));
    fast_two_sum(p, e, ph, pl);
}

// exp(d) for d = dh + dl <= 0 in double-binary32: d = n ln2 + r with ln2
// split into 0.693145751953125 + 1.428606765330187e-06 + 5.497923148104107e-14
// (the first part exact in n * part), |r| <= ln2 / 2, then the degree-13
// Taylor polynomial of e^r (coefficients 1/k! as pairs) in Horner form, and
// the scaling by 2^n. Relative error near 2^-44 for d >= -87.
__device__ __forceinline__ void ff_exp_nonpos(float dh, float dl, float &eh, float &el) {
    dh = fmaxf(dh, -100.0f);
    const float nf = rintf(__fmul_rn(dh, 1.4426950216293335f));
    const float t1 = __fsub_rn(dh, __fmul_rn(nf, 0.693145751953125f));
    const float p2 = __fmul_rn(nf, 1.428606765330187e-06f);
    const float e2 = __fmaf_rn(nf, 1.428606765330187e-06f, -p2);
    float rh, rl;
    ff_add(t1, dl, -p2, -e2, rh, rl);
    rl = __fsub_rn(rl, __fmul_rn(nf, 5.497923148104107e-14f));
    fast_two_sum(rh, rl, rh, rl);
    // 1/k!, k = 13 .. 0, as (hi, lo)
    const float ch[14] = {1.6059044372074283e-10f, 2.0876755879584152e-09f, 2.5052107943679403e-08f,
                          2.755731998149713e-07f,  2.7557318844628753e-06f, 2.4801587642286904e-05f,
                          0.00019841270113829523f, 0.0013888889225199819f,  0.008333333767950535f,
                          0.0416666679084301f,     0.1666666716337204f,     0.5f,
                          1.0f,                    1.0f};
    const float cl[14] = {-5.352526511562726e-18f, 1.1082839147459852e-16f, 4.4176230446483665e-16f,
                          -7.575112209051195e-15f, 3.793571224297229e-14f,  -3.40699609366682e-13f,
                          -2.725596874933456e-12f, -3.3631094437103215e-11f, -4.34617203337595e-10f,
                          -1.2417634698280722e-09f, -4.967053879312289e-09f, 0.0f,
                          0.0f,                    0.0f};
    float ph = ch[0], pl = cl[0];
#pragma unroll
    for (int i = 1; i < 14; ++i) {
        float mh, ml;
        ff_mul(ph, pl, rh, rl, mh, ml);
        ff_add(mh, ml, ch[i], cl[i], ph, pl);
    }
    const int n = static_cast<int>(nf);
    eh = ldexpf(ph, n);
    el = ldexpf(pl, n);
}

// Softmax weights of the selected logits sel[0..k) (k <= 32) by one warp:
// w_j = exp(l_j - l_0) / sum_i exp(l_i - l_0), in double-binary32
// arithmetic, each w_j rounded once to binary32 (so it matches a binary64
// evaluation rounded to binary32). Writes w[0..k) (any memory) from lanes
// j < k (followed by __syncwarp). All lanes must call.
__device__ __forceinline__ void softmax_ff_warp(const float *lhi, const float *llo, const int *sel, int k,
                                                float *w) {
    const int lane = threadIdx.x & 31;
    const int e0 = sel[0];
    const float h0 = __ldcg(lhi + e0), l0 = __ldcg(llo + e0);
    float eh = 0.0f, el = 0.0f;
    if (lane < k) {
        const int e = sel[lane];
        float dh, dl;
        ff_add(__ldcg(lhi + e), __ldcg(llo + e), -h0, -l0, dh, dl);
        ff_exp_nonpos(dh, dl, eh, el);
    }
    float sh = eh, sl = el;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xffffffffu, sh, o), ol = __shfl_xor_sync(0xffffffffu, sl, o);
        ff_add(sh, sl, oh, ol, sh, sl);
    }
    if (lane < k) {
        // q = e / s: one binary32 quotient, then a correction from the exact residual
        const float q = __fdiv_rn(eh, sh);
        float ph, pl;
        ff_mul(q, 0.0f, sh, sl, ph, pl);
        float rh, rl;
        ff_add(eh, el, -ph, -pl, rh, rl);
        const float q2 = __fdiv_rn(rh, sh);
        w[lane] = __fadd_rn(q, q2);
    }
    __syncwarp();
}

// ---- staging of up to two byte ranges on one barrier -----------------------------

// Stages `n` (1 or 2) ranges, each a multiple of 8 bytes from an 8-byte
// aligned source, into 16-byte aligned destinations on one mbarrier phase.
// Lane 0 arms the barrier with the sum of the 16-byte aligned interiors and
// issues their bulk copies; lanes 1..4 copy the 8-byte heads and tails.
// Returns through `ofs` the offset of each range's data in its destination.
__device__ __forceinline__ void stage_ranges(int lane, int n, uint8_t *const dst[2], const uint8_t *const src[2],
                                             const uint32_t bytes[2], uint64_t *bar, uint32_t ofs[2]) {
    uint32_t head[2], body[2], tail[2], total = 0;
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        if (p < n) {
            ofs[p] = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(src[p]) & 15u);
            head[p] = (ofs[p] != 0u && bytes[p] >= 8u) ? 8u : 0u;
            body[p] = ((bytes[p] - head[p]) / 16u) * 16u;
            tail[p] = bytes[p] - head[p] - body[p];
            total += body[p];
        }
    }
    if (lane == 0) {
        mbar_arrive_expect_tx(bar, total);
        // weight blocks are read once per call: evict-first keeps L2 for reused data
        const uint64_t pol = l2_policy_evict_first();
#pragma unroll
        for (int p = 0; p < 2; ++p)
            if (p < n && body[p]) bulk_g2s_hint(dst[p] + ofs[p] + head[p], src[p] + head[p], body[p], bar, pol);
    }
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        if (p < n) {
            if (lane == 1 + 2 * p && head[p])
                *reinterpret_cast<uint2 *>(dst[p] + ofs[p]) = __ldg(reinterpret_cast<const uint2 *>(src[p]));
            if (lane == 2 + 2 * p && tail[p])
                *reinterpret_cast<uint2 *>(dst[p] + ofs[p] + head[p] + body[p]) =
                    __ldg(reinterpret_cast<const uint2 *>(src[p] + head[p] + body[p]));
        }
    }
}

__device__ __forceinline__ uint32_t src_ofs(const void *p) {
    return static_cast<uint32_t>(reinterpret_cast<uintptr_t>(p) & 15u);
}

// Row groups per unit: the largest power of two r (at least 1) with
// r * per_rg <= cap blocks, where per_rg is the blocks one row group brings.
__host__ __device__ inline int pow2_rows(int cap, int per_rg) {
    int r = 1;
    while (r * 2 * per_rg <= cap) r *= 2;
    return r;
}

}  // namespace tq
