// tqfx4_moe_ffn in one launch: the routed-expert MoE layer for one token
// (Tied Trit-Planes, Sec. 1 and 2.2: only the selected experts' blocks are
// read, each through the integer dot pass), as a cooperative grid of one
// CTA per SM, so that the expert weights stream from HBM without the gaps
// that kernel boundaries leave.
//
//   router   the logits of experts blockIdx.x, blockIdx.x + G, ... are
//            computed by the CTA's warps (a compensated Dot2 product kept as
//            a double-binary32 pair, the warps sharing an expert adding their
//            parts in a fixed order); one count per CTA after a fence
//            publishes them. While that count completes, the CTA quantizes x
//            into its shared memory (the quantizer of tqfx4_quantize_act).
//            Every CTA then selects the top-k from all logits itself: the
//            same routine on the same values, hence the same selection.
//   gate/up  the items (selected expert, gate or up, a 16-block slot of row
//            groups) are split into contiguous shares, one per CTA; its warps
//            take the share's items in turn and stream them through per-warp
//            rings of bulk copies (8320-byte slots). A lane forms the exact
//            block sums of two rows of one block (dp4a on the nibbles,
//            unsigned code times signed activation, S = sum u q - 4 bsum),
//            the products float(S) * (d * da) go to shared memory and the
//            slot is refilled at once; one lane per row then adds them in
//            block order and stores the row of g or u.
//   exchange with its gate/up items done a CTA issues one down slot per warp,
//            counts itself in after a fence (little in flight then, so the
//            fence is short), and waits for every CTA's count; it then reads
//            g and u of its expert (L2), issues the rest of its down slots,
//            forms h = silu(g) u and quantizes it per 256-block.
//   down     CTA (j, p) streams row range p of expert j's down matrix and
//            stores o_j for those rows; the last of the top-k CTAs of range p
//            (one counter per range, after a fence) adds out = sum_j w_j o_j
//            in rank order.
// The float schedule of every dot product is the fixed one (per row,
// acc = acc + float(S) * (d * da) over the blocks in ascending order, each
// operation rounded once), so the outputs are those of the three-kernel
// path and of the oracle bit for bit. Counters only decide when data is
// ready; they are zero between calls (the last CTA past each one resets
// it). Every wait is bounded: a wait that runs out records TQFX4_ETIMEOUT,
// raises an abort flag that ends the other CTAs' waits, and its warp drains
// its own copies before it returns (the workspace must then be zeroed
// again before the next call).
#include "tq_launch.h"
#include "tq_moe_common.cuh"

namespace tq {

namespace {

#ifndef FZ_WARPS_CFG
#define FZ_WARPS_CFG 8
#endif
constexpr int FZ_WARPS = FZ_WARPS_CFG;
constexpr int FZ_THREADS = FZ_WARPS * 32;
constexpr int FZ_SB = 16;                     // blocks a slot
constexpr int FZ_SLOT = FZ_SB * BLOCK_BYTES;  // 8320 bytes
constexpr int FZ_TB = 64 * 4;                 // per warp: the block terms of one slot (64 (row, block) pairs)
// Down slots a warp issues before the exchange: none, so that the exchange's
// fence, count and L2 reads do not queue behind copies of its own SM.
#ifndef FZ_D_EARLY
#define FZ_D_EARLY 0
#endif

// Counters at the top of the workspace's counter area (ctr[n_ctr - k]),
// away from the slots the three-kernel path uses; zero between calls.
constexpr int FZ_C_ROUTER = 1;  // CTAs whose logits are published
constexpr int FZ_C_H = 2;       // CTAs whose g and u rows are written
constexpr int FZ_C_DONE = 3;    // CTAs finished
constexpr int FZ_C_ABORT = 4;   // a bounded wait ran out
constexpr int FZ_C_RANGE = 16;  // + p: experts done with down row range p

struct FusedGeo {
    int G;            // CTAs (one per SM)
    int stages;       // slots a warp's ring holds
    int Lh, Rh, Qh;   // gate/up: blocks a row, row groups a slot (Lh <= 16), 16-block chunks a row (Lh >= 16)
    int Li, Rd, Qd;   // down: the same
    int gu_per_m;     // gate/up items (Rh row groups, Qh slots each) of one matrix: I / 4 / Rh
    int gu_items;     // top_k * 2 * gu_per_m
    int parts;        // down row ranges per expert: G / top_k
    int n_rgd;        // down row groups: H / 4
    int act_x;        // shared bytes of quantized x: 16 words x Lh blocks, then da and bsum
    int act_h;        // the same for the expert's h (Li blocks)
    int off_rings;    // start of the warps' rings
    int warp_bytes;   // one warp's ring, block terms and barriers
    int smem;
};

__host__ __device__ inline int fz_act_bytes(int L) { return ((L * (QK + 8) + 15) / 16) * 16; }

__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

__device__ __forceinline__ int ld_acquire(const int *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ int ld_relaxed(const int *p) {
    int v;
    asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// One thread waits (bounded) until *p >= target (acquire), or the abort flag
// is raised. Returns false on abort or timeout (raising the flag itself).
__device__ bool fz_wait_count(const int *p, int target, int *abortp, int *status, int where) {
    const long long t0 = clock64();
    for (int it = 0;; ++it) {
        if (ld_acquire(p) >= target) return true;
        if ((it & 31) == 31) {
            if (ld_relaxed(abortp)) return false;
            if (clock64() - t0 > kWaitBudgetCycles) {
                report(status, TQFX4_ETIMEOUT, K_ROUTER, where);
                atomicExch(abortp, 1);
                return false;
            }
        }
    }
}

// Quantizes the 256-element block whose 8 consecutive floats per lane are
// in v into the shared activation `act` of L blocks ([16-byte word][block],
// then da[L], bsum[L]) at block b, with the quantizer of
// tqfx4_quantize_act. Returns false if an element is not finite.
__device__ __forceinline__ bool fz_quant_into(const float v[8], uint8_t *act, int L, int b, uint2 &packed, float &d,
                                              int &sum) {
    const int lane = threadIdx.x & 31;
    const bool ok = quant_block_warp(v, packed, d, sum);
    *reinterpret_cast<uint2 *>(act + ((lane >> 1) * L + b) * 16 + 8 * (lane & 1)) = packed;
    if (lane == 0) {
        reinterpret_cast<float *>(act + QK * L)[b] = d;
        reinterpret_cast<int *>(act + QK * L + 4 * L)[b] = sum;
    }
    return ok;
}

// Block terms of one 16-block slot: lane l takes rows 2 rp, 2 rp + 1 (rp =
// l / 16) of the slot's block l % 16, which is block `b` of its row group
// `rgs` (row group within the slot); act holds the activation of L blocks.
// Writes float(S) * (d * da) to tb[(4 rgs + row) * tw + tcol].
__device__ __forceinline__ void fz_slot_terms(const uint8_t *slot, const uint8_t *act, int L, int rgs, int b,
                                              int tw, int tcol, float *tb) {
    const int lane = threadIdx.x & 31;
    const int bis = lane & 15, rp = lane >> 4;
    const uint8_t *blk = slot + bis * BLOCK_BYTES;
    int S0, S1;
    fx_row2_dot(reinterpret_cast<const uint2 *>(blk + CODE_OFS + 256 * rp), reinterpret_cast<const uint4 *>(act) + b,
                L, reinterpret_cast<const int *>(act + QK * L + 4 * L)[b], S0, S1);
    const float da = reinterpret_cast<const float *>(act + QK * L)[b];
    tb[(rgs * 4 + 2 * rp) * tw + tcol] = __fmul_rn(static_cast<float>(S0), __fmul_rn(block_scale(blk, 2 * rp), da));
    tb[(rgs * 4 + 2 * rp + 1) * tw + tcol] =
        __fmul_rn(static_cast<float>(S1), __fmul_rn(block_scale(blk, 2 * rp + 1), da));
}

// acc + the tw terms of row `row` in order (tw <= 16), loads issued first.
__device__ __forceinline__ float fz_row_sum(const float *tb, int row, int tw, float acc) {
    float t[FZ_SB];
#pragma unroll
    for (int i = 0; i < FZ_SB; ++i) t[i] = i < tw ? tb[row * tw + i] : 0.0f;
#pragma unroll
    for (int i = 0; i < FZ_SB; ++i)
        if (i < tw) acc = __fadd_rn(acc, t[i]);
    return acc;
}

// The gate/up item `it`: expert rank j, matrix m (0 gate, 1 up), first row
// group rg0. An item is Qh slots (the 16-block chunks of its rows, in
// order), all streamed by one warp, which carries the row sums across them.
__device__ __forceinline__ void fz_gu_item(const FusedGeo &f, int it, int &j, int &m, int &rg0) {
    j = it / (2 * f.gu_per_m);
    const int rem = it - j * 2 * f.gu_per_m;
    m = rem >= f.gu_per_m;
    rg0 = (rem - m * f.gu_per_m) * f.Rh;
}

// The down item k of row range [r0, r1): first row group rg and row groups
// nrg in its slots (Qd of them, one warp).
__device__ __forceinline__ void fz_d_item(const FusedGeo &f, int k, int r0, int r1, int &rg, int &nrg) {
    rg = r0 + k * f.Rd;
    nrg = min(f.Rd, r1 - rg);
}

// Warp-uniform bounded wait until *p >= target (acquire): lane 0 polls, the
// warp agrees on the outcome, so the warp stays converged for the barriers
// that follow. Returns false on abort or timeout.
__device__ __forceinline__ bool fz_warp_wait_count(const int *p, int target, int *abortp, int *status, int where) {
    int ok = 0;
    if ((threadIdx.x & 31) == 0) ok = fz_wait_count(p, target, abortp, status, where);
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

__global__ void __launch_bounds__(FZ_THREADS, 1) moe_fused_kernel(MoeArgs a, FusedGeo f) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int sel_s[TQFX4_MAX_TOP_K];
    __shared__ float w_s[TQFX4_MAX_TOP_K], selh_s[TQFX4_MAX_TOP_K], sell_s[TQFX4_MAX_TOP_K];
    __shared__ float part_h[FZ_WARPS], part_l[FZ_WARPS];
    __shared__ int ok_s, last_s, fail_s, hbad_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = a.top_k, G = f.G, S = f.stages;
    const int H = a.H, I = a.I;
    int *const ctr_top = a.ctr + a.n_ctr;
    int *const c_router = ctr_top - FZ_C_ROUTER, *const c_h = ctr_top - FZ_C_H;
    int *const c_done = ctr_top - FZ_C_DONE, *const c_abort = ctr_top - FZ_C_ABORT;

    uint8_t *const act = smem;  // quantized x during gate/up, then the expert's quantized h
    uint8_t *const slots = smem + f.off_rings + warp * f.warp_bytes;
    float *const tb = reinterpret_cast<float *>(slots + S * FZ_SLOT);
    uint64_t *const bars = reinterpret_cast<uint64_t *>(slots + S * FZ_SLOT + FZ_TB);
    if (threadIdx.x == 0) fail_s = hbad_s = 0;
    if (lane == 0)
        for (int i = 0; i < S; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
    TQ_STAMP(3, 0);

    // ---------------- router: this CTA's logits ----------------
    // experts e_i = blockIdx.x + G i (i < ne); warp w works on expert
    // i = w % ne together with the warps w' = i (mod ne), each on its slice
    // of H; the warps' parts are added in warp order
    const int ne = a.E > static_cast<int>(blockIdx.x) ? (a.E - static_cast<int>(blockIdx.x) + G - 1) / G : 0;
    int e_mine = -1, r_mine = 0;
    if (ne > 0) {
        const int i = warp % ne, r = warp / ne;
        const int nw = (FZ_WARPS - i + ne - 1) / ne;  // warps on expert i
        const int e = static_cast<int>(blockIdx.x) + G * i;
        e_mine = e;
        r_mine = r;
        const float4 *w4 = reinterpret_cast<const float4 *>(a.wr + static_cast<int64_t>(e) * H);
        const float4 *x4 = reinterpret_cast<const float4 *>(a.x);
        const uint64_t pol = l2_policy_evict_last();  // the router is read by every call
        float s4[4] = {0.f, 0.f, 0.f, 0.f}, c4[4] = {0.f, 0.f, 0.f, 0.f};
        const int n4 = H >> 2;
#pragma unroll 4
        for (int k4 = lane + 32 * r; k4 < n4; k4 += 32 * nw) {
            const float4 wv = ldg_f4_hint(w4 + k4, pol), xv = __ldg(x4 + k4);
            const float ww[4] = {wv.x, wv.y, wv.z, wv.w}, xx[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float pr = __fmul_rn(ww[q], xx[q]);
                const float pe = __fmaf_rn(ww[q], xx[q], -pr);
                float t, te;
                two_sum(s4[q], pr, t, te);
                s4[q] = t;
                c4[q] = __fadd_rn(c4[q], __fadd_rn(te, pe));
            }
        }
        float hi, lo, h01, l01, h23, l23;
        ff_add(s4[0], c4[0], s4[1], c4[1], h01, l01);
        ff_add(s4[2], c4[2], s4[3], c4[3], h23, l23);
        ff_add(h01, l01, h23, l23, hi, lo);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_xor_sync(0xffffffffu, hi, o), ol = __shfl_xor_sync(0xffffffffu, lo, o);
            ff_add(hi, lo, oh, ol, hi, lo);
        }
        if (lane == 0) {
            part_h[warp] = hi;
            part_l[warp] = lo;
        }
    }
    __syncwarp();
    __syncthreads();
    if (ne > 0 && r_mine == 0 && lane == 0) {
        const int i = warp % ne;
        float th = part_h[i], tl = part_l[i];
        for (int w2 = i + ne; w2 < FZ_WARPS; w2 += ne) ff_add(th, tl, part_h[w2], part_l[w2], th, tl);
        if (a.bias) ff_add(th, tl, __ldg(a.bias + e_mine), 0.0f, th, tl);
        a.logits[e_mine] = th;
        a.logits_lo[e_mine] = tl;
    }
    __syncwarp();
    __syncthreads();
    TQ_STAMP(3, 1);
    if (threadIdx.x == 0) {
        fence_acq_rel_gpu();  // the logits before the count (nothing else in flight: a short fence)
        atomicAdd(c_router, 1);
    }
    __syncwarp();
    // x into shared memory while the count completes
    bool finite = true;
    for (int b = warp; b < f.Lh; b += FZ_WARPS) {
        const float4 *src = reinterpret_cast<const float4 *>(a.x + b * QK + 8 * lane);
        const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
        const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        uint2 packed;
        float d;
        int sum;
        finite &= fz_quant_into(v, act, f.Lh, b, packed, d, sum);
        if (blockIdx.x == 0) {  // the quantized x for inspection
            *reinterpret_cast<uint2 *>(a.qx + b * QK + 8 * lane) = packed;
            if (lane == 0) {
                a.dx[b] = d;
                a.bx[b] = sum;
            }
        }
    }
    if (!finite && lane == 0 && blockIdx.x == 0) report(a.status, TQFX4_EDATA, K_ROUTER, -1);
    if (warp == 0) {
        const bool ok = fz_warp_wait_count(c_router, G, c_abort, a.status, -2);
        if (lane == 0) ok_s = ok;
    }
    __syncwarp();
    __syncthreads();
    TQ_STAMP(3, 2);
    if (!ok_s) return;  // every thread sees the same flag; no copy issued yet
    if (warp == 0) {
        topk_warp(a.logits, a.logits_lo, a.E, K, sel_s);
        if (blockIdx.x == 0 && lane < K) {
            a.sel[lane] = sel_s[lane];
            a.sel_out[lane] = sel_s[lane];
        }
    }
    __syncwarp();
    __syncthreads();
    TQ_STAMP(3, 3);

    // ---------------- the warp's slot sequence ----------------
    // gate/up items of this CTA: [gi0, gi1), the warp's are gi0 + warp + 8 k
    const int gi0 = static_cast<int>(static_cast<int64_t>(f.gu_items) * blockIdx.x / G);
    const int gi1 = static_cast<int>(static_cast<int64_t>(f.gu_items) * (blockIdx.x + 1) / G);
    const int gu_slots = (gi0 + warp < gi1 ? (gi1 - gi0 - warp + FZ_WARPS - 1) / FZ_WARPS : 0) * f.Qh;
    // down: CTA (dj, dp) streams row range dp of expert dj (CTAs past
    // parts * top_k have no down work); the warp's slots are the range's
    // items warp + 8 m, each Rd row groups or one 16-block chunk of one
    const bool has_d = static_cast<int>(blockIdx.x) < f.parts * K;
    const int dj = has_d ? static_cast<int>(blockIdx.x) / f.parts : 0;
    const int dp = has_d ? static_cast<int>(blockIdx.x) - dj * f.parts : 0;
    const int r0 = static_cast<int>(static_cast<int64_t>(f.n_rgd) * dp / f.parts);
    const int r1 = static_cast<int>(static_cast<int64_t>(f.n_rgd) * (dp + 1) / f.parts);
    const int d_items = has_d ? (r1 - r0 + f.Rd - 1) / f.Rd : 0;
    const int d_slots = (warp < d_items ? (d_items - warp + FZ_WARPS - 1) / FZ_WARPS : 0) * f.Qd;
    const int total = gu_slots + d_slots;
    const uint64_t policy = l2_policy_evict_first();

    // slot n of the sequence into ring slot n % S (lane 0 issues)
    auto issue = [&](int n) {
        uint8_t *dst = slots + (n % S) * FZ_SLOT;
        uint64_t *bar = &bars[n % S];
        const uint8_t *src;
        uint32_t bytes;
        if (n < gu_slots) {
            int j, m, rg0;
            const int k = n / f.Qh, q = n - k * f.Qh;
            fz_gu_item(f, gi0 + warp + FZ_WARPS * k, j, m, rg0);
            src = (m ? a.up : a.gate) + static_cast<int64_t>(sel_s[j]) * a.mb_gu +
                  (static_cast<int64_t>(rg0) * f.Lh + q * FZ_SB) * BLOCK_BYTES;
            bytes = FZ_SLOT;
        } else {
            int rg, nrg;
            const int t = n - gu_slots, k = t / f.Qd, q = t - k * f.Qd;
            fz_d_item(f, warp + FZ_WARPS * k, r0, r1, rg, nrg);
            src = a.down + static_cast<int64_t>(sel_s[dj]) * a.mb_d +
                  (static_cast<int64_t>(rg) * f.Li + q * FZ_SB) * BLOCK_BYTES;
            bytes = f.Li >= FZ_SB ? FZ_SLOT : static_cast<uint32_t>(nrg * f.Li * BLOCK_BYTES);
        }
        if (lane == 0) {
            mbar_arrive_expect_tx(bar, bytes);
            bulk_g2s_hint(dst, src, bytes, bar, policy);
        }
    };
    int next = 0;  // the next slot of the sequence to issue
    auto issue_upto = [&](int limit) {
        limit = min(limit, total);
        for (; next < limit; ++next) issue(next);
    };
    // one slot of the sequence: its block terms, its refill, its rows
    const int bis = lane & 15;
    float racc = 0.0f;
    auto consume = [&](int sn, int refill_limit) -> bool {
        const int rs = sn % S;
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[rs], static_cast<uint32_t>((sn / S) & 1)))) {
            if (lane == 0) {  // where the copy was lost: CTA, warp, slot
                report(a.status, TQFX4_ETIMEOUT, sn < gu_slots ? K_GATEUP : K_DOWN,
                       (static_cast<int>(blockIdx.x) << 16) | (warp << 12) | (sn & 0xfff));
                atomicExch(c_abort, 1);
                fail_s = 1;
            }
            return false;
        }
        const uint8_t *slot = slots + rs * FZ_SLOT;
        const bool gu = sn < gu_slots;
        int j = 0, m = 0, rg0 = 0, q = 0, nrg = 0;
        if (gu) {
            const int k = sn / f.Qh;
            q = sn - k * f.Qh;
            fz_gu_item(f, gi0 + warp + FZ_WARPS * k, j, m, rg0);
            nrg = f.Rh;
        } else {
            const int t = sn - gu_slots, k = t / f.Qd;
            q = t - k * f.Qd;
            fz_d_item(f, warp + FZ_WARPS * k, r0, r1, rg0, nrg);
        }
        const int L = gu ? f.Lh : f.Li;
        const int Q = gu ? f.Qh : f.Qd;
        const int tw = L <= FZ_SB ? L : FZ_SB;  // terms a row of this slot
        int rgs, b, tcol;
        if (L <= FZ_SB) {
            rgs = bis / L;
            b = bis - rgs * L;
            tcol = b;
        } else {
            rgs = 0;
            b = q * FZ_SB + bis;
            tcol = bis;
        }
        if (rgs < nrg) fz_slot_terms(slot, act, L, rgs, b, tw, tcol, tb);
        __syncwarp();
        fence_proxy_async_smem();  // the slot's reads before its refill
        issue_upto(refill_limit);
        if (lane < 4 * nrg) {
            if (q == 0) racc = 0.0f;
            racc = fz_row_sum(tb, lane, tw, racc);
            if (q == Q - 1) {
                const int row = rg0 * 4 + lane;
                if (gu)
                    (m ? a.u : a.g)[static_cast<int64_t>(j) * I + row] = racc;
                else
                    a.o[static_cast<int64_t>(dj) * H + row] = racc;
            }
        }
        __syncwarp();
        return true;
    };

    // ---------------- gate/up ----------------
    bool ok = true;
    int s = 0;
    issue_upto(min(S, gu_slots + FZ_D_EARLY));
    for (; s < gu_slots; ++s)
        if (!consume(s, min(s + 1 + S, gu_slots + FZ_D_EARLY))) {
            ok = false;
            break;
        }
    if (!ok)  // drain this warp's copies in flight (bounded) before anything else
        for (int n = s; n < next; ++n) mbar_wait(&bars[n % S], static_cast<uint32_t>((n / S) & 1));
    __syncwarp();
    __syncthreads();  // (A) this CTA's g and u rows are written
    TQ_STAMP(3, 4);

    // ---------------- exchange ----------------
    if (warp == 0) {
        if (lane == 0 && !fail_s) {
            fence_acq_rel_gpu();
            const int old = atomicAdd(c_h, 1);
            if (old == G - 1) *c_router = 0;  // every CTA is past the router: reset for the next call
        }
        const bool okw = fz_warp_wait_count(c_h, G, c_abort, a.status, -3);
        if (lane == 0) ok_s = okw && !fail_s;
    } else if (warp == 1) {  // the routing weights, for the combine
        if (lane < K) {
            selh_s[lane] = __ldcg(a.logits + sel_s[lane]);
            sell_s[lane] = __ldcg(a.logits_lo + sel_s[lane]);
        }
        __syncwarp();
        softmax_ff_sel(selh_s, sell_s, K, w_s);
        if (blockIdx.x == 0 && lane < K) {
            a.selw[lane] = w_s[lane];
            a.selw_out[lane] = w_s[lane];
        }
    }
    __syncwarp();
    __syncthreads();  // (B)
    TQ_STAMP(3, 5);
    if (!ok_s) {
        // drain the down copies issued before the exchange (bounded), then leave
        if (ok)
            for (int n = s; n < next; ++n) mbar_wait(&bars[n % S], static_cast<uint32_t>((n / S) & 1));
        return;
    }
    if (has_d) {
        // h of expert dj: warp w forms blocks w, w + 8, ... (its g and u
        // loads go out before the rest of the warp's down copies)
        const float *gj = a.g + static_cast<int64_t>(dj) * I;
        const float *uj = a.u + static_cast<int64_t>(dj) * I;
        for (int b0 = 0; b0 < f.Li; b0 += 2 * FZ_WARPS) {
            float4 gv[2][2], uv[2][2];
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int b = b0 + warp + r * FZ_WARPS;
                if (b < f.Li) {
                    const float4 *g4 = reinterpret_cast<const float4 *>(gj + b * QK + 8 * lane);
                    const float4 *u4 = reinterpret_cast<const float4 *>(uj + b * QK + 8 * lane);
                    gv[r][0] = __ldcg(g4);
                    gv[r][1] = __ldcg(g4 + 1);
                    uv[r][0] = __ldcg(u4);
                    uv[r][1] = __ldcg(u4 + 1);
                }
            }
            if (b0 == 0) issue_upto(gu_slots + S);
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int b = b0 + warp + r * FZ_WARPS;
                if (b < f.Li) {
                    const float gg[8] = {gv[r][0].x, gv[r][0].y, gv[r][0].z, gv[r][0].w,
                                         gv[r][1].x, gv[r][1].y, gv[r][1].z, gv[r][1].w};
                    const float uu[8] = {uv[r][0].x, uv[r][0].y, uv[r][0].z, uv[r][0].w,
                                         uv[r][1].x, uv[r][1].y, uv[r][1].z, uv[r][1].w};
                    float hv[8];
#pragma unroll
                    for (int t = 0; t < 8; ++t) hv[t] = tq_swiglu(gg[t], uu[t]);
                    uint2 packed;
                    float d;
                    int sum;
                    const bool fin = fz_quant_into(hv, act, f.Li, b, packed, d, sum);
                    if (!fin) hbad_s = 1;  // every lane alike (the flag is warp-uniform)
                    if (dp == 0) {  // h for inspection
                        const int64_t o = static_cast<int64_t>(dj) * I + b * QK + 8 * lane;
                        reinterpret_cast<float4 *>(a.h + o)[0] = make_float4(hv[0], hv[1], hv[2], hv[3]);
                        reinterpret_cast<float4 *>(a.h + o)[1] = make_float4(hv[4], hv[5], hv[6], hv[7]);
                    }
                }
            }
        }
    }
    issue_upto(gu_slots + S);
    __syncwarp();
    __syncthreads();  // (C) the expert's h is in shared memory
    TQ_STAMP(3, 6);
    if (has_d && dp == 0) {
        // the quantized h for inspection, from shared memory ([16-byte word][block])
        for (int t = threadIdx.x; t < 16 * f.Li; t += FZ_THREADS) {
            const int w = t / f.Li, b = t - w * f.Li;
            *reinterpret_cast<uint4 *>(a.qh + static_cast<int64_t>(dj) * I + b * QK + 16 * w) =
                reinterpret_cast<const uint4 *>(act)[t];
        }
        for (int b = threadIdx.x; b < f.Li; b += FZ_THREADS) {
            a.dh[dj * f.Li + b] = reinterpret_cast<const float *>(act + QK * f.Li)[b];
            a.bh[dj * f.Li + b] = reinterpret_cast<const int *>(act + QK * f.Li + 4 * f.Li)[b];
        }
        if (threadIdx.x == 0 && hbad_s) report(a.status, TQFX4_EDATA, K_DOWN, dj);
    }

    // ---------------- down ----------------
    for (; s < total; ++s)
        if (!consume(s, s + 1 + S)) {
            ok = false;
            break;
        }
    if (!ok)
        for (int n = s; n < next; ++n) mbar_wait(&bars[n % S], static_cast<uint32_t>((n / S) & 1));
    __syncwarp();
    __syncthreads();  // (D) this CTA's o rows are written
    TQ_STAMP(3, 7);
    if (fail_s) return;  // every thread sees the same flag

    // ---------------- combine: the last expert of row range dp adds them up ----------------
    if (warp == 0) {
        int last = 0;
        if (has_d && lane == 0) {
            fence_acq_rel_gpu();
            int old;
            asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(ctr_top - FZ_C_RANGE - dp)
                         : "memory");
            last = old == K - 1;
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (lane == 0) last_s = last;
    }
    __syncwarp();
    __syncthreads();  // (E)
    if (has_d && last_s) {
        const int n0 = r0 * 4, n1 = r1 * 4;
        for (int n = n0 + threadIdx.x; n < n1; n += FZ_THREADS) {
            float acc = 0.0f;
            for (int jj = 0; jj < K; ++jj)
                acc = __fadd_rn(acc, __fmul_rn(w_s[jj], __ldcg(a.o + static_cast<int64_t>(jj) * H + n)));
            a.out[n] = acc;
        }
        if (threadIdx.x == 0) ctr_top[-FZ_C_RANGE - dp] = 0;  // for the next call
    }
    // the last CTA resets the exchange counter for the next call (every CTA is past it)
    if (threadIdx.x == 0 && atomicAdd(c_done, 1) == G - 1) {
        *c_h = 0;
        *c_done = 0;
    }
}

}  // namespace

// Geometry of the fused decode for these shapes, or false if it does not
// apply (block counts per row in {2, 4, 8, 16} or a multiple of 16, the
// shared memory within bounds); the three-kernel path serves the rest.
static bool fused_geo(const MoeArgs &a, FusedGeo &f) {
    f = FusedGeo{};
    const int K = a.top_k;
    f.G = num_sms();
    f.Lh = a.H / QK;
    f.Li = a.I / QK;
    auto ok_l = [](int L) { return L % FZ_SB == 0 || (L >= 2 && FZ_SB % L == 0); };
    if (!ok_l(f.Lh) || !ok_l(f.Li) || K > TQFX4_MAX_TOP_K || a.E > TQFX4_MAX_EXPERTS) return false;
    if ((a.E + f.G - 1) / f.G > FZ_WARPS) return false;  // a CTA's logits: one warp per expert at least
    f.Rh = f.Lh >= FZ_SB ? 1 : FZ_SB / f.Lh;
    f.Qh = f.Lh >= FZ_SB ? f.Lh / FZ_SB : 1;
    f.Rd = f.Li >= FZ_SB ? 1 : FZ_SB / f.Li;
    f.Qd = f.Li >= FZ_SB ? f.Li / FZ_SB : 1;
    if ((a.I / 4) % f.Rh != 0) return false;
    f.gu_per_m = a.I / 4 / f.Rh;
    f.gu_items = K * 2 * f.gu_per_m;
    f.parts = f.G / K;
    f.n_rgd = a.H / 4;
    if (f.parts < 1 || f.parts + FZ_C_RANGE > a.n_ctr) return false;
    f.act_x = fz_act_bytes(f.Lh);
    f.act_h = fz_act_bytes(f.Li);
    const int act = f.act_x > f.act_h ? f.act_x : f.act_h;
    f.off_rings = ((act + 127) / 128) * 128;
    const int budget = max_smem_optin() - 512;  // the kernel's static shared memory
    for (f.stages = 3; f.stages >= 2; --f.stages) {
        f.warp_bytes = ((f.stages * FZ_SLOT + FZ_TB + 8 * f.stages + 127) / 128) * 128;
        f.smem = f.off_rings + FZ_WARPS * f.warp_bytes;
        if (f.smem <= budget) return true;
    }
    return false;
}

bool moe_fused_applies(const MoeArgs &a) {
    FusedGeo f;
    return fused_geo(a, f);
}

cudaError_t launch_moe_fused(const MoeArgs &a0, const float *x, float *out, int32_t *sel_idx, float *sel_w,
                             cudaStream_t st) {
    MoeArgs a = a0;
    a.x = x;
    a.out = out;
    a.sel_out = sel_idx;
    a.selw_out = sel_w;
    FusedGeo f;
    if (!fused_geo(a, f)) return cudaErrorInvalidValue;
    static unsigned char set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(moe_fused_kernel), set);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(f.G);
    cfg.blockDim = dim3(FZ_THREADS);
    cfg.dynamicSmemBytes = f.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident: they wait on one another's counts
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void *args[] = {&a, &f};
    return cudaLaunchKernelExC(&cfg, reinterpret_cast<const void *>(moe_fused_kernel), args);
}

}  // namespace tq
