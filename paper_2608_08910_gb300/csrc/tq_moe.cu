// tqfx4_moe_ffn: one token through a routed-expert MoE layer whose gate/up/
// down projections are tq2_0_fx4 matrices (Tied Trit-Planes, Sec. 1 and 2.2).
//
// Three launches, reading only the selected experts' bytes:
//   router   one CTA per expert: logit W_r[e] x + bias[e] by a compensated
//            binary32 dot product kept as a double-binary32 pair; extra CTAs
//            quantize x. The CTA that finishes last (one counter) selects
//            the top-k experts (one warp, registers and warp reductions).
//   gate_up  the CTAs stream the units (row-group ranges) of the selected
//            experts' gate and up matrices (tq_stream.cuh) and write g_j and
//            u_j.
//   down     CTA (j, p) issues its first weight copies (the selection is
//            known), then forms h_j = silu(g_j) u_j and quantizes it into
//            shared memory while one warp evaluates the softmax weights,
//            streams row range p of down_j and writes o_j. The last of the
//            top_k CTAs sharing row range p (one counter per range) combines
//            out = sum_j w_j o_j in rank order.
// gate/up hands out three quarters of its units statically and the rest
// through a shared counter, so that its CTAs finish together.
// gate_up and down are launched as programmatic dependents: each starts its
// prologue while its predecessor drains and waits (griddepcontrol.wait)
// before reading what the predecessor wrote.
// Counters only decide which CTA finishes a reduction; every output is a
// fixed sequence of binary32 operations, so results are bit-reproducible.
#include "tq_launch.h"
#include "tq_stream.cuh"

namespace tq {

// Counter slots at the start of the workspace's counter area (all but the
// first are zeroed by the router at every call).
constexpr int kCtrRouter = 0;   // router CTAs done
constexpr int kCtrZero = 1;     // first slot the router zeroes at every call
constexpr int kCtrGateUp = 1;   // gate/up: shared unit counter
constexpr int kCtrDown = 2;     // down: one counter per row range
constexpr int kMaxStages = 2;   // ring depth of the gate/up kernel

// ---------------------------------------------------------------- router

__global__ void __launch_bounds__(128) router_kernel(MoeArgs a) {
    TQ_STAMP(0, 0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __shared__ float part_hi[4], part_lo[4];
    __shared__ int last;
    __shared__ int sel_s[TQFX4_MAX_TOP_K];
    if (static_cast<int>(blockIdx.x) >= a.E) {
        // x quantization, one warp per 256-block
        const int b = (blockIdx.x - a.E) * 4 + warp;
        if (b >= a.nbh) return;
        const float4 *src = reinterpret_cast<const float4 *>(a.x + b * QK + 8 * lane);
        const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
        const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        uint2 packed;
        float d;
        int sum;
        const bool ok = quant_block_warp(v, packed, d, sum);
        *reinterpret_cast<uint2 *>(a.qx + b * QK + 8 * lane) = packed;
        if (lane == 0) {
            a.dx[b] = d;
            a.bx[b] = sum;
            if (!ok) report(a.status, TQFX4_EDATA, K_ROUTER, b);
        }
        return;
    }
    grid_dependents_launch();  // let the gate/up kernel's CTAs get resident early
    const int e = blockIdx.x;
    if (e == 0)  // the down kernel's counters start every call at zero
        for (int i = threadIdx.x; i < a.n_ctr - kCtrZero; i += blockDim.x) a.ctr[kCtrZero + i] = 0;
    float hi, lo;
    router_logit_block(a.wr + static_cast<int64_t>(e) * a.H, a.x, a.H, hi, lo);
    TQ_STAMP(0, 1);
    if (lane == 0) {
        part_hi[warp] = hi;
        part_lo[warp] = lo;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float h01, l01, h23, l23;
        ff_add(part_hi[0], part_lo[0], part_hi[1], part_lo[1], h01, l01);
        ff_add(part_hi[2], part_lo[2], part_hi[3], part_lo[3], h23, l23);
        ff_add(h01, l01, h23, l23, hi, lo);
        if (a.bias) ff_add(hi, lo, __ldg(a.bias + e), 0.0f, hi, lo);
        a.logits[e] = hi;
        a.logits_lo[e] = lo;
        // one expert: this CTA is the last (its logit is its own), no count
        last = a.E == 1 || atomic_add_acq_rel(&a.ctr[kCtrRouter], 1) == a.E - 1;
    }
    __syncthreads();
    TQ_STAMP(0, 2);
    if (!last) return;
    if (warp == 0) topk_warp(a.logits, a.logits_lo, a.E, a.top_k, sel_s);
    __syncthreads();
    TQ_STAMP(0, 5);
    if (threadIdx.x < a.top_k) {
        a.sel[threadIdx.x] = sel_s[threadIdx.x];
        a.sel_out[threadIdx.x] = sel_s[threadIdx.x];
    }
    if (a.route_only && warp == 1) {  // the routing weights (else the down kernel forms them)
        float w_s[TQFX4_MAX_TOP_K];
        softmax_ff_warp(a.logits, a.logits_lo, sel_s, a.top_k, w_s);
        if (lane < a.top_k) {
            a.selw[lane] = w_s[lane];
            a.selw_out[lane] = w_s[lane];
        }
    }
    if (threadIdx.x == 0) a.ctr[kCtrRouter] = 0;
    TQ_STAMP(0, 3);
}

// ---------------------------------------------------------------- gate/up

// Work of gate_up: the units (rpu_gu row groups) of every selected expert's
// gate and up matrices, numbered u = (j * 2 + q) * upm + r. Each CTA streams
// a static contiguous share, then takes units from one shared counter.
__global__ void __launch_bounds__(256, 1) gate_up_kernel(MoeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    TQ_STAMP(1, 0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nbh = a.nbh;
    __shared__ int sel_s[TQFX4_MAX_TOP_K];
    __shared__ const uint8_t *ptr_s[2 * TQFX4_MAX_TOP_K];
    uint8_t *qs = smem;
    float *das = reinterpret_cast<float *>(qs + nbh * QS_STRIDE);
    int *bss = reinterpret_cast<int *>(das + nbh);
    const WarpRing ring = carve_ring(
        smem + act_bytes(nbh) + warp * stream_warp_bytes(a.stages_gu, a.slot_gu, a.rpu_gu, nbh), a.stages_gu,
        a.slot_gu, a.rpu_gu, nbh);
    ring_init(ring);
    fence_barrier_init();
    grid_dependency_wait();  // the router's selection and quantized x
    TQ_STAMP(1, 1);
    grid_dependents_launch();
    // issue the activation loads first: weight copies issued before them
    // would queue ahead in the memory system
    ActRegs act;
    if (!a.single) act_load(a.qx, a.dx, a.bx, nbh, act);
    if (threadIdx.x < a.top_k) {
        int e = a.single ? 0 : __ldcg(a.sel + threadIdx.x);
        if (!TQ_DEBUG_CHECK(e >= 0 && e < a.E, a.status, K_GATEUP, -2)) e = 0;
        sel_s[threadIdx.x] = e;
    }
    if (a.ptrs && threadIdx.x < 2 * a.top_k) ptr_s[threadIdx.x] = a.ptrs[threadIdx.x];
    __syncthreads();
    const int64_t n_rg = a.I / 4;
    const int64_t upm = (n_rg + a.rpu_gu - 1) / a.rpu_gu;
    const int64_t total = static_cast<int64_t>(a.top_k) * 2 * upm;
    UnitQueue q;
    q.next = static_cast<int64_t>(blockIdx.x) * a.static_gu + warp;
    q.end = static_cast<int64_t>(blockIdx.x + 1) * a.static_gu;
    q.step = a.warps_gu;
    q.dyn_ctr = a.ctr + kCtrGateUp;
    q.dyn_base = static_cast<int64_t>(gridDim.x) * a.static_gu;
    q.total = total;
    const int upm32 = static_cast<int>(upm);  // units are few: 32-bit index arithmetic
    auto map = [&](int64_t u) {
        const int u32 = static_cast<int>(u);
        const int j = u32 / (2 * upm32);
        const int rem = u32 - j * 2 * upm32;
        const int qq = rem >= upm32;
        const int64_t r = rem - qq * upm32;
        UnitRef U;
        U.mat = a.ptrs ? ptr_s[qq * a.top_k + j] : (qq ? a.up : a.gate) + static_cast<int64_t>(sel_s[j]) * a.mb_gu;
        U.rg0 = r * a.rpu_gu;
        U.rgs = static_cast<int>(imin64(a.rpu_gu, n_rg - U.rg0));
        U.y = (qq ? a.u : a.g) + static_cast<int64_t>(j) * a.I;
        return U;
    };
    int64_t slot_u[kMaxStages];
    warp_units_prefetch(ring, q, nbh, map, slot_u);
    if (a.single) {
        // x quantized here while the first copies fly (the quantizer of
        // tqfx4_quantize_act, one warp per 256-block); CTA 0 keeps it in the
        // workspace for inspection
        bool finite = true;
        for (int b = warp; b < nbh; b += a.warps_gu) {
            const float4 *src = reinterpret_cast<const float4 *>(a.x + b * QK + 8 * lane);
            const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
            const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            uint2 packed;
            float d;
            int sum;
            finite &= quant_block_warp(v, packed, d, sum);
            *reinterpret_cast<uint2 *>(qs + b * QS_STRIDE + 8 * lane) = packed;
            if (lane == 0) {
                das[b] = d;
                bss[b] = sum;
            }
            if (blockIdx.x == 0) {
                *reinterpret_cast<uint2 *>(a.qx + b * QK + 8 * lane) = packed;
                if (lane == 0) {
                    a.dx[b] = d;
                    a.bx[b] = sum;
                }
            }
        }
        if (!finite && blockIdx.x == 0 && lane == 0) report(a.status, TQFX4_EDATA, K_GATEUP, -1);
        __syncwarp();
    } else {
        act_store(act, nbh, qs, das, bss);
    }
    __syncthreads();
    TQ_STAMP(1, 2);
    warp_units_run(ring, q, nbh, qs, das, bss, map, [](int64_t) {}, slot_u, a.status, K_GATEUP);
    TQ_STAMP(1, 3);
}

// ---------------------------------------------------------------- down

__global__ void __launch_bounds__(256, 1) down_kernel(MoeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    TQ_STAMP(2, 0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nbi = a.nbi, K = a.top_k;
    __shared__ int last;
    __shared__ float selw_s[TQFX4_MAX_TOP_K];
    uint8_t *qs = smem;
    float *das = reinterpret_cast<float *>(qs + nbi * QS_STRIDE);
    int *bss = reinterpret_cast<int *>(das + nbi);
    const WarpRing ring = carve_ring(
        smem + act_bytes(nbi) + warp * stream_warp_bytes(a.stages_d, a.slot_d, a.rpu_d, nbi), a.stages_d,
        a.slot_d, a.rpu_d, nbi);
    ring_init(ring);
    fence_barrier_init();
    const int j = blockIdx.x / a.parts_d, p = blockIdx.x - j * a.parts_d;
    int64_t e = (a.ptrs || a.single) ? 0 : __ldcg(a.sel + j);
    if (!TQ_DEBUG_CHECK(e >= 0 && e < a.E, a.status, K_DOWN, -2)) e = 0;
    const int64_t n_rg = a.H / 4;
    MatJob job;
    job.mat = a.ptrs ? a.ptrs[2 * K + j] : a.down + e * a.mb_d;
    job.rg_begin = part_begin(n_rg, a.rpu_d, a.parts_d, p);
    job.rg_end = part_begin(n_rg, a.rpu_d, a.parts_d, p + 1);
    job.y = a.o + static_cast<int64_t>(j) * a.H;
    job.s_out = nullptr;
    job.qs = qs;
    job.das = das;
    job.bss = bss;
    job.nb = nbi;
    const bool any = job.rg_begin < job.rg_end;
    if (any) warp_stream_prefetch(ring, job, a.rpu_d, warp, a.warps_d, 1);
    if (a.single) {
        if (threadIdx.x == 0) selw_s[0] = 1.0f;  // the one expert's weight
    } else if (warp == a.warps_d - 1) {
        // the routing weights (needed by the combine at the end); the router
        // has completed, so this runs while gate/up drains
        int sel_l[TQFX4_MAX_TOP_K];
        for (int i = 0; i < K; ++i) sel_l[i] = __ldcg(a.sel + i);
        softmax_ff_warp(a.logits, a.logits_lo, sel_l, K, selw_s);
        if (blockIdx.x == 0 && lane < K) {
            a.selw[lane] = selw_s[lane];
            if (a.selw_out) a.selw_out[lane] = selw_s[lane];
        }
    }
    TQ_STAMP(2, 1);
    grid_dependency_wait();  // g and u of the gate/up kernel
    TQ_STAMP(2, 2);
    if (blockIdx.x == 0 && threadIdx.x == 0) {  // for the next call
        a.ctr[kCtrRouter] = 0;
        if (a.single) a.ctr[kCtrGateUp] = 0;  // no router zeroes it
    }
    // h_j = silu(g_j) u_j and its int8 quantization, one 256-block per warp;
    // the g/u loads go out before the rest of the weight prefetch
    const float *gj = a.g + static_cast<int64_t>(j) * a.I;
    const float *uj = a.u + static_cast<int64_t>(j) * a.I;
    for (int b0 = 0; b0 < nbi; b0 += a.warps_d) {
        const int b = b0 + warp;
        const bool mine = b < nbi;
        float gg[8], uu[8];
        if (mine) {
            const int o = b * QK + 8 * lane;
            const float4 g0 = __ldcg(reinterpret_cast<const float4 *>(gj + o));
            const float4 g1 = __ldcg(reinterpret_cast<const float4 *>(gj + o) + 1);
            const float4 u0 = __ldcg(reinterpret_cast<const float4 *>(uj + o));
            const float4 u1 = __ldcg(reinterpret_cast<const float4 *>(uj + o) + 1);
            gg[0] = g0.x; gg[1] = g0.y; gg[2] = g0.z; gg[3] = g0.w;
            gg[4] = g1.x; gg[5] = g1.y; gg[6] = g1.z; gg[7] = g1.w;
            uu[0] = u0.x; uu[1] = u0.y; uu[2] = u0.z; uu[3] = u0.w;
            uu[4] = u1.x; uu[5] = u1.y; uu[6] = u1.z; uu[7] = u1.w;
        }
        if (!mine) continue;
        const int o = b * QK + 8 * lane;
        TQ_STAMP(2, 6);
        float hv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) hv[i] = tq_swiglu(gg[i], uu[i]);
        TQ_STAMP(2, 7);
        uint2 packed;
        float d;
        int sum;
        const bool ok = quant_block_warp(hv, packed, d, sum);
        *reinterpret_cast<uint2 *>(qs + b * QS_STRIDE + 8 * lane) = packed;
        if (lane == 0) {
            das[b] = d;
            bss[b] = sum;
        }
        if (p == 0) {  // one CTA per expert leaves h and its quantization in the workspace
            float *hj = a.h + static_cast<int64_t>(j) * a.I + o;
            reinterpret_cast<float4 *>(hj)[0] = make_float4(hv[0], hv[1], hv[2], hv[3]);
            reinterpret_cast<float4 *>(hj)[1] = make_float4(hv[4], hv[5], hv[6], hv[7]);
            *reinterpret_cast<uint2 *>(a.qh + static_cast<int64_t>(j) * a.I + o) = packed;
            if (lane == 0) {
                a.dh[j * nbi + b] = d;
                a.bh[j * nbi + b] = sum;
                if (!ok) report(a.status, TQFX4_EDATA, K_DOWN, j * nbi + b);
            }
        }
    }
    if (any) warp_stream_prefetch_from(ring, job, a.rpu_d, warp, a.warps_d, 1);
    __syncthreads();
    TQ_STAMP(2, 3);
    if (any) warp_stream_run(ring, job, a.rpu_d, warp, a.warps_d, a.status, K_DOWN);
    __syncthreads();
    TQ_STAMP(2, 4);
    // top-1: this CTA alone holds row range p (its rows are its own), no count
    if (threadIdx.x == 0) last = K == 1 || atomic_add_acq_rel(&a.ctr[kCtrDown + p], 1) == K - 1;
    __syncthreads();
    if (!last) return;
    const int64_t r0 = job.rg_begin * 4, r1 = job.rg_end * 4;
    for (int64_t n = r0 + threadIdx.x; n < r1; n += blockDim.x) {
        float acc = 0.0f;
        for (int jj = 0; jj < K; ++jj)
            acc = __fadd_rn(acc, __fmul_rn(selw_s[jj], __ldcg(a.o + static_cast<int64_t>(jj) * a.H + n)));
        a.out[n] = acc;
    }
    TQ_STAMP(2, 5);
}

// ---------------------------------------------------------------- one expert, one launch

// tqfx4_expert_ffn in one cooperative launch of G CTAs (one per SM, all
// resident at once). The expert's bytes fit the SMs' shared memory, so
// every CTA requests its whole share of gate, up and down at its start, one
// bulk copy and one mbarrier per row group: CTA c owns row groups
// [c T / G, (c + 1) T / G) of gate and the same of up (T = I / 4), so it
// forms h = silu(g) u for its rows itself, and [c T' / G, (c + 1) T' / G) of
// down (T' = H / 4). While the copies fly it quantizes x (every CTA the
// whole vector); after its g, u and h rows, a grid-wide barrier (bounded)
// precedes the quantization of h, which every CTA forms for itself from
// the h rows of all, and the down rows follow from bytes already on chip.
// Arithmetic, intermediates in the workspace and output are those of the
// two-launch path (gate_up_kernel, down_kernel with `single`), bit for bit.
struct FfnGeo {
    int G;               // CTAs
    int rg_i, rg_d;      // row groups of gate (= of up), I / 4, and of down, H / 4
    int max_i, max_d;    // most row groups of gate (= of up) and of down a CTA owns
    int tb_bytes;        // block terms [row][block] (padded stride), then the row sums
    int smem;            // dynamic shared memory
    unsigned long long *arrived;  // grid barrier: CTAs arrived over all calls (8-byte aligned word of the counters)
};

__device__ __forceinline__ unsigned long long ld_acquire_gpu(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_release_gpu(unsigned long long *p, unsigned long long v) {
    asm volatile("red.release.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Grid-wide barrier of G resident CTAs over a 64-bit count of arrivals that
// only grows (G a call; it never wraps in practice). Every call starts with
// the count a multiple of G, and a CTA reads it before its own arrival, so
// target = (count / G + 1) G is this call's full count whatever the other
// CTAs have done by then. Arrival: one thread, after a CTA barrier, adds 1
// with release semantics (the CTA's writes before it) and polls with
// acquire loads until the target; gives up after kWaitBudgetCycles.
__device__ __forceinline__ unsigned long long grid_barrier_target(const unsigned long long *arrived, int G) {
    return (ld_acquire_gpu(arrived) / G + 1) * G;
}
__device__ __forceinline__ bool grid_barrier(unsigned long long *arrived, unsigned long long target) {
    red_release_gpu(arrived, 1ull);
    const long long t0 = clock64();
    while (ld_acquire_gpu(arrived) < target)
        if (clock64() - t0 > kWaitBudgetCycles) return false;
    return true;
}

// Exact sum S of one row of a block (the row's 128 code bytes at `codes`)
// against the activation block `qb` with sum `bsum`: block_dot's arithmetic
// for a single row.
__device__ __forceinline__ int row_dot(const uint8_t *codes, const uint8_t *qb, int bsum) {
    const uint2 *c2 = reinterpret_cast<const uint2 *>(codes);
    const uint2 *q2 = reinterpret_cast<const uint2 *>(qb);
    int lo0 = 0, lo1 = 0, hi0 = 0, hi1 = 0;  // four chains: integer sums, exact in any order
#pragma unroll 4
    for (int w = 0; w < 16; ++w) {
        const uint2 qa = q2[w], qh = q2[16 + w], c = c2[w];
        lo0 = dp4a_us(c.x & 0x0f0f0f0fu, qa.x, lo0);
        lo1 = dp4a_us(c.y & 0x0f0f0f0fu, qa.y, lo1);
        hi0 = dp4a_us(c.x & 0xf0f0f0f0u, qh.x, hi0);
        hi1 = dp4a_us(c.y & 0xf0f0f0f0u, qh.y, hi1);
    }
    return (lo0 + lo1) + ((hi0 + hi1) >> 4) - 4 * bsum;
}

// Terms t = float(S) * (d * da) of every (row, block) of the n_rg row
// groups at `w` into tb[(4 r + row) (nb + 1) + b], one item a thread (the
// row slowest, so that neighbouring threads read neighbouring blocks); each
// thread waits for its row group's copy. False if a copy never arrived.
__device__ __forceinline__ bool ffn_terms(const uint8_t *w, uint64_t *bars, int n_rg, int nb, const uint8_t *qs,
                                          const float *das, const int *bss, float *tb) {
    bool ok = true;
    const int per_row = n_rg * nb, rg_bytes = nb * BLOCK_BYTES;
    for (int i = threadIdx.x; i < 4 * per_row; i += blockDim.x) {
        const int rr = i / per_row, rem = i - rr * per_row;
        const int r = rem / nb, b = rem - r * nb;
        if (!mbar_wait(&bars[r], 0)) {
            ok = false;
            continue;
        }
        const uint8_t *blk = w + r * rg_bytes + b * BLOCK_BYTES;
        const int S = row_dot(blk + CODE_OFS + rr * ROW_BYTES, qs + b * QS_STRIDE, bss[b]);
        const float sc = __fmul_rn(block_scale(blk, rr), das[b]);
        tb[(r * 4 + rr) * (nb + 1) + b] = __fmul_rn(static_cast<float>(S), sc);
    }
    return ok;
}

constexpr int FFN_THREADS = 256;  // 512 measured 1.6 % slower at 4096 x 2048 (the copies bind, not the arithmetic)

__global__ void __launch_bounds__(FFN_THREADS, 1) expert_ffn_kernel(MoeArgs a, FfnGeo f) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    const int nbh = a.nbh, nbi = a.nbi, c = blockIdx.x;
    const int gu_bytes = nbh * BLOCK_BYTES, d_bytes = nbi * BLOCK_BYTES;  // one row group's
    uint8_t *wgu = smem;  // this CTA's gate row groups, then the same row groups of up
    uint8_t *wd = wgu + 2 * f.max_i * gu_bytes;
    uint8_t *qx = wd + f.max_d * d_bytes;
    float *dxs = reinterpret_cast<float *>(qx + nbh * QS_STRIDE);
    int *bxs = reinterpret_cast<int *>(dxs + nbh);
    uint8_t *qh = qx + act_bytes(nbh);
    float *dhs = reinterpret_cast<float *>(qh + nbi * QS_STRIDE);
    int *bhs = reinterpret_cast<int *>(dhs + nbi);
    float *tb = reinterpret_cast<float *>(qh + act_bytes(nbi));
    float *ys = tb + (f.tb_bytes / 4 - 8 * f.max_i);  // the g rows, then the u rows
    uint64_t *bars = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(tb) + f.tb_bytes);
    __shared__ int ok_s;
    unsigned long long target = 0;
    if (tid == 0) target = grid_barrier_target(f.arrived, f.G);
    const int i0 = static_cast<int>(static_cast<int64_t>(c) * f.rg_i / f.G);
    const int i1 = static_cast<int>(static_cast<int64_t>(c + 1) * f.rg_i / f.G);
    const int d0 = static_cast<int>(static_cast<int64_t>(c) * f.rg_d / f.G);
    const int d1 = static_cast<int>(static_cast<int64_t>(c + 1) * f.rg_d / f.G);
    const int ni = i1 - i0, ngu = 2 * ni, nd = d1 - d0;
    if (tid < ngu + nd) mbar_init(&bars[tid], 1);
    fence_barrier_init();
    __syncthreads();
    // x first (its loads would queue behind the weight copies), then every
    // weight byte of this CTA, one row group a thread: gate/up now, down
    // once the g and u terms are formed (gate/up's bytes are needed first;
    // down's still arrive before the grid barrier ends)
    float4 xv[2][2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const int b = warp + j * nw;
        if (b < nbh) {
            const float4 *src = reinterpret_cast<const float4 *>(a.x + b * QK + 8 * lane);
            xv[j][0] = __ldg(src);
            xv[j][1] = __ldg(src + 1);
        }
    }
    auto issue = [&](int i) {  // row-group copy i of this CTA: gate, up, then down
        const uint64_t policy = l2_policy_evict_first();
        const uint8_t *src;
        uint8_t *dst;
        int bytes;
        if (i < ngu) {
            const int64_t rg = i0 + (i < ni ? i : i - ni);
            src = (i < ni ? a.gate : a.up) + rg * gu_bytes;
            dst = wgu + i * gu_bytes;
            bytes = gu_bytes;
        } else {
            src = a.down + static_cast<int64_t>(d0 + i - ngu) * d_bytes;
            dst = wd + (i - ngu) * d_bytes;
            bytes = d_bytes;
        }
        mbar_arrive_expect_tx(&bars[i], static_cast<uint32_t>(bytes));
        bulk_g2s_hint(dst, src, static_cast<uint32_t>(bytes), &bars[i], policy);
    };
    if (tid < ngu) issue(tid);
    __syncwarp();
    // x quantized per 256-block while the copies fly (the quantizer of
    // tqfx4_quantize_act); CTA 0 leaves it in the workspace
    bool finite = true;
    for (int b = warp, j = 0; b < nbh; b += nw, ++j) {
        float4 v0, v1;
        if (j < 2) {
            v0 = j == 0 ? xv[0][0] : xv[1][0];
            v1 = j == 0 ? xv[0][1] : xv[1][1];
        } else {
            const float4 *src = reinterpret_cast<const float4 *>(a.x + b * QK + 8 * lane);
            v0 = __ldg(src);
            v1 = __ldg(src + 1);
        }
        const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        uint2 packed;
        float d;
        int sum;
        finite &= quant_block_warp(v, packed, d, sum);
        *reinterpret_cast<uint2 *>(qx + b * QS_STRIDE + 8 * lane) = packed;
        if (lane == 0) {
            dxs[b] = d;
            bxs[b] = sum;
        }
        if (c == 0) {
            *reinterpret_cast<uint2 *>(a.qx + b * QK + 8 * lane) = packed;
            if (lane == 0) {
                a.dx[b] = d;
                a.bx[b] = sum;
            }
        }
    }
    if (!finite && c == 0 && lane == 0) report(a.status, TQFX4_EDATA, K_GATEUP, -1);
    __syncwarp();
    __syncthreads();
    // g and u rows (the terms, then one thread per row adds its blocks in
    // order), then h = silu(g) u of the same rows
    bool ok = ffn_terms(wgu, bars, ngu, nbh, qx, dxs, bxs, tb);
    if (!__syncthreads_and(ok) && tid == 0) report(a.status, TQFX4_ETIMEOUT, K_GATEUP, c);
    if (tid >= ngu && tid < ngu + nd) issue(tid);
    __syncwarp();
    for (int t = tid; t < ngu * 4; t += blockDim.x) {
        const float *row = tb + t * (nbh + 1);
        float acc = 0.0f;
        for (int b = 0; b < nbh; ++b) acc = __fadd_rn(acc, row[b]);
        ys[t] = acc;
        const int up = t >= ni * 4;
        (up ? a.u : a.g)[i0 * 4 + t - up * ni * 4] = acc;
    }
    __syncthreads();
    for (int t = tid; t < ni * 4; t += blockDim.x) a.h[i0 * 4 + t] = tq_swiglu(ys[t], ys[ni * 4 + t]);
    __syncthreads();
    if (tid == 0) {
        ok_s = grid_barrier(f.arrived, target);
        if (!ok_s) report(a.status, TQFX4_ETIMEOUT, K_DOWN, -3);
    }
    __syncthreads();
    // the quantization of h, one 256-block per warp, in every CTA (its down
    // rows need all of it); CTA 0 leaves it in the workspace
    for (int b = warp; b < nbi; b += nw) {
        const int o = b * QK + 8 * lane;
        const float4 h0 = __ldcg(reinterpret_cast<const float4 *>(a.h + o));
        const float4 h1 = __ldcg(reinterpret_cast<const float4 *>(a.h + o) + 1);
        const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
        uint2 packed;
        float d;
        int sum;
        const bool hok = quant_block_warp(hv, packed, d, sum);
        *reinterpret_cast<uint2 *>(qh + b * QS_STRIDE + 8 * lane) = packed;
        if (lane == 0) {
            dhs[b] = d;
            bhs[b] = sum;
        }
        if (c == 0) {
            *reinterpret_cast<uint2 *>(a.qh + o) = packed;
            if (lane == 0) {
                a.dh[b] = d;
                a.bh[b] = sum;
                if (!hok) report(a.status, TQFX4_EDATA, K_DOWN, b);
            }
        }
    }
    __syncwarp();
    __syncthreads();
    // down rows, then out = 0 + 1 * o (the combine of a top-1 layer)
    ok = ffn_terms(wd, bars + ngu, nd, nbi, qh, dhs, bhs, tb);
    if (!__syncthreads_and(ok) && tid == 0) report(a.status, TQFX4_ETIMEOUT, K_DOWN, c);
    for (int t = tid; t < nd * 4; t += blockDim.x) {
        const float *row = tb + t * (nbi + 1);
        float acc = 0.0f;
        for (int b = 0; b < nbi; ++b) acc = __fadd_rn(acc, row[b]);
        const int n = d0 * 4 + t;
        a.o[n] = acc;
        a.out[n] = __fadd_rn(0.0f, __fmul_rn(1.0f, acc));
    }
}

// ---------------------------------------------------------------- host side

namespace {

// Launch `kernel(a)` as a programmatic dependent of the previous kernel in
// the stream (plain stream order when `plain`).
cudaError_t launch_pdl(const void *kernel, int grid, int block, int smem, cudaStream_t st, bool plain,
                       MoeArgs &a) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = plain ? 0 : 1;
    void *args[] = {&a};
    return cudaLaunchKernelExC(&cfg, kernel, args);
}

// Warps per CTA that fit the shared memory left after `act` bytes, 2 stages.
int fit_warps(int slot, int rpu, int nb, int act, int max_warps) {
    const int budget = max_smem_optin() - 1024 - act;
    int w = max_warps;
    while (w > 1 && w * stream_warp_bytes(2, slot, rpu, nb) > budget) --w;
    return w;
}

}  // namespace

// Geometry and workspace views for the decode (T = 1) path.
bool moe_decode_args(const tqfx4_experts *ex, const tqfx4_router *rt, void *ws, MoeArgs &a, MoeLayout &L) {
    a = MoeArgs{};
    a.E = static_cast<int>(ex->n_experts);
    a.H = static_cast<int>(ex->hidden);
    a.I = static_cast<int>(ex->inter);
    a.top_k = rt->top_k;
    a.nbh = a.H / QK;
    a.nbi = a.I / QK;
    a.mb_gu = static_cast<int64_t>(a.I / 4) * a.nbh * BLOCK_BYTES;
    a.mb_d = static_cast<int64_t>(a.H / 4) * a.nbi * BLOCK_BYTES;
    a.gate = static_cast<const uint8_t *>(ex->gate);
    a.up = static_cast<const uint8_t *>(ex->up);
    a.down = static_cast<const uint8_t *>(ex->down);
    a.wr = rt->weight;
    a.bias = rt->bias;
    L = moe_layout(a.E, a.H, a.I, a.top_k, 1, false, true);
    uint8_t *base = static_cast<uint8_t *>(ws);
    a.n_ctr = static_cast<int>(L.n_ctr);
    if (base) {
        a.status = reinterpret_cast<int *>(base);
        a.ctr = reinterpret_cast<int *>(base + L.ctr);
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
    }
    const int sms = num_sms();
    // gate/up: top_k x parts CTAs, each a contiguous range of row groups
    a.rpu_gu = pow2_rows(32, a.nbh);
    a.slot_gu = stream_slot_bytes(a.rpu_gu, a.nbh);
    a.stages_gu = 2;
    a.warps_gu = fit_warps(a.slot_gu, a.rpu_gu, a.nbh, act_bytes(a.nbh), 8);
    a.parts_gu = static_cast<int>(imax64(1, sms / a.top_k));

    // down: the same partition over the hidden rows
    a.rpu_d = pow2_rows(32, a.nbi);
    a.slot_d = stream_slot_bytes(a.rpu_d, a.nbi);
    a.stages_d = 2;
    a.warps_d = fit_warps(a.slot_d, a.rpu_d, a.nbi, act_bytes(a.nbi), 8);
    a.parts_d = static_cast<int>(imax64(1, sms / a.top_k));

    // gate/up's static share: three quarters of the units, split evenly; the
    // rest is handed out by the shared counter
    const int64_t upm_gu = (a.I / 4 + a.rpu_gu - 1) / a.rpu_gu;
    a.static_gu = static_cast<int>((static_cast<int64_t>(a.top_k) * 2 * upm_gu * 3 / 4) / (a.top_k * a.parts_gu));
    return static_cast<int64_t>(a.n_ctr) >= kCtrDown + a.parts_d;
}

int gate_up_smem(const MoeArgs &a) {
    return act_bytes(a.nbh) + a.warps_gu * stream_warp_bytes(a.stages_gu, a.slot_gu, a.rpu_gu, a.nbh);
}
int down_smem(const MoeArgs &a) {
    return act_bytes(a.nbi) + a.warps_d * stream_warp_bytes(a.stages_d, a.slot_d, a.rpu_d, a.nbi);
}

cudaError_t launch_moe_decode(const MoeArgs &a0, const float *x, float *out, int32_t *sel_idx, float *sel_w,
                              cudaStream_t st, void *const *events) {
    MoeArgs a = a0;
    a.x = x;
    a.out = out;
    a.sel_out = sel_idx;
    a.selw_out = sel_w;
    static unsigned char set_gu[64], set_dn[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(gate_up_kernel), set_gu);
    if (e == cudaSuccess) e = allow_max_smem(reinterpret_cast<const void *>(down_kernel), set_dn);
    if (e != cudaSuccess) return e;
    // under stream capture the records become event nodes of the graph
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (events) cudaStreamIsCapturing(st, &cap);
    auto rec = [&](int i) {
        if (events && events[i])
            cudaEventRecordWithFlags(static_cast<cudaEvent_t>(events[i]), st,
                                     cap == cudaStreamCaptureStatusActive ? cudaEventRecordExternal
                                                                          : cudaEventRecordDefault);
    };
    rec(0);
    router_kernel<<<a.E + (a.nbh + 3) / 4, 128, 0, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    rec(1);
    if ((e = launch_pdl(reinterpret_cast<const void *>(gate_up_kernel), a.top_k * a.parts_gu, a.warps_gu * 32,
                        gate_up_smem(a), st, events != nullptr, a)) != cudaSuccess)
        return e;
    rec(2);
    if ((e = launch_pdl(reinterpret_cast<const void *>(down_kernel), a.top_k * a.parts_d, a.warps_d * 32,
                        down_smem(a), st, events != nullptr, a)) != cudaSuccess)
        return e;
    rec(3);
    return cudaSuccess;
}

// n fp32 values (both ends 16-byte aligned, n a multiple of 4) from src to
// dst; src may be page-locked host memory seen through its device address.
__global__ void __launch_bounds__(256) copy_f32_kernel(float4 *dst, const float4 *__restrict__ src, int n4) {
    const int i = blockIdx.x * 256 + threadIdx.x;
    if (i < n4) dst[i] = src[i];
}

cudaError_t launch_copy_f32(float *dst, const float *src, int64_t n, cudaStream_t st) {
    const int n4 = static_cast<int>(n / 4);
    copy_f32_kernel<<<(n4 + 255) / 256, 256, 0, st>>>(reinterpret_cast<float4 *>(dst),
                                                       reinterpret_cast<const float4 *>(src), n4);
    return cudaGetLastError();
}

// The two halves of launch_moe_decode for callers that place the selected
// experts' blocks themselves between routing and the expert projections
// (an expert tier): the router alone (selection and routing weights), then
// gate/up and down over the given pointers.
cudaError_t launch_moe_route(const MoeArgs &a0, const float *x, int32_t *sel_idx, float *sel_w, cudaStream_t st) {
    MoeArgs a = a0;
    a.x = x;
    a.sel_out = sel_idx;
    a.selw_out = sel_w;
    a.route_only = 1;
    router_kernel<<<a.E + (a.nbh + 3) / 4, 128, 0, st>>>(a);
    return cudaGetLastError();
}

// Geometry of expert_ffn_kernel, or false where it does not apply (the two
// launches serve the call then): row-group copies 16-byte aligned (an even
// number of blocks a row), one copy per thread, every share in shared
// memory. The grid barrier's count takes two of the counter area's last
// three words, which no other kernel of the one-expert call uses.
static bool expert_ffn_geo(const MoeArgs &a, FfnGeo &f) {
    if (a.nbh % 2 != 0 || a.nbi % 2 != 0 || a.n_ctr < kCtrDown + a.parts_d + 3) return false;
    f.G = num_sms();
    f.rg_i = a.I / 4;
    f.rg_d = a.H / 4;
    f.max_i = (f.rg_i + f.G - 1) / f.G;
    f.max_d = (f.rg_d + f.G - 1) / f.G;
    if (2 * f.max_i + f.max_d > FFN_THREADS) return false;
    const int64_t tb = 4 * (imax64(static_cast<int64_t>(2 * f.max_i) * 4 * (a.nbh + 1),
                                   static_cast<int64_t>(f.max_d) * 4 * (a.nbi + 1)) +
                            8 * f.max_i);
    f.tb_bytes = static_cast<int>((tb + 15) / 16 * 16);
    const int64_t smem = static_cast<int64_t>(2 * f.max_i) * a.nbh * BLOCK_BYTES +
                         static_cast<int64_t>(f.max_d) * a.nbi * BLOCK_BYTES + act_bytes(a.nbh) + act_bytes(a.nbi) +
                         f.tb_bytes + 8 * (2 * f.max_i + f.max_d);
    if (smem > max_smem_optin() - 1024) return false;  // room for the static shared memory
    f.smem = static_cast<int>(smem);
    f.arrived = nullptr;
    if (a.ctr) {
        int *w = a.ctr + a.n_ctr - 2;  // the last two counters, or the two before them: 8-byte aligned
        if (reinterpret_cast<uintptr_t>(w) % 8 != 0) --w;
        f.arrived = reinterpret_cast<unsigned long long *>(w);
    }
    return true;
}

bool expert_ffn_one_launch(const MoeArgs &a) {
    FfnGeo f;
    return expert_ffn_geo(a, f);
}

// One expert's FFN without a router: one cooperative launch of
// expert_ffn_kernel where its geometry applies, else gate/up (x quantized
// inside) and down as programmatic dependents; events[0..2] (optional)
// before, between and after the two (after the one launch: events[1] and
// events[2] together).
cudaError_t launch_expert_ffn(const MoeArgs &a0, const float *x, float *out, cudaStream_t st,
                              void *const *events) {
    MoeArgs a = a0;
    a.x = x;
    a.out = out;
    a.sel_out = nullptr;
    a.selw_out = nullptr;
    a.single = 1;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (events) cudaStreamIsCapturing(st, &cap);
    auto rec = [&](int i) {
        if (events && events[i])
            cudaEventRecordWithFlags(static_cast<cudaEvent_t>(events[i]), st,
                                     cap == cudaStreamCaptureStatusActive ? cudaEventRecordExternal
                                                                          : cudaEventRecordDefault);
    };
    cudaError_t e;
    FfnGeo f;
    if (expert_ffn_geo(a, f)) {
        static unsigned char set_ffn[64];
        if ((e = allow_max_smem(reinterpret_cast<const void *>(expert_ffn_kernel), set_ffn)) != cudaSuccess)
            return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(f.G);
        cfg.blockDim = dim3(FFN_THREADS);
        cfg.dynamicSmemBytes = f.smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeCooperative;
        attr[0].val.cooperative = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        void *args[] = {&a, &f};
        rec(0);
        if ((e = cudaLaunchKernelExC(&cfg, reinterpret_cast<const void *>(expert_ffn_kernel), args)) != cudaSuccess)
            return e;
        rec(1);
        rec(2);
        return cudaSuccess;
    }
    static unsigned char set_gu[64], set_dn[64];
    e = allow_max_smem(reinterpret_cast<const void *>(gate_up_kernel), set_gu);
    if (e == cudaSuccess) e = allow_max_smem(reinterpret_cast<const void *>(down_kernel), set_dn);
    if (e != cudaSuccess) return e;
    rec(0);
    if ((e = launch_pdl(reinterpret_cast<const void *>(gate_up_kernel), a.top_k * a.parts_gu, a.warps_gu * 32,
                        gate_up_smem(a), st, events != nullptr, a)) != cudaSuccess)
        return e;
    rec(1);
    if ((e = launch_pdl(reinterpret_cast<const void *>(down_kernel), a.top_k * a.parts_d, a.warps_d * 32,
                        down_smem(a), st, events != nullptr, a)) != cudaSuccess)
        return e;
    rec(2);
    return cudaSuccess;
}

cudaError_t launch_moe_experts(const MoeArgs &a0, const void *const *ptrs, float *out, cudaStream_t st) {
    MoeArgs a = a0;
    a.out = out;
    a.ptrs = reinterpret_cast<const uint8_t *const *>(ptrs);
    a.sel_out = nullptr;
    a.selw_out = nullptr;
    static unsigned char set_gu[64], set_dn[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(gate_up_kernel), set_gu);
    if (e == cudaSuccess) e = allow_max_smem(reinterpret_cast<const void *>(down_kernel), set_dn);
    if (e != cudaSuccess) return e;
    if ((e = launch_pdl(reinterpret_cast<const void *>(gate_up_kernel), a.top_k * a.parts_gu, a.warps_gu * 32,
                        gate_up_smem(a), st, false, a)) != cudaSuccess)
        return e;
    return launch_pdl(reinterpret_cast<const void *>(down_kernel), a.top_k * a.parts_d, a.warps_d * 32, down_smem(a),
                      st, false, a);
}

}  // namespace tq
