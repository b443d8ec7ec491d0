// Warp-level streaming of tq2_0_fx4 row groups through shared memory: the
// engine under the GEMV, the MoE gate/up/down kernels and the grouped decode.
//
// Each warp owns a ring of `stages` slots and an mbarrier per slot. A "job"
// is a contiguous range of row groups of one matrix; its rows are cut into
// units of `rpu` row groups (<= 32 blocks), copied with cp.async.bulk a few
// units ahead. In a unit, lane i owns block i: it forms the block's four
// exact int32 sums S with dp4a and the four products t = float(S) * (d * da)
// of the fixed float schedule, and stores t in shared memory; then one lane
// per row adds its row's t over the blocks in ascending order.
#pragma once

#include "tq_moe_common.cuh"

namespace tq {

struct MatJob {
    const uint8_t *mat;    // first byte of the matrix
    int64_t rg_begin;      // row-group range handled by this CTA
    int64_t rg_end;
    float *y;              // output rows (indexed by matrix row)
    int32_t *s_out;        // optional exact block sums [n][nb] (matrix rows)
    const uint8_t *qs;     // activation blocks in shared memory (QS_STRIDE apart)
    const float *das;      // activation scales (shared memory)
    const int *bss;        // activation block sums (shared memory)
    int nb;                // blocks per row group
};

__host__ __device__ inline int stream_tbuf_bytes(int rpu, int nb) { return ((rpu * 4 * (nb + 1) * 4 + 15) / 16) * 16; }

__host__ __device__ inline int stream_warp_bytes(int stages, int slot_bytes, int rpu, int nb) {
    return ((stages * slot_bytes + stream_tbuf_bytes(rpu, nb) + stages * 8 + 127) / 128) * 128;
}

__host__ __device__ inline int stream_slot_bytes(int rpu, int nb) { return ((rpu * nb * BLOCK_BYTES + 16 + 15) / 16) * 16; }

// Units of `job`, with `rpu` row groups each.
__device__ __forceinline__ int64_t job_units(const MatJob &j, int rpu) {
    return (j.rg_end - j.rg_begin + rpu - 1) / rpu;
}

struct WarpRing {
    uint8_t *slots;
    float *tbuf;
    uint64_t *bars;
    int stages;
    int slot_bytes;
    long long budget;  // cycles a copy may take before it is reported lost
};

__device__ __forceinline__ WarpRing carve_ring(uint8_t *wbase, int stages, int slot_bytes, int rpu, int nb) {
    WarpRing r;
    r.slots = wbase;
    r.tbuf = reinterpret_cast<float *>(wbase + stages * slot_bytes);
    r.bars = reinterpret_cast<uint64_t *>(wbase + stages * slot_bytes + stream_tbuf_bytes(rpu, nb));
    r.stages = stages;
    r.slot_bytes = slot_bytes;
    r.budget = kWaitBudgetCycles;
    return r;
}

// Initialize the ring's barriers (lane 0); the caller fences and syncs.
__device__ __forceinline__ void ring_init(const WarpRing &r) {
    if ((threadIdx.x & 31) == 0)
        for (int s = 0; s < r.stages; ++s) mbar_init(&r.bars[s], 1);
}

// Unit u of a job: rgs row groups from rg0 (a multiplication, no division).
__device__ __forceinline__ void unit_locate(const MatJob &j, int rpu, int64_t u, int64_t &rg0, int &rgs) {
    rg0 = j.rg_begin + u * rpu;
    rgs = static_cast<int>(imin64(rpu, j.rg_end - rg0));
}

__device__ __forceinline__ void unit_issue(const WarpRing &r, const MatJob &j, int rpu, int64_t u, int slot) {
    int rgs;
    int64_t rg0;
    unit_locate(j, rpu, u, rg0, rgs);
    const int64_t stripe = static_cast<int64_t>(j.nb) * BLOCK_BYTES;
    uint8_t *dst[2] = {r.slots + slot * r.slot_bytes, nullptr};
    const uint8_t *src[2] = {j.mat + rg0 * stripe, nullptr};
    const uint32_t bytes[2] = {static_cast<uint32_t>(rgs * stripe), 0u};
    uint32_t ofs[2];
    stage_ranges(threadIdx.x & 31, 1, dst, src, bytes, &r.bars[slot], ofs);
}

// Issue the first `stages` units of this warp's share (units first, first +
// step, ...) of the job. Only its matrix pointer and row range are used, so
// this may run before the activations are in shared memory.
__device__ __forceinline__ void warp_stream_prefetch(const WarpRing &r, const MatJob &j, int rpu, int64_t first,
                                                     int64_t step, int max_stages = 1 << 30) {
    const int64_t total = job_units(j, rpu);
    int64_t nx = first;
    for (int s = 0; s < r.stages && s < max_stages; ++s, nx += step)
        if (nx < total) unit_issue(r, j, rpu, nx, s);
}

// Issue the remaining prefetch slots [from, stages) after a partial
// warp_stream_prefetch(..., from).
__device__ __forceinline__ void warp_stream_prefetch_from(const WarpRing &r, const MatJob &j, int rpu,
                                                          int64_t first, int64_t step, int from) {
    const int64_t total = job_units(j, rpu);
    int64_t nx = first + from * step;
    for (int s = from; s < r.stages; ++s, nx += step)
        if (nx < total) unit_issue(r, j, rpu, nx, s);
}

// Consume this warp's units (prefetched by warp_stream_prefetch), refilling
// each slot with the unit `stages` steps ahead. Returns false if a copy
// never arrived (status recorded).
__device__ __forceinline__ bool warp_stream_run(const WarpRing &r, const MatJob &J, int rpu, int64_t first,
                                                int64_t step, int *status, int kernel_id) {
    const int lane = threadIdx.x & 31;
    const int64_t total = job_units(J, rpu);
    const int nb = J.nb;
    const int64_t stripe = static_cast<int64_t>(nb) * BLOCK_BYTES;
    const int rgl0 = lane / nb, b00 = lane - rgl0 * nb;  // the lane's first block of a unit
    int slot = 0;
    uint32_t parity = 0;
    for (int64_t u = first; u < total; u += step) {
        if (!__all_sync(0xffffffffu, mbar_wait(&r.bars[slot], parity, r.budget))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, kernel_id, static_cast<int>(u));
            return false;
        }
        __syncwarp();
        int rgs;
        int64_t rg0;
        unit_locate(J, rpu, u, rg0, rgs);
        const uint8_t *data = r.slots + slot * r.slot_bytes + src_ofs(J.mat + rg0 * stripe);
        const int nblk = rgs * nb;
        for (int i = lane, rgl = rgl0, b = b00; i < nblk; i += 32) {
            if (i != lane) {
                rgl = i / nb;
                b = i - rgl * nb;
            }
            const uint8_t *blk = data + i * BLOCK_BYTES;
            int S[4];
            block_dot(blk + CODE_OFS, J.qs + b * QS_STRIDE, J.bss[b], S);
            const float da = J.das[b];
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
                const float sc = __fmul_rn(block_scale(blk, rr), da);
                r.tbuf[(rgl * 4 + rr) * (nb + 1) + b] = __fmul_rn(static_cast<float>(S[rr]), sc);
            }
            if (J.s_out) {
#pragma unroll
                for (int rr = 0; rr < 4; ++rr) J.s_out[((rg0 + rgl) * 4 + rr) * nb + b] = S[rr];
            }
        }
        __syncwarp();
        for (int t = lane; t < rgs * 4; t += 32) {
            const float *tb = r.tbuf + t * (nb + 1);
            float acc = 0.0f;
            for (int b = 0; b < nb; ++b) acc = __fadd_rn(acc, tb[b]);
            J.y[rg0 * 4 + t] = acc;
        }
        __syncwarp();
        const int64_t nu = u + static_cast<int64_t>(r.stages) * step;
        if (nu < total) {
            fence_proxy_async_smem();
            unit_issue(r, J, rpu, nu, slot);
        }
        if (++slot == r.stages) {
            slot = 0;
            parity ^= 1u;
        }
    }
    return true;
}

}  // namespace tq

namespace tq {

// ---- units handed out partly statically, partly by a shared counter ----
//
// A warp first takes its static units (first, first + step, ... < end), then
// units dyn_base + atomicAdd(dyn_ctr, 1) while they are below total. The
// static share lets every warp prefetch before anything is known about its
// peers; the shared tail lets the CTAs that stream faster take more, so that
// all finish together.
struct UnitQueue {
    int64_t next, end, step;  // remaining static units of this warp
    int *dyn_ctr;
    int64_t dyn_base, total;

    // The warp's next unit, or -1 (warp-uniform; lane 0 takes dynamic units).
    __device__ __forceinline__ int64_t take() {
        if (next < end) {
            const int64_t u = next;
            next += step;
            return u;
        }
        int v = 0;
        if ((threadIdx.x & 31) == 0) v = atomicAdd(dyn_ctr, 1);
        v = __shfl_sync(0xffffffffu, v, 0);
        const int64_t u = dyn_base + v;
        return u < total ? u : -1;
    }
};

// A unit of streamed work: rgs row groups of a matrix starting at row group
// rg0, results to y (indexed by matrix row).
struct UnitRef {
    const uint8_t *mat;
    int64_t rg0;
    int rgs;
    float *y;
};

// Prefetch the first ring.stages units of the queue into the ring; the unit
// ids go to slot_u (register array of the caller). `map(u)` gives the
// UnitRef of unit u (matrix pointer and rows only are used here).
template <int MAXST, class Map>
__device__ __forceinline__ void warp_units_prefetch(const WarpRing &r, UnitQueue &q, int nb, Map map,
                                                    int64_t (&slot_u)[MAXST]) {
    const int64_t stripe = static_cast<int64_t>(nb) * BLOCK_BYTES;
#pragma unroll
    for (int s = 0; s < MAXST; ++s) {
        slot_u[s] = -1;
        if (s >= r.stages) continue;
        slot_u[s] = q.take();
        if (slot_u[s] < 0) continue;
        const UnitRef U = map(slot_u[s]);
        uint8_t *dst[2] = {r.slots + s * r.slot_bytes, nullptr};
        const uint8_t *src[2] = {U.mat + U.rg0 * stripe, nullptr};
        const uint32_t bytes[2] = {static_cast<uint32_t>(U.rgs * stripe), 0u};
        uint32_t ofs[2];
        stage_ranges(threadIdx.x & 31, 1, dst, src, bytes, &r.bars[s], ofs);
    }
}

// Consume the prefetched units and the rest of the queue, refilling each
// slot as it frees; after a unit's rows are written, done(u) runs on the
// whole warp. Activations: qs / das / bss in shared memory. Returns false
// if a copy never arrived (status recorded).
template <int MAXST, class Map, class Done>
__device__ __forceinline__ bool warp_units_run(const WarpRing &r, UnitQueue &q, int nb, const uint8_t *qs,
                                               const float *das, const int *bss, Map map, Done done,
                                               int64_t (&slot_u)[MAXST], int *status, int kernel_id) {
    const int lane = threadIdx.x & 31;
    const int64_t stripe = static_cast<int64_t>(nb) * BLOCK_BYTES;
    const int rgl0 = lane / nb, b00 = lane - rgl0 * nb;  // the lane's first block of a unit
    int slot = 0;
    uint32_t parity = 0;
    for (;; slot = (slot + 1 == r.stages) ? 0 : slot + 1, parity ^= (slot == 0) ? 1u : 0u) {
        int64_t u = -1;
#pragma unroll
        for (int s = 0; s < MAXST; ++s)
            if (s == slot) u = slot_u[s];
        if (u < 0) break;
        if (!__all_sync(0xffffffffu, mbar_wait(&r.bars[slot], parity, r.budget))) {
            if (lane == 0) report(status, TQFX4_ETIMEOUT, kernel_id, static_cast<int>(u));
            return false;
        }
        __syncwarp();
        const UnitRef U = map(u);
        const uint8_t *data = r.slots + slot * r.slot_bytes + src_ofs(U.mat + U.rg0 * stripe);
        const int nblk = U.rgs * nb;
        for (int i = lane, rgl = rgl0, b = b00; i < nblk; i += 32) {
            if (i != lane) {
                rgl = i / nb;
                b = i - rgl * nb;
            }
            const uint8_t *blk = data + i * BLOCK_BYTES;
            int S[4];
            block_dot(blk + CODE_OFS, qs + b * QS_STRIDE, bss[b], S);
            const float da = das[b];
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
                const float sc = __fmul_rn(block_scale(blk, rr), da);
                r.tbuf[(rgl * 4 + rr) * (nb + 1) + b] = __fmul_rn(static_cast<float>(S[rr]), sc);
            }
        }
        __syncwarp();
        for (int t = lane; t < U.rgs * 4; t += 32) {
            const float *tb = r.tbuf + t * (nb + 1);
            float acc = 0.0f;
            for (int b = 0; b < nb; ++b) acc = __fadd_rn(acc, tb[b]);
            U.y[U.rg0 * 4 + t] = acc;
        }
        __syncwarp();
        // refill this slot before the callback, so the copy is in flight meanwhile
        const int64_t nu = q.take();
#pragma unroll
        for (int s = 0; s < MAXST; ++s)
            if (s == slot) slot_u[s] = nu;
        if (nu >= 0) {
            fence_proxy_async_smem();
            const UnitRef N = map(nu);
            uint8_t *dst[2] = {r.slots + slot * r.slot_bytes, nullptr};
            const uint8_t *src[2] = {N.mat + N.rg0 * stripe, nullptr};
            const uint32_t bytes[2] = {static_cast<uint32_t>(N.rgs * stripe), 0u};
            uint32_t ofs[2];
            stage_ranges(lane, 1, dst, src, bytes, &r.bars[slot], ofs);
        }
        done(u);
    }
    return true;
}

}  // namespace tq
