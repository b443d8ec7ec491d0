// Device-side building blocks shared by the tqfx4 kernels (sm_103a only):
// the block geometry of tq2_0_fx4 (Tied Trit-Planes, Sec. 2.2), the device
// status word, mbarrier + cp.async.bulk staging, and the integer dot step.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "tqfx4.h"

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "libtqfx4 targets Blackwell (sm_103a) only"
#endif

namespace tq {

// Phase timestamps for development builds (-DTQ_INSTRUMENT): thread 0 of a
// CTA records %globaltimer into tq_stamps[kernel][cta][slot]. Compiled out
// otherwise.
#ifdef TQ_INSTRUMENT
extern __device__ unsigned long long tq_stamps[8][2048][8];
#define TQ_STAMP(k, s)                                                                              \
    do {                                                                                            \
        if (threadIdx.x == 0 && blockIdx.x < 2048) {                                                \
            unsigned long long t_;                                                                  \
            asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                                  \
            tq_stamps[k][blockIdx.x][s] = t_;                                                       \
        }                                                                                           \
    } while (0)
// Accumulate `v` into tq_stamps[k][cta][slot] (lane 0 of the calling warp).
#define TQ_ADD(k, s, v)                                                                             \
    do {                                                                                            \
        if ((threadIdx.x & 31) == 0 && blockIdx.x < 2048) atomicAdd(&tq_stamps[k][blockIdx.x][s], (unsigned long long)(v)); \
    } while (0)
#else
#define TQ_STAMP(k, s) ((void)0)
#define TQ_ADD(k, s, v) ((void)0)
#endif

constexpr int QK = 256;           // elements per block along K
constexpr int ROWS = 4;           // rows per block
constexpr int BLOCK_BYTES = 520;  // 8 scale bytes + 4 x 128 code bytes
constexpr int CODE_OFS = 8;       // codes follow the four f16 scales
constexpr int ROW_BYTES = 128;    // code bytes per row (256 nibbles)
constexpr int QS_STRIDE = 264;    // shared-memory stride of one 256-byte activation block
                                  // (33 x 8 bytes: consecutive blocks land on distinct banks)

// Kernel ids recorded with a device error (status word slot 1).
enum KernelId : int {
    K_PACK = 1, K_QUANT = 2, K_GEMV = 3, K_ROUTER = 4, K_GATEUP = 5, K_DOWN = 6,
    K_TOPK = 7, K_GROUP = 8, K_GGATEUP = 9, K_GDOWN = 10, K_COMBINE = 11, K_PREFILL = 12,
    K_SELFTEST = 13, K_VALIDATE = 14,
};

// Checks of data-dependent indices inside the kernels, compiled in by the
// debug build (-DTQFX4_DEBUG, libtqfx4_debug.so): a failed check records
// TQFX4_EDATA with the kernel and `detail`, and the caller then keeps its
// access in bounds instead of faulting. The release build compiles them out.
#ifdef TQFX4_DEBUG
#define TQ_DEBUG_CHECK(cond, status, kernel, detail) \
    ((cond) ? true : (::tq::report((status), TQFX4_EDATA, (kernel), (detail)), false))
#else
#define TQ_DEBUG_CHECK(cond, status, kernel, detail) true
#endif

// Roughly two seconds at the GB300's 2 GHz clock: any mbarrier wait longer
// than this is treated as lost, reported, and abandoned.
constexpr long long kWaitBudgetCycles = 4000000000LL;

__host__ __device__ __forceinline__ int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ int64_t imax64(int64_t a, int64_t b) { return a > b ? a : b; }

__device__ __forceinline__ void report(int *status, int code, int kernel, int detail) {
    if (atomicCAS(status, 0, code) == 0) {
        atomicExch(status + 1, kernel);
        atomicExch(status + 2, detail);
    }
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---- mbarrier ---------------------------------------------------------------

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ uint32_t mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok;
}

// Waits for phase `parity` of `bar` to complete; gives up after `budget`
// cycles (kWaitBudgetCycles by default) and returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, long long budget = kWaitBudgetCycles) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (clock64() - t0 > budget) return false;
    }
}

// One-dimensional bulk copy global -> shared, completing on `bar`
// (dst and src 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// L2 eviction policies for cache hints: weights streamed once per call go
// in as evict-first, data reused by every call (the router) as evict-last.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// bulk_g2s with an L2 cache policy.
__device__ __forceinline__ void bulk_g2s_hint(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                              uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
        "%4;" ::"r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

// 16-byte read-only load with an L2 cache policy.
__device__ __forceinline__ float4 ldg_f4_hint(const float4 *p, uint64_t policy) {
    float4 v;
    asm volatile("ld.global.nc.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p), "l"(policy));
    return v;
}

// Stage `bytes` (a multiple of 8) of global memory starting at the 8-byte
// aligned `src` into the 16-byte aligned shared buffer `dst`, on barrier
// `bar`, issued by one warp. The data lands at dst + (src & 15): its 16-byte
// aligned interior goes by one cp.async.bulk, a leading or trailing 8-byte
// piece by ordinary loads (visible to the warp after the wait plus
// __syncwarp). Returns the offset of the data inside `dst`.
__device__ __forceinline__ uint32_t stage_range(int lane, uint8_t *dst, const uint8_t *src, uint32_t bytes,
                                                uint64_t *bar) {
    const uint32_t o = static_cast<uint32_t>(reinterpret_cast<uintptr_t>(src) & 15u);
    const uint32_t head = (o != 0u && bytes >= 8u) ? 8u : 0u;
    const uint32_t body = ((bytes - head) / 16u) * 16u;
    const uint32_t tail = bytes - head - body;
    if (lane == 0) {
        mbar_arrive_expect_tx(bar, body);
        if (body) bulk_g2s(dst + o + head, src + head, body, bar);
    } else if (lane == 1 && head) {
        *reinterpret_cast<uint2 *>(dst + o) = __ldg(reinterpret_cast<const uint2 *>(src));
    } else if (lane == 2 && tail) {
        *reinterpret_cast<uint2 *>(dst + o + head + body) =
            __ldg(reinterpret_cast<const uint2 *>(src + head + body));
    }
    return o;
}

// ---- integer dot step ----------------------------------------------------------

// d = c + dot(bytes of a as unsigned, bytes of b as signed)
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

// Exact block sums S[r] = sum_j c[r][j] q[j] of one 520-byte block whose code
// bytes start at `codes` (8-byte aligned, shared memory) against one 256-byte
// activation block `qb` (8-byte aligned, shared memory) with sum `bsum`.
// Nibbles hold u = c + 4, so S = sum u q - 4 bsum. Low nibbles (elements
// j) are taken in place; high nibbles (elements j + 128) are kept at 16 u
// and divided out at the end (the sum is an exact multiple of 16).
__device__ __forceinline__ void block_dot(const uint8_t *codes, const uint8_t *qb, int bsum, int S[4]) {
    const uint2 *c2 = reinterpret_cast<const uint2 *>(codes);
    const uint2 *q2 = reinterpret_cast<const uint2 *>(qb);
    int lo[4] = {0, 0, 0, 0}, hi[4] = {0, 0, 0, 0};
#pragma unroll 4
    for (int w = 0; w < 16; ++w) {
        const uint2 qa = q2[w];
        const uint2 qh = q2[16 + w];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const uint2 c = c2[r * 16 + w];
            lo[r] = dp4a_us(c.x & 0x0f0f0f0fu, qa.x, lo[r]);
            lo[r] = dp4a_us(c.y & 0x0f0f0f0fu, qa.y, lo[r]);
            hi[r] = dp4a_us(c.x & 0xf0f0f0f0u, qh.x, hi[r]);
            hi[r] = dp4a_us(c.y & 0xf0f0f0f0u, qh.y, hi[r]);
        }
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) S[r] = lo[r] + (hi[r] >> 4) - 4 * bsum;
}

// Scale of row r (0..3) of the block at `blk` (shared memory), as fp32.
__device__ __forceinline__ float block_scale(const uint8_t *blk, int r) {
    const __half h = *reinterpret_cast<const __half *>(blk + 2 * r);
    return __half2float(h);
}

// Copy one quantized activation vector (q: k bytes, 16-byte aligned; da,
// bsum: k/256 entries) into shared memory with the padded block stride,
// cooperatively by the whole thread block.
__device__ __forceinline__ void load_act_smem(const int8_t *q, const float *da, const int32_t *bsum, int nb,
                                              uint8_t *qs, float *das, int *bss) {
    const int chunks = nb * 16;  // 16-byte chunks
    for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
        const int b = c >> 4, w = c & 15;
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(q) + c);
        uint2 *dst = reinterpret_cast<uint2 *>(qs + b * QS_STRIDE + w * 16);
        dst[0] = make_uint2(v.x, v.y);
        dst[1] = make_uint2(v.z, v.w);
    }
    for (int b = threadIdx.x; b < nb; b += blockDim.x) {
        das[b] = __ldg(da + b);
        bss[b] = __ldg(bsum + b);
    }
}

// Activation vector staged through registers: loads issued early (ahead of
// bulk weight copies in the memory queues), stored to shared memory later.
// Holds nb <= 64 blocks for thread blocks of at least 128 threads.
struct ActRegs {
    uint4 q[8];
    float da;
    int bs;
};

__device__ __forceinline__ void act_load(const int8_t *q, const float *da, const int32_t *bsum, int nb, ActRegs &r) {
    const int chunks = nb * 16;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int c = threadIdx.x + i * blockDim.x;
        if (c < chunks) r.q[i] = __ldcg(reinterpret_cast<const uint4 *>(q) + c);
    }
    if (static_cast<int>(threadIdx.x) < nb) {
        r.da = __ldcg(da + threadIdx.x);
        r.bs = __ldcg(bsum + threadIdx.x);
    }
}

__device__ __forceinline__ void act_store(const ActRegs &r, int nb, uint8_t *qs, float *das, int *bss) {
    const int chunks = nb * 16;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int c = threadIdx.x + i * blockDim.x;
        if (c < chunks) {
            uint2 *dst = reinterpret_cast<uint2 *>(qs + (c >> 4) * QS_STRIDE + (c & 15) * 16);
            dst[0] = make_uint2(r.q[i].x, r.q[i].y);
            dst[1] = make_uint2(r.q[i].z, r.q[i].w);
        }
    }
    if (static_cast<int>(threadIdx.x) < nb) {
        das[threadIdx.x] = r.da;
        bss[threadIdx.x] = r.bs;
    }
}

// ---- inter-kernel ordering ----------------------------------------------------------

// Programmatic dependent launch: wait until the preceding kernel in the
// stream has completed and its writes are visible (a no-op when the kernel
// was launched without the programmatic-serialization attribute).
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Allow the next kernel in the stream (if launched as a programmatic
// dependent) to start launching.
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// atomicAdd with acquire-release semantics at GPU scope: orders this
// thread's earlier writes before the add and later reads after it.
__device__ __forceinline__ int atomic_add_acq_rel(int *p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// First row group of part p when n_rg row groups, in units of rpu, are split
// into `parts` nearly equal parts.
__host__ __device__ inline int64_t part_begin(int64_t n_rg, int rpu, int parts, int p) {
    const int64_t units = (n_rg + rpu - 1) / rpu;
    const int64_t u = units * p / parts;
    return imin64(n_rg, u * rpu);
}

// ---- binary32 helpers with a fixed operation order ------------------------------

// exp in binary32: Cody-Waite reduction z = n ln2 + r (ln2 split as
// 0.693359375 + -2.12194440e-4, the Cephes split), degree-7 Taylor polynomial
// of e^r in Horner form, scaled by 2^n; inputs clamped to [-87, 88]. Every
// step is one correctly rounded binary32 operation (no contraction), so the
// result is reproducible on any IEEE binary32 machine.
__device__ __forceinline__ float tq_expf(float z) {
    if (z != z) return z;
    z = fminf(fmaxf(z, -87.0f), 88.0f);
    const float t = __fmul_rn(z, 1.44269502f);
    const float nf = rintf(t);
    float r = __fsub_rn(z, __fmul_rn(nf, 0.693359375f));
    r = __fsub_rn(r, __fmul_rn(nf, -2.12194440e-4f));
    float p = 1.98412698e-4f;
    p = __fadd_rn(__fmul_rn(p, r), 1.38888889e-3f);
    p = __fadd_rn(__fmul_rn(p, r), 8.33333333e-3f);
    p = __fadd_rn(__fmul_rn(p, r), 4.16666667e-2f);
    p = __fadd_rn(__fmul_rn(p, r), 1.66666667e-1f);
    p = __fadd_rn(__fmul_rn(p, r), 0.5f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    p = __fadd_rn(__fmul_rn(p, r), 1.0f);
    // p * 2^n as one correctly rounded multiplication (n in -126..127, so 2^n
    // is a normal binary32 built from its exponent bits)
    const float two_n = __int_as_float((static_cast<int>(nf) + 127) << 23);
    return __fmul_rn(p, two_n);
}

// h = silu(g) * u = g / (1 + exp(-g)) * u in binary32.
__device__ __forceinline__ float tq_swiglu(float g, float u) {
    const float e = tq_expf(-g);
    const float s = __fdiv_rn(g, __fadd_rn(1.0f, e));
    return __fmul_rn(s, u);
}

// Quantization of one 256-element activation block held by a warp, 8
// consecutive elements per lane (lane l holds elements 8l .. 8l+7):
// da = absmax / 127, q = clamp(round(x * (1/da)), -127, 127), bsum = sum q.
// Returns false if an element is not finite.
__device__ __forceinline__ bool quant_block_warp(const float v[8], uint2 &packed, float &da_out, int &bsum_out) {
    bool finite = true;
    float amax = 0.0f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        finite &= isfinite(v[i]);
        amax = fmaxf(amax, fabsf(v[i]));
    }
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, s));
    const float da = __fdiv_rn(amax, 127.0f);
    const float id = (da != 0.0f) ? __fdiv_rn(1.0f, da) : 0.0f;
    int sum = 0;
    uint32_t w[2] = {0u, 0u};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float t = roundf(__fmul_rn(v[i], id));
        t = fminf(fmaxf(t, -127.0f), 127.0f);
        const int qi = finite ? static_cast<int>(t) : 0;
        sum += qi;
        w[i >> 2] |= (static_cast<uint32_t>(qi) & 0xffu) << (8 * (i & 3));
    }
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
    packed = make_uint2(w[0], w[1]);
    da_out = da;
    bsum_out = sum;
    return __all_sync(0xffffffffu, finite);
}

// e4m3 byte of the integer a in 0..8 (exact): 0, 1 -> 0x38 (2^0), 2 -> 0x40,
// 3 -> 0x44, 4 -> 0x48, 5 -> 0x4A, 6 -> 0x4C, 7 -> 0x4E, 8 -> 0x50, by a
// byte permute over the first eight.
__device__ __forceinline__ uint32_t e4m3_mag(uint32_t a) {
    const uint32_t t = __byte_perm(0x44403800u, 0x4E4C4A48u, a & 7u) & 0xFFu;
    return a == 8u ? 0x50u : t;
}

// Eight int8 activations q as the two e4m3 planes of q = 16 h + l, with
// h = floor((q + 8) / 16) in -8..8 and l in -8..7: bytes of 16 h and of l.
__device__ __forceinline__ void q_planes8(uint2 v, uint2 &hi, uint2 &lo) {
    uint32_t hw[2], lw[2];
#pragma unroll
    for (int w = 0; w < 2; ++w) {
        const uint32_t word = w ? v.y : v.x;
        hw[w] = lw[w] = 0u;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int q = static_cast<int>(word << (24 - 8 * i)) >> 24;  // signed byte i
            const int h = (q + 8) >> 4;                                  // arithmetic shift: floor
            const int l = q - 16 * h;
            const uint32_t ah = static_cast<uint32_t>(h < 0 ? -h : h), al = static_cast<uint32_t>(l < 0 ? -l : l);
            // 16 h: four more in the exponent than h
            const uint32_t hb = ah ? ((e4m3_mag(ah) + 0x20u) | (h < 0 ? 0x80u : 0u)) : 0u;
            const uint32_t lb = e4m3_mag(al) | (l < 0 ? 0x80u : 0u);
            hw[w] |= hb << (8 * i);
            lw[w] |= lb << (8 * i);
        }
    }
    hi = make_uint2(hw[0], hw[1]);
    lo = make_uint2(lw[0], lw[1]);
}

}  // namespace tq
