// Grouped expert GEMM on the 5th-generation tensor cores (tcgen05), the
// contraction of the prefill path: one work item is 128 weight rows (32 row
// groups) of one expert times one chunk of <= TC_CHUNK (token, slot) pairs of
// that expert.
//
// tcgen05.mma has no integer kind on sm_103a, so the integer block sums
// S = sum_j c_j q_j of the dot pass (Sec. 2.2) are formed with kind::f8f6f4 on e4m3 operands
// that hold small dyadic numbers exactly:
//   A  the nibble u = c + 4 (0..8) as the e4m3 byte 0x0u, which is exactly
//      u * 2^-9 (subnormals, and 0x08 = 2^-6), so unpacking a 32-bit word of
//      codes is one mask (four low nibbles) or a shift and a mask (four high
//      nibbles);
//   B  q = 16 h + l with h = floor((q + 8) / 16) in -8..8 and l in -8..7, as
//      two e4m3 planes 16 h and l (both exact).
// Each 256-element block takes 8 K-steps of 32 x 2 planes, accumulated in
// fp32: every product is a multiple of 2^-9 below 2 in magnitude and the
// block sum D = 2^-9 sum u q stays below 2^9, so the accumulator holds it
// exactly (checked against exact integer sums at the extremes); the
// epilogue recovers S = 512 D - 4 bsum with one exact fused multiply-add.
// The accumulator restarts at every block and the epilogue applies the
// fixed float schedule y = y + float(S) * (d * da) block by block, the same
// operations in the same order as the streaming kernels and the oracle.
//
// Operands: A (the unpacked weights) is written by the math warps straight
// into tensor memory with tcgen05.st (thread = row = TMEM lane), so it never
// passes through shared memory; B (the activation planes of the chunk) is
// staged by TMA in the 128-byte swizzled K-major layout.
// Tile rows are ordered r4-major (tile row = 32 * r4 + row group), so that a
// warp (one TMEM lane quadrant) reads the codes of one row of 32 row groups,
// 1040 bytes apart: the 16-byte loads of odd blocks are conflict-free and
// the 8-byte loads of even blocks (codes 8 bytes off 16-byte alignment)
// two-way.
//
// Warp roles (448 threads, one CTA per SM):
//   warps 0-3  unpacking. Warp w serves TMEM lanes 32 w .. + 31 (rows with
//              r4 = w) and writes their codes into A, into the buffer of
//              block b - 2 once that block's MMAs are complete;
//   warps 4-11 epilogue. Warp w serves TMEM lanes 32 (w % 4) .. + 31 and
//              the 16-column pieces (pairs) q, q + 2 and q + 4 of the chunk,
//              q = (w - 4) / 4: per block it reads both plane halves of its
//              pieces of the accumulator, hands the buffer back to the MMAs
//              after its last read, and adds float(S) * (d * da) to the
//              running outputs y, kept in registers; at the end of the item
//              it stores y;
//   warp 12    producer: TMA copies of the raw weight blocks (one box per
//              two blocks of the tile), of the activation planes (one 4-D
//              box per block, into a byte ring where a block takes the
//              chunk's pairs rounded up to 16, times 512 bytes) and a bulk
//              copy of the chunk's block scales;
//   warp 13    TMEM allocation; one thread issues the MMAs (M = 128, K = 32)
//              and two commits per block: one MMA of N = 2 x (pairs rounded up
//              to 16) per K-step, with both planes side by side (the two halves
//              of the accumulator are added by the epilogue, exactly). An MMA
//              takes about the same issue time whatever N, so the chunk
//              (TC_CHUNK pairs) is as wide as two accumulator buffers allow.
//              Each shared-memory access the thread makes stalls its issue,
//              and the tensor pipe with it, so it reads the abort flag only
//              when it actually has to wait.
// TMEM: A in columns [0, 128) (two blocks of 64), two accumulator buffers of
// TC_DCOLS columns from column 128.
// The epilogue uses scalar fp32 operations: the packed f32x2 forms were
// measured to give results that differ from them.
// Every wait is bounded. On a timeout the CTA records the error, all roles
// leave their loops, the producer waits (bounded) for its copies in flight,
// the MMA thread for its MMAs, and TMEM is freed before the CTA exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "tq_launch.h"
#include "tq_moe_common.cuh"

namespace tq {

namespace {

constexpr int TC_ROWS = 128;                   // weight rows per tile = TMEM lanes
constexpr int TC_RG = TC_ROWS / 4;             // row groups per tile
constexpr int TC_CONV_WARPS = 4, TC_EPI_WARPS = 8;
constexpr int TC_MATH_WARPS = TC_CONV_WARPS + TC_EPI_WARPS;  // warps 0-3 unpack A, 4-11 the epilogue
constexpr int TC_SC_STAGES = 4;                // scale ring: runs ahead of the epilogue
constexpr int TC_DW_STAGES = 4;                // weight-scale ring: unpacking -> epilogue
constexpr int TC_THREADS = (TC_MATH_WARPS + 2) * 32;
constexpr int TC_RAW_ROW = 2 * BLOCK_BYTES;    // two blocks of one row group: 1040 bytes
constexpr int TC_RAW_BYTES = 33 * 1024;        // 32 x 1040 bytes, padded
// B, the activation planes of a block: four regions (k-stage ks, plane pl)
// of R rows (pairs) x 128 bytes, R = the chunk's pairs rounded up to 16, so a
// block takes R * 512 bytes (32 KB for 64 pairs), loaded by one 4-D TMA copy.
// Blocks are placed one after another in a byte ring (never split at its
// end), which keeps more small blocks in flight than fixed slots sized for
// the largest chunk.
constexpr int TC_B_ROW = 128;                  // one pair's 128 elements of one plane
constexpr int TC_B_RING = 144 * 1024;          // ring bytes
constexpr int TC_B_SLOTS = 8;                  // full / empty barrier pairs: blocks in flight at most
constexpr int TC_SC_BYTES = 2 * TC_CHUNK * 4;  // da and -4 bsum of the chunk's pairs: 1 KB
constexpr int TC_OFF_RAW = 0;
constexpr int TC_OFF_B = TC_OFF_RAW + 2 * TC_RAW_BYTES;
constexpr int TC_OFF_SC = TC_OFF_B + TC_B_RING;
constexpr int TC_OFF_DW = TC_OFF_SC + TC_SC_STAGES * TC_SC_BYTES;  // [TC_DW_STAGES][128] fp32
constexpr int TC_OFF_BAR = TC_OFF_DW + TC_DW_STAGES * TC_ROWS * 4;
constexpr int TC_NBAR = 11 + 2 * TC_B_SLOTS + 2 * TC_SC_STAGES + 2 * TC_DW_STAGES;  // barriers
constexpr int TC_OFF_BSTART = TC_OFF_BAR + TC_NBAR * 8;  // [TC_B_SLOTS] int64: producer's ring history
constexpr int TC_SMEM = TC_OFF_BSTART + TC_B_SLOTS * 8 + 16 + 1024;  // + TMEM address, abort flag, alignment slack
constexpr int TC_TMEM_COLS = 512;
constexpr uint32_t TC_TMEM_D = 128;            // first accumulator column
constexpr int TC_DCOLS = 192;                  // columns of one accumulator buffer
constexpr int TC_SIDE_MAX = TC_DCOLS / 2;      // pairs up to which both planes go side by side
constexpr int TC_A_COLS = 64;                  // TMEM columns of one block of A (256 bytes per row)

static_assert(TC_OFF_B % 1024 == 0, "swizzled tiles need 1024-byte alignment");
static_assert(TC_B_RING % 2048 == 0 && TC_B_RING >= 2 * TC_CHUNK * 4 * TC_B_ROW, "ring: two blocks of a full chunk");
static_assert(TC_SMEM <= 227 * 1024, "shared memory per CTA");
static_assert(TC_RG * TC_RAW_ROW <= TC_RAW_BYTES, "raw stage too small");
static_assert(TC_CHUNK <= TC_SIDE_MAX && TC_CHUNK % 16 == 0 && TC_CHUNK / 16 <= 6,
              "both planes side by side; at most three 16-column pieces per epilogue warp");
static_assert(TC_TMEM_D + 2 * TC_DCOLS <= TC_TMEM_COLS, "accumulators within the allocation");

// Instruction descriptor of tcgen05.mma kind::f8f6f4: D fp32 (bits 4-5 = 1),
// A and B e4m3 (bits 7-9 = 0, 10-12 = 0), both K-major (bits 15, 16 = 0),
// N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__device__ __forceinline__ uint32_t tc_idesc(int n) {
    return (1u << 4) | (static_cast<uint32_t>(n >> 3) << 17) | (static_cast<uint32_t>(TC_ROWS >> 4) << 24);
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte
// swizzle canonical layout: rows of 128 bytes, 8-row atoms of 1024 bytes
// (stride byte offset), start address advanced by 32 bytes per K = 16 step.
__device__ __forceinline__ uint64_t umma_desc(uint32_t saddr) {
    uint64_t d = static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);  // bits 0-13: start address >> 4
    d |= static_cast<uint64_t>(1) << 16;                           // bits 16-29: leading byte offset (unused)
    d |= static_cast<uint64_t>(1024 >> 4) << 32;                   // bits 32-45: stride byte offset >> 4
    d |= static_cast<uint64_t>(1) << 46;                           // bits 46-47: descriptor version 1
    d |= static_cast<uint64_t>(2) << 61;                           // bits 61-63: 128-byte swizzle
    return d;
}

// D (tmem) [+]= A (tmem) x B (smem descriptor)
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrives on `bar` once every tcgen05 operation issued so far by this thread
// has completed.
__device__ __forceinline__ void tc_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

#define TC_R32(r)                                                                                                    \
    "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),    \
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),   \
        "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),   \
        "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
#define TC_LIST32                                                                                                    \
    "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,"  \
    "%30,%31}"

// TMEM loads and stores of 32 lanes x 16 or 32 columns of 32 bits: each
// thread of the warp its own lane, columns taddr .. taddr + 15 (or 31).
__device__ __forceinline__ void tc_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tc_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%32], " TC_LIST32 ";" ::TC_R32(r), "r"(taddr) : "memory");
}
__device__ __forceinline__ void tc_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%16], "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15};" ::"r"(r[0]),
        "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]),
        "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void tma_4d(void *dst, const CUtensorMap *map, int c0, int c1, int c2, int c3,
                                       uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
        "[%6];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tma_prefetch_map(const CUtensorMap *map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// Activation-plane tensor maps: dims (128 elements, pairs, plane, K / 128),
// map i copies boxes of 16 (i + 1) pairs.
struct TcBMaps {
    CUtensorMap m[TC_CHUNK / 16];
};

__device__ __forceinline__ void tma_2d(void *dst, const CUtensorMap *map, int c0, int c1, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// Placement of the blocks of B in the ring. The producer and the MMA thread
// walk the same blocks with the same sizes, so they compute the same offsets.
struct BRing {
    int64_t pos = 0;  // virtual byte position (grows without wrapping)
    // virtual start of the next block of `bytes` (ring offset = start % ring)
    __device__ __forceinline__ int64_t place(int bytes) {
        const int64_t r = pos % TC_B_RING;
        if (r + bytes > TC_B_RING) pos += TC_B_RING - r;  // do not straddle the end
        const int64_t v = pos;
        pos += bytes;
        return v;
    }
};

struct TcJob {
    int N, nb;   // rows and 256-blocks per row of one expert matrix
    float *Y;    // [P][N] output in pair order
};

// Single-thread bounded wait (producer and MMA threads).
// Polling wait with a suspend-time hint: a thread whose phase is not yet
// complete sleeps in the barrier unit (until the phase completes or the hint
// runs out) instead of re-issuing shared-memory requests, which slow every
// other warp's barrier and shared-memory traffic. Bounded like mbar_wait.
__device__ __forceinline__ uint32_t tc_try_wait_sleep(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)  // hint: 1 ms
        : "memory");
    return ok;
}
__device__ __forceinline__ bool tc_poll(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (true) {
        if (tc_try_wait_sleep(bar, parity)) return true;
        if (clock64() - t0 > kWaitBudgetCycles) return false;
    }
}

// A phase that is already complete costs one try_wait: shared-memory
// accesses of the MMA thread stall it (and with it the tensor pipe), so the
// abort flag is read only when the thread has to wait.
__device__ __forceinline__ bool tc_wait(uint64_t *bar, uint32_t parity, int *abort, int *status, int where) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*reinterpret_cast<volatile int *>(abort)) return false;
    if (tc_poll(bar, parity)) return true;
    *reinterpret_cast<volatile int *>(abort) = 1;
    report(status, TQFX4_ETIMEOUT, K_PREFILL, where);
    return false;
}

// Warp-uniform bounded wait (math warps): all lanes observe the phase, and
// all agree on the outcome so that the .sync.aligned TMEM accesses that
// follow are executed by the whole warp or by none of it. (Every lane polls:
// a single polling lane followed by a confirming wait measured slower.)
__device__ __forceinline__ bool tc_warp_wait(uint64_t *bar, uint32_t parity, int *abort, int *status, int where) {
    const int lane = threadIdx.x & 31;
    if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;  // already complete
    int ab = lane == 0 ? *reinterpret_cast<volatile int *>(abort) : 0;
    ab = __shfl_sync(0xffffffffu, ab, 0);
    if (ab) return false;
    const bool ok = __all_sync(0xffffffffu, tc_poll(bar, parity));
    if (!ok && lane == 0) {
        *reinterpret_cast<volatile int *>(abort) = 1;
        report(status, TQFX4_ETIMEOUT, K_PREFILL, where);
    }
    return ok;
}

// Waits on three barriers: the three try_waits go out back to back, so a set
// of phases that is already complete costs one round trip instead of three;
// otherwise the bounded waits run one after another.
__device__ __forceinline__ bool tc_wait3(uint64_t *b0, uint32_t p0, uint64_t *b1, uint32_t p1, uint64_t *b2,
                                         uint32_t p2, int *abort, int *status, int where) {
    const uint32_t ok = mbar_try_wait(b0, p0) & mbar_try_wait(b1, p1) & mbar_try_wait(b2, p2);
    if (ok) return true;
    return tc_wait(b0, p0, abort, status, where) && tc_wait(b1, p1, abort, status, where) &&
           tc_wait(b2, p2, abort, status, where);
}
__device__ __forceinline__ bool tc_warp_wait3(uint64_t *b0, uint32_t p0, uint64_t *b1, uint32_t p1, uint64_t *b2,
                                              uint32_t p2, int *abort, int *status, int where) {
    const uint32_t ok = mbar_try_wait(b0, p0) & mbar_try_wait(b1, p1) & mbar_try_wait(b2, p2);
    if (__all_sync(0xffffffffu, ok)) return true;
    return tc_warp_wait(b0, p0, abort, status, where) && tc_warp_wait(b1, p1, abort, status, where) &&
           tc_warp_wait(b2, p2, abort, status, where);
}

}  // namespace

__global__ void __launch_bounds__(TC_THREADS, 1)
    tc_gemm_kernel(GroupedArgs a, TcJob j0, TcJob j1, int njobs, const float *__restrict__ scales,
                   const __grid_constant__ CUtensorMap wmap0, const __grid_constant__ CUtensorMap wmap1,
                   const __grid_constant__ TcBMaps bmaps) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + TC_OFF_BAR);
    uint64_t *raw_full = bars, *raw_empty = bars + 2;
    uint64_t *a_full = bars + 4;                        // [2]: the block's codes are in A
    uint64_t *d_full = bars + 6, *d_empty = bars + 8;   // accumulator written / read out
    uint64_t *fin = bars + 10;                          // MMA drain at exit
    uint64_t *b_full = bars + 11, *b_empty = b_full + TC_B_SLOTS;
    uint64_t *sc_full = b_empty + TC_B_SLOTS, *sc_empty = sc_full + TC_SC_STAGES;
    uint64_t *dw_full = sc_empty + TC_SC_STAGES, *dw_empty = dw_full + TC_DW_STAGES;
    float *dw_ring = reinterpret_cast<float *>(smem + TC_OFF_DW);
    int64_t *b_start = reinterpret_cast<int64_t *>(smem + TC_OFF_BSTART);  // virtual starts of the last blocks of B
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(b_start + TC_B_SLOTS);
    int *abort = reinterpret_cast<int *>(tmem_slot + 1);

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&raw_full[i], 1);
            mbar_init(&raw_empty[i], TC_CONV_WARPS);
            mbar_init(&a_full[i], TC_CONV_WARPS);
            mbar_init(&d_full[i], 1);
            mbar_init(&d_empty[i], TC_EPI_WARPS);
        }
        for (int i = 0; i < TC_B_SLOTS; ++i) {
            mbar_init(&b_full[i], 1);
            mbar_init(&b_empty[i], 1);
        }
        for (int i = 0; i < TC_SC_STAGES; ++i) {
            mbar_init(&sc_full[i], 1);
            mbar_init(&sc_empty[i], TC_EPI_WARPS);
        }
        for (int i = 0; i < TC_DW_STAGES; ++i) {
            mbar_init(&dw_full[i], TC_CONV_WARPS);
            mbar_init(&dw_empty[i], TC_EPI_WARPS);
        }
        mbar_init(fin, 1);
        *abort = 0;
    }
    if (warp == TC_MATH_WARPS && lane == 0) {
        tma_prefetch_map(&wmap0);
        tma_prefetch_map(&wmap1);
        for (int i = 0; i < TC_CHUNK / 16; ++i) tma_prefetch_map(&bmaps.m[i]);
    }
    if (warp == TC_MATH_WARPS + 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TC_TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_barrier_init();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(tmem_slot);

    // Items are dealt out over the chunks of more than small_max pairs alone
    // (the work list's tensor-core share, in chunk order), so every CTA gets
    // the same number to within one.
    const int n_tc = __ldcg(a.n_tc);
    const int64_t tiles0 = (j0.N / 4 + TC_RG - 1) / TC_RG;
    const int64_t tiles1 = njobs > 1 ? (j1.N / 4 + TC_RG - 1) / TC_RG : 0;
    const int64_t per_chunk = tiles0 + tiles1;
    const int64_t items = static_cast<int64_t>(n_tc) * per_chunk;

    // All roles walk the same items and blocks, so each keeps identical
    // counts of raw stages and blocks used so far (the ring positions).
    int nraw = 0, nblk = 0;  // a CTA's blocks stay far below 2^31
    BRing bring;
    // Producer: uses issued on each raw stage's full barrier, and the last
    // block of B and of scales issued (for the drain).
    int n_rf0 = 0, n_rf1 = 0, last_b = -1, last_sc = -1;
    for (int64_t w = blockIdx.x; w < items; w += gridDim.x) {
        if (*reinterpret_cast<volatile int *>(abort)) break;
        const int ci = static_cast<int>(w / per_chunk);
        const int4 t = __ldcg(a.tc_list + ci);  // (chunk, expert, first pair, pairs)
        const int chunk = t.x;
        int64_t tl = w - ci * per_chunk;
        const bool second = tl >= tiles0;
        if (second) tl -= tiles0;
        const TcJob &J = second ? j1 : j0;
        const int e = t.y;
        const int pb = t.z;
        const int m = t.w;
        // every role reads the same record, so all skip a bad one alike
        if (!TQ_DEBUG_CHECK(e >= 0 && e < a.E && m >= 1 && m <= TC_CHUNK && pb >= 0 && pb + m <= a.P, a.status,
                            K_PREFILL, ci))
            continue;
        const int n_rg = J.N / 4;
        const int rg0 = static_cast<int>(tl) * TC_RG;
        const int nb = J.nb;
        const int nmma = (m + 15) & ~15;          // pairs rounded up to 16
        // Both planes side by side in one MMA of N = 2 nmma (B rows 0..nmma-1
        // the high plane, then the low one; the epilogue adds the two halves
        // of the accumulator, exactly).
        const int brows = nmma;                   // B rows per (k-stage, plane)
        const int bbytes = 4 * brows * TC_B_ROW;  // one block of B

        if (warp == TC_MATH_WARPS) {
            // ---------------- producer ----------------
            if (lane == 0) {
                const CUtensorMap *wmap = second ? &wmap1 : &wmap0;
                const float *sc = scales + static_cast<int64_t>(chunk) * nb * (2 * TC_CHUNK);
                for (int b = 0; b < nb; ++b) {
                    const int bb = nblk + b;
                    if ((b & 1) == 0) {
                        const int rb = nraw + b / 2;
                        const int rs = static_cast<int>(rb & 1);
                        if (!tc_wait(&raw_empty[rs], static_cast<uint32_t>(((rb >> 1) & 1) ^ 1), abort, a.status, 1))
                            break;
                        mbar_arrive_expect_tx(&raw_full[rs], TC_RG * TC_RAW_ROW);
                        tma_2d(smem + TC_OFF_RAW + rs * TC_RAW_BYTES, wmap, (b / 2) * (TC_RAW_ROW / 8),
                               e * n_rg + rg0, &raw_full[rs]);
                        if (rs) ++n_rf1; else ++n_rf0;
                    }
                    // B: first wait until the blocks whose bytes this one reuses
                    // are consumed: the latest block that starts less than one
                    // ring before this block's end, and at least the previous
                    // user of this barrier pair (in-order consumption makes
                    // the latest of them sufficient)
                    const int64_t v = bring.place(bbytes);
                    int need = bb - TC_B_SLOTS;
                    for (int j = bb - 1; j > need && j >= 0; --j)
                        if (b_start[j % TC_B_SLOTS] < v + bbytes - TC_B_RING) {
                            need = j;
                            break;
                        }
                    if (need >= 0 && !tc_wait(&b_empty[need % TC_B_SLOTS],
                                              static_cast<uint32_t>((need / TC_B_SLOTS) & 1), abort, a.status, 2))
                        break;
                    const int bs = static_cast<int>(bb % TC_B_SLOTS);
                    b_start[bs] = v;
                    mbar_arrive_expect_tx(&b_full[bs], bbytes);
                    // both k-stages, both planes, brows pairs: [ks][pl][pair][128]
                    tma_4d(smem + TC_OFF_B + v % TC_B_RING, &bmaps.m[brows / 16 - 1], 0, pb, 0, 2 * b, &b_full[bs]);
                    last_b = bb;
                    const int ss = static_cast<int>(bb % TC_SC_STAGES);
                    if (!tc_wait(&sc_empty[ss], static_cast<uint32_t>(((bb / TC_SC_STAGES) & 1) ^ 1), abort, a.status, 3))
                        break;
                    mbar_arrive_expect_tx(&sc_full[ss], TC_SC_BYTES);
                    bulk_g2s(smem + TC_OFF_SC + ss * TC_SC_BYTES, sc + b * (2 * TC_CHUNK), TC_SC_BYTES, &sc_full[ss]);
                    last_sc = bb;
                }
            }
            __syncwarp();
        } else if (warp == TC_MATH_WARPS + 1) {
            // ---------------- MMA issuer ----------------
            if (lane == 0) {
                const uint32_t idesc = tc_idesc(2 * nmma);
                // B descriptors: ring start; the others differ by constant
                // byte offsets (>> 4) in the start-address field
                const uint64_t bdesc0 = umma_desc(smem_u32(smem + TC_OFF_B));
                const int region = brows * TC_B_ROW;  // one (k-stage, plane) of B
                for (int b = 0; b < nb; ++b) {
                    const int bb = nblk + b;
                    const int bs = static_cast<int>(bb & 1);
                    const int64_t v = bring.place(bbytes);
                    const int slot = static_cast<int>(bb % TC_B_SLOTS);
                    // the epilogue has read out block bb - 2 (this accumulator
                    // buffer), the codes are in A and B has landed
                    if (!tc_wait3(&d_empty[bs], static_cast<uint32_t>(((bb >> 1) & 1) ^ 1), &a_full[bs],
                                  static_cast<uint32_t>((bb >> 1) & 1), &b_full[slot],
                                  static_cast<uint32_t>((bb / TC_B_SLOTS) & 1), abort, a.status, 4))
                        break;
                    tc_fence_after();
                    const uint32_t d_tmem = tmem + TC_TMEM_D + bs * TC_DCOLS;
                    const uint32_t a_tmem = tmem + bs * TC_A_COLS;
                    const uint64_t bd = bdesc0 + static_cast<uint64_t>((v % TC_B_RING) >> 4);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)  // 32-element step: A columns 8 kk .. 8 kk + 7
                        tc_mma_ts(d_tmem, a_tmem + 8 * kk, bd + (((kk >> 2) * 2 * region + (kk & 3) * 32) >> 4),
                                  idesc, kk != 0 ? 1u : 0u);
                    tc_commit(&b_empty[slot]);
                    tc_commit(&d_full[bs]);
                }
            }
            __syncwarp();
        } else {
            // ---------------- math warps ----------------
            const int r4 = warp & 3;                   // TMEM lane quadrant = row r4 of each row group
            const int rgl = lane;                      // row group within the tile
            const uint32_t lane_base = static_cast<uint32_t>(r4 * 32) << 16;
            bool ok = true;
            if (warp < TC_CONV_WARPS) {
                // ---- unpacking: codes of row (rgl, r4) into A, one block at a time
                for (int b = 0; b < nb && ok; ++b) {
                    const int bb = nblk + b;
                    const int as = static_cast<int>(bb & 1);
                    const int rb = nraw + b / 2;
                    const int rs = static_cast<int>(rb & 1);
                    // the raw blocks (for odd b the phase its even partner already
                    // waited for), a free slot of the weight-scale ring, and the A
                    // buffer, free once the MMAs of block bb - 2 are complete
                    // (d_full of that block; block bb's own MMAs need this block's
                    // codes, so the phase cannot have moved on)
                    const int ds = static_cast<int>(bb % TC_DW_STAGES);
                    if (!tc_warp_wait3(&raw_full[rs], static_cast<uint32_t>((rb >> 1) & 1), &dw_empty[ds],
                                       static_cast<uint32_t>(((bb / TC_DW_STAGES) & 1) ^ 1), &d_full[as],
                                       static_cast<uint32_t>(((bb >> 1) & 1) ^ 1), abort, a.status, 7)) {
                        ok = false;
                        break;
                    }
                    const uint8_t *blk = smem + TC_OFF_RAW + rs * TC_RAW_BYTES + rgl * TC_RAW_ROW + (b & 1) * BLOCK_BYTES;
                    const uint8_t *codes = blk + CODE_OFS + ROW_BYTES * r4;
                    // this row's weight scale, handed to the epilogue
                    dw_ring[ds * TC_ROWS + r4 * 32 + rgl] = block_scale(blk, r4);
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&dw_full[ds]);
                    tc_fence_after();
                    // A columns: element j (< 128) is byte j % 4 of column j / 4,
                    // element 128 + j of column 32 + j / 4: code word i gives
                    // column i (its low nibbles) and column 32 + i (its high
                    // ones). Two passes of 16 words keep the registers low.
                    const uint32_t acol = tmem + lane_base + as * TC_A_COLS;
                    uint32_t hi[32];
#pragma unroll
                    for (int pass = 0; pass < 2; ++pass) {
                        uint32_t x[16];
                        if (b & 1) {  // 16-byte aligned codes
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const uint4 v = *reinterpret_cast<const uint4 *>(codes + 64 * pass + 16 * i);
                                x[4 * i] = v.x, x[4 * i + 1] = v.y, x[4 * i + 2] = v.z, x[4 * i + 3] = v.w;
                            }
                        } else {
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const uint2 v = *reinterpret_cast<const uint2 *>(codes + 64 * pass + 8 * i);
                                x[2 * i] = v.x, x[2 * i + 1] = v.y;
                            }
                        }
                        uint32_t lo[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            lo[i] = x[i] & 0x0f0f0f0fu;
                            hi[16 * pass + i] = (x[i] >> 4) & 0x0f0f0f0fu;
                        }
                        tc_st16(acol + 16 * pass, lo);
                    }
                    tc_st32(acol + 32, hi);
                    tc_wait_st();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(&a_full[as]);
                        if (b & 1) mbar_arrive(&raw_empty[rs]);
                    }
                }
            } else {
                // ---- epilogue: y (registers) += float(S) * (d * da), block after
                // block; two warps per lane quadrant, warp q2 takes the 16-column
                // pieces (pairs) q2, q2 + 2 and q2 + 4
                const int q2 = (warp - TC_CONV_WARPS) >> 2;
                const int npc = (m + 15) >> 4;  // pieces of the chunk (at most 6)
                const int mine = npc > q2 ? (npc - q2 + 1) / 2 : 0;  // this warp's pieces (0..3)
                float y[3][16];
#pragma unroll
                for (int k = 0; k < 3; ++k)
#pragma unroll
                    for (int i = 0; i < 16; ++i) y[k][i] = 0.0f;
                for (int b = 0; b < nb && ok; ++b) {
                    const int bb = nblk + b;
                    const int bs = static_cast<int>(bb & 1);
                    const int ss = static_cast<int>(bb % TC_SC_STAGES);
                    const int ds = static_cast<int>(bb % TC_DW_STAGES);
                    if (!tc_warp_wait3(&d_full[bs], static_cast<uint32_t>((bb >> 1) & 1), &sc_full[ss],
                                       static_cast<uint32_t>((bb / TC_SC_STAGES) & 1), &dw_full[ds],
                                       static_cast<uint32_t>((bb / TC_DW_STAGES) & 1), abort, a.status, 9)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const float dw = dw_ring[ds * TC_ROWS + r4 * 32 + rgl];
                    const float *sc = reinterpret_cast<const float *>(smem + TC_OFF_SC + ss * TC_SC_BYTES);
                    const uint32_t dcol = tmem + lane_base + TC_TMEM_D + bs * TC_DCOLS;
                    if (mine == 0) {  // nothing to read: hand the buffer back at once
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&d_empty[bs]);
                    }
#pragma unroll
                    for (int k = 0; k < 3; ++k) {
                        if (k >= mine) break;
                        const int pc = q2 + 2 * k;
                        // piece pc's accumulator columns, both plane halves; after
                        // the warp's last read of the buffer it goes back to the MMAs
                        uint32_t hv[16], lv[16];
                        tc_ld16(dcol + 16 * pc, hv);
                        tc_ld16(dcol + nmma + 16 * pc, lv);
                        tc_wait_ld();
                        if (k == mine - 1) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&d_empty[bs]);
                        }
#pragma unroll
                        for (int n4 = 0; n4 < 4; ++n4) {
                            const float4 da = *reinterpret_cast<const float4 *>(sc + 16 * pc + 4 * n4);
                            const float4 bi = *reinterpret_cast<const float4 *>(sc + TC_CHUNK + 16 * pc + 4 * n4);
                            const float dav[4] = {da.x, da.y, da.z, da.w}, biv[4] = {bi.x, bi.y, bi.z, bi.w};
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int i = 4 * n4 + q;
                                // D = high-plane half + low-plane half (exact); S = 512 D - 4 bsum,
                                // exact (integers below 2^18)
                                const float D = __fadd_rn(__uint_as_float(hv[i]), __uint_as_float(lv[i]));
                                const float S = __fmaf_rn(512.0f, D, biv[q]);
                                y[k][i] = __fadd_rn(y[k][i], __fmul_rn(S, __fmul_rn(dw, dav[q])));
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(&sc_empty[ss]);
                        mbar_arrive(&dw_empty[ds]);
                    }
                }
                if (ok && rg0 + rgl < n_rg) {
                    // row (rg0 + rgl, r4) of the pairs' outputs: pair n at yr[n N]
                    float *yr = J.Y + static_cast<int64_t>(pb) * J.N + (static_cast<int64_t>(rg0 + rgl) * 4 + r4);
                    const int N = J.N;
#pragma unroll
                    for (int k = 0; k < 3; ++k) {
                        if (k >= mine) break;
                        const int n0 = 16 * (q2 + 2 * k);
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            if (n0 + i < m) yr[(n0 + i) * N] = y[k][i];
                    }
                }
            }
        }
        nraw += (nb + 1) / 2;
        nblk += nb;
    }

    // Drain: nothing asynchronous may still target this CTA's shared memory
    // or TMEM when it exits. After a normal run these waits return at once.
    if (warp == TC_MATH_WARPS && lane == 0) {
        if (n_rf0 > 0) mbar_wait(&raw_full[0], static_cast<uint32_t>((n_rf0 - 1) & 1));
        if (n_rf1 > 0) mbar_wait(&raw_full[1], static_cast<uint32_t>((n_rf1 - 1) & 1));
        // the last TC_B_SLOTS blocks of B, oldest first
        for (int u = max(0, last_b - TC_B_SLOTS + 1); u <= last_b; ++u)
            mbar_wait(&b_full[u % TC_B_SLOTS], static_cast<uint32_t>((u / TC_B_SLOTS) & 1));
        // the last TC_SC_STAGES scale copies, oldest first
        for (int u = max(0, last_sc - TC_SC_STAGES + 1); u <= last_sc; ++u)
            mbar_wait(&sc_full[u % TC_SC_STAGES], static_cast<uint32_t>((u / TC_SC_STAGES) & 1));
    }
    if (warp == TC_MATH_WARPS + 1 && lane == 0) {
        tc_commit(fin);
        mbar_wait(fin, 0);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TC_MATH_WARPS + 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_TMEM_COLS) : "memory");
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode_tc = nullptr;

cudaError_t encode_tiled(CUtensorMap *m, CUtensorMapDataType dt, int rank, const void *base, const cuuint64_t *dims,
                         const cuuint64_t *strides, const cuuint32_t *box, CUtensorMapSwizzle sw) {
    if (!g_encode_tc) {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess) return e;
        if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
        g_encode_tc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = g_encode_tc(m, dt, rank, const_cast<void *>(base), dims, strides, box, estr,
                             CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t encode_2d(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t d0, uint64_t d1,
                      uint64_t stride1, uint32_t b0, uint32_t b1, CUtensorMapSwizzle sw) {
    const cuuint64_t dims[2] = {d0, d1};
    const cuuint64_t strides[1] = {stride1};
    const cuuint32_t box[2] = {b0, b1};
    return encode_tiled(m, dt, 2, base, dims, strides, box, sw);
}

}  // namespace

int tc_gemm_smem() { return TC_SMEM; }

// One grouped projection pass on tensor cores: gate and up into g and u
// (down = false), or down into o (down = true). Needs the e4m3 activation
// planes (xq or hq) and the chunk-aligned scales (xs or hs).
cudaError_t launch_tc_gemm(const GroupedArgs &a, bool down, cudaStream_t st) {
    static unsigned char set_tc[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(tc_gemm_kernel), set_tc);
    if (e != cudaSuccess) return e;
    const int nb = down ? a.nbi : a.nbh;
    const int N = down ? a.H : a.I;
    const int K = nb * QK;
    const uint8_t *m0 = down ? a.down : a.gate;
    const uint8_t *m1 = down ? a.down : a.up;
    // weights: one row per row group (E * N / 4 rows of nb * 520 bytes) as
    // 8-byte elements; boxes of two blocks x 32 row groups
    const uint64_t wd0 = static_cast<uint64_t>(nb) * BLOCK_BYTES / 8;
    const uint64_t wd1 = static_cast<uint64_t>(a.E) * (N / 4);
    const uint64_t wstride = static_cast<uint64_t>(nb) * BLOCK_BYTES;
    CUtensorMap w0, w1;
    if ((e = encode_2d(&w0, CU_TENSOR_MAP_DATA_TYPE_UINT64, m0, wd0, wd1, wstride, TC_RAW_ROW / 8, TC_RG,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) != cudaSuccess)
        return e;
    if ((e = encode_2d(&w1, CU_TENSOR_MAP_DATA_TYPE_UINT64, m1, wd0, wd1, wstride, TC_RAW_ROW / 8, TC_RG,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) != cudaSuccess)
        return e;
    // activation planes: [2][P][K] bytes (16 h, then l, as e4m3), seen as
    // (128 elements, P pairs, 2 planes, K / 128); boxes of (128, 16 (i + 1),
    // 2, 2): one block of both planes for up to 16 (i + 1) pairs, laid out
    // [k-stage][plane][pair][128 bytes], 128-byte swizzled
    const uint8_t *act = down ? a.hq : a.xq;
    TcBMaps bm;
    for (int i = 0; i < TC_CHUNK / 16; ++i) {
        const cuuint64_t dims[4] = {128, static_cast<cuuint64_t>(a.P), 2, static_cast<cuuint64_t>(K / 128)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(a.P) * K, 128};
        const cuuint32_t box[4] = {128, static_cast<cuuint32_t>(16 * (i + 1)), 2, 2};
        if ((e = encode_tiled(&bm.m[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, act, dims, strides, box,
                              CU_TENSOR_MAP_SWIZZLE_128B)) != cudaSuccess)
            return e;
    }
    const TcJob j0{N, nb, down ? a.o : a.g};
    const TcJob j1{N, nb, down ? a.o : a.u};
    tc_gemm_kernel<<<num_sms(), TC_THREADS, TC_SMEM, st>>>(a, j0, j1, down ? 1 : 2, down ? a.hs : a.xs, w0, w1, bm);
    return cudaGetLastError();
}

}  // namespace tq
