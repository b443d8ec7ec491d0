// Grouped MoE, experts with few tokens: the chunks of at most SG_MAX
// (token, slot) pairs of the grouped work list (batched decode leaves many
// experts with one to four), which the tensor-core contraction would run at
// its full per-block cost. Here each such expert's matrix is streamed once
// and every lane forms the exact block sums of two rows against each of
// the chunk's activations (the nibble masks shared between them), then the
// fixed float schedule y = y + float(S) * (d * da) over the blocks in order,
// so the outputs are the oracle's bit for bit, as on the other paths.
//
// Work: each CTA first lists the small chunks in ascending chunk order (the
// same list in every CTA, so that item numbers name the same work
// everywhere and the items spread evenly over the CTAs), then takes items
// (chunk, matrix, range of units);
// a unit is 16 blocks (8320 bytes, 16 / L whole row groups for L = k / 256
// blocks a row, L dividing 16). A CTA's warps issue their first copies of
// the range, then stage the chunk's activations ([16-byte word][block] per
// pair, so that lanes on different blocks read different banks) while the
// copies fly, then stream the range's units through two-slot rings; in a
// unit, lane l takes rows 2 (l / 16), 2 (l / 16) + 1 of the unit's block
// l % 16 (row group (l % 16) / L, block (l % 16) % L).
#include "tq_launch.h"
#include "tq_moe_common.cuh"

namespace tq {

namespace {

constexpr int SG_MAX = 4;          // pairs a chunk may hold to take this path
// 12 warps of two-slot rings: the pass is bound by instruction latency, so
// more warps (issue parallelism) beat deeper rings (8 x 3 and 6 x 4 measured
// 2 % and 11 % slower on the 64-token batch)
constexpr int SG_WARPS = 12, SG_SLOTS = 2, SG_UNIT = 16;  // blocks a unit
constexpr int SG_UBYTES = SG_UNIT * BLOCK_BYTES;           // 8320
constexpr int SG_RANGE = 64;       // units an item
constexpr int SG_LIST = 640;        // small chunks a launch can take (the work list's capacity at most)

struct SgJob {
    const uint8_t *mat[2];  // stacked expert matrices (gate, up; or down twice)
    int64_t mat_bytes;
    float *y[2];            // outputs [P][N] (pair order)
    int n_mat, N, K;        // matrices, rows, columns
    int down;               // activation: 0 the tokens' x (token order), 1 the pairs' h
};

__host__ __device__ inline int sg_act_bytes(int K) {
    const int L = K / QK;
    return SG_MAX * (((K + 8 * L) + 127) / 128) * 128;
}
// a warp: the ring's slots, the block terms [pair][row][block] of one unit
// (64 per pair: 64 / L rows of L blocks), the ring's barriers
constexpr int SG_TB_BYTES = SG_MAX * 4 * SG_UNIT * 4;
__host__ __device__ inline int sg_warp_bytes() { return SG_SLOTS * SG_UBYTES + SG_TB_BYTES + 32; }

// S (two rows: codes, codes + 128 bytes) against the m activations of the
// chunk; qv[j] points at the lane's block of activation j, whose 16-byte
// words lie L apart.
__device__ __forceinline__ void sg_dot(const uint2 *codes, const uint4 *const (&qv)[SG_MAX], int L, int m,
                                       int (&S)[SG_MAX][2]) {
    int lo[SG_MAX][2], hi[SG_MAX][2];
#pragma unroll
    for (int j = 0; j < SG_MAX; ++j) lo[j][0] = lo[j][1] = hi[j][0] = hi[j][1] = 0;
#pragma unroll 2
    for (int i = 0; i < 8; ++i) {
        uint32_t cl[2][4], ch[2][4];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const uint2 c0 = codes[16 * r + 2 * i], c1 = codes[16 * r + 2 * i + 1];
            const uint32_t w[4] = {c0.x, c0.y, c1.x, c1.y};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                cl[r][e] = w[e] & 0x0f0f0f0fu;
                ch[r][e] = w[e] & 0xf0f0f0f0u;
            }
        }
#pragma unroll
        for (int j = 0; j < SG_MAX; ++j) {
            if (j >= m) break;
            const uint4 ql = qv[j][i * L], qh = qv[j][(8 + i) * L];
            const uint32_t qlw[4] = {ql.x, ql.y, ql.z, ql.w}, qhw[4] = {qh.x, qh.y, qh.z, qh.w};
#pragma unroll
            for (int r = 0; r < 2; ++r)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    lo[j][r] = dp4a_us(cl[r][e], qlw[e], lo[j][r]);
                    hi[j][r] = dp4a_us(ch[r][e], qhw[e], hi[j][r]);
                }
        }
    }
#pragma unroll
    for (int j = 0; j < SG_MAX; ++j) {
        S[j][0] = lo[j][0] + (hi[j][0] >> 4);
        S[j][1] = lo[j][1] + (hi[j][1] >> 4);
    }
}

__global__ void __launch_bounds__(SG_WARPS * 32) small_groups_kernel(GroupedArgs a, SgJob J) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = J.K, L = K / QK, N = J.N;
    const int unit_rg = SG_UNIT / L;                 // row groups a unit
    const int rows = 4 * unit_rg;                    // rows a unit
    const int units = N / rows;                      // units a matrix
    const int ranges = (units + SG_RANGE - 1) / SG_RANGE;
    const int act_one = sg_act_bytes(K) / SG_MAX;    // bytes of one staged activation
    uint8_t *wbase = smem + sg_act_bytes(K) + warp * sg_warp_bytes();
    uint8_t *slots = wbase;
    float *tb = reinterpret_cast<float *>(wbase + SG_SLOTS * SG_UBYTES);  // [pair][row][block]
    uint64_t *bars = reinterpret_cast<uint64_t *>(wbase + SG_SLOTS * SG_UBYTES + SG_TB_BYTES);
    int *list = reinterpret_cast<int *>(smem + sg_act_bytes(K) + SG_WARPS * sg_warp_bytes());
    __shared__ int abort_all, n_small;
    if (threadIdx.x == 0) abort_all = n_small = 0;
    if (lane == 0)
        for (int i = 0; i < SG_SLOTS; ++i) mbar_init(&bars[i], 1);
    fence_barrier_init();
    __syncthreads();
    // the chunks this pass takes, in ascending chunk order: every CTA must
    // build the same list, since item w means the same (chunk, matrix,
    // range) to all of them (warp 0 compacts 32 chunks at a time)
    const int n_chunks = __ldcg(a.n_chunks);
    if (warp == 0) {
        int base = 0;
        for (int c0 = 0; c0 < n_chunks; c0 += 32) {
            const int c = c0 + lane;
            const int m = c < n_chunks ? __ldcg(a.chunk_len + c) : 0;
            const bool small = m > 0 && m <= SG_MAX;
            const uint32_t bal = __ballot_sync(0xffffffffu, small);
            const int i = base + __popc(bal & ((1u << lane) - 1u));
            if (small && i < SG_LIST) list[i] = c;
            base += __popc(bal);
        }
        if (lane == 0) n_small = base;
    }
    __syncthreads();
    const int ns = min(n_small, SG_LIST);
    const int items = ns * J.n_mat * ranges;
    const uint64_t policy = l2_policy_evict_first();
    const int ub = lane & 15, rp = lane >> 4;  // the lane's block of a unit and row pair
    const int rgl = ub / L, b = ub - rgl * L;
    int s = 0, ph = 0;  // this warp's ring position, kept across items
    bool dead = false;  // a copy of this warp's never arrived
    for (int w = blockIdx.x; w < items; w += gridDim.x) {
        const int c = list[w / (J.n_mat * ranges)];
        const int rem = w % (J.n_mat * ranges);
        const int mi = rem / ranges, rng = rem - mi * ranges;
        const int m = __ldcg(a.chunk_len + c);
        const int e = __ldcg(a.chunk_expert + c), pb = __ldcg(a.chunk_begin + c);
        const uint8_t *mat = (mi ? J.mat[1] : J.mat[0]) + static_cast<int64_t>(e) * J.mat_bytes;
        float *Y = mi ? J.y[1] : J.y[0];  // selects: a dynamic index would copy the parameter array to the stack
        const int u0 = rng * SG_RANGE, u1 = min(units, u0 + SG_RANGE);
        const int first = u0 + warp;
        const int my = first < u1 ? (u1 - first + SG_WARPS - 1) / SG_WARPS : 0;
        auto issue = [&](int k, int slot) {  // the warp's k-th unit of the range
            if (lane == 0) {
                mbar_arrive_expect_tx(&bars[slot], SG_UBYTES);
                bulk_g2s_hint(slots + slot * SG_UBYTES, mat + static_cast<int64_t>(first + k * SG_WARPS) * SG_UBYTES,
                              SG_UBYTES, &bars[slot], policy);
            }
        };
        // the weights first: their copies overlap the staging of the activations
        fence_proxy_async_smem();  // the slots' last generic reads come before the refills
        if (!dead)
            for (int k = 0; k < SG_SLOTS && k < my; ++k) issue(k, (s + k) % SG_SLOTS);
        __syncthreads();  // the previous item's reads of the staged activations are done
        if (abort_all) {  // a copy never arrived; every warp leaves here together, after its own copies
            for (int k = 0; k < SG_SLOTS && k < my && !dead; ++k) {
                const int sk = (s + k) % SG_SLOTS;
                mbar_wait(&bars[sk], static_cast<uint32_t>(s + k >= SG_SLOTS ? ph ^ 1 : ph));
            }
            return;
        }
        const int tot = m * 16 * L;
#pragma unroll 4
        for (int idx = threadIdx.x; idx < tot; idx += blockDim.x) {
            const int j = idx / (16 * L), r = idx - j * 16 * L;
            const int bb = r % L, wd = r / L;
            const int64_t p = pb + j;
            const int8_t *row = J.down ? a.qh + p * K : a.qx + static_cast<int64_t>(__ldcg(a.pair_token + p)) * K;
            reinterpret_cast<uint4 *>(smem + j * act_one)[r] =
                __ldcg(reinterpret_cast<const uint4 *>(row + bb * QK + 16 * wd));
        }
        for (int idx = threadIdx.x; idx < m * L; idx += blockDim.x) {
            const int j = idx / L, bb = idx - j * L;
            const int64_t p = pb + j;
            const int64_t sb = J.down ? p * L + bb : static_cast<int64_t>(__ldcg(a.pair_token + p)) * L + bb;
            float *das = reinterpret_cast<float *>(smem + j * act_one + K);
            das[bb] = __ldcg((J.down ? a.dh : a.dx) + sb);
            reinterpret_cast<int *>(das + L)[bb] = __ldcg((J.down ? a.bh : a.bx) + sb);
        }
        __syncthreads();
        const uint4 *qv[SG_MAX];
        float da[SG_MAX];
        int bs[SG_MAX];
#pragma unroll
        for (int j = 0; j < SG_MAX; ++j) {
            const uint8_t *base = smem + (j < m ? j : 0) * act_one;
            qv[j] = reinterpret_cast<const uint4 *>(base) + b;
            da[j] = reinterpret_cast<const float *>(base + K)[b];
            bs[j] = reinterpret_cast<const int *>(base + K + 4 * L)[b];
        }
        for (int k = 0; k < my; ++k) {
            if (!__all_sync(0xffffffffu, mbar_wait(&bars[s], static_cast<uint32_t>(ph)))) {
                if (lane == 0) {
                    report(a.status, TQFX4_ETIMEOUT, J.down ? K_GDOWN : K_GGATEUP, c);
                    abort_all = 1;
                }
                // the later copies of the range may still be in flight: wait for them (bounded) before leaving
                for (int k2 = k + 1; k2 < my && k2 < k + SG_SLOTS; ++k2) {
                    const int sk = (s + k2 - k) % SG_SLOTS;
                    mbar_wait(&bars[sk], static_cast<uint32_t>(s + k2 - k >= SG_SLOTS ? ph ^ 1 : ph));
                }
                dead = true;
                break;
            }
            const uint8_t *blk = slots + s * SG_UBYTES + ub * BLOCK_BYTES;
            int S[SG_MAX][2];
            sg_dot(reinterpret_cast<const uint2 *>(blk + CODE_OFS + 256 * rp), qv, L, m, S);
            const float d0 = block_scale(blk, 2 * rp), d1 = block_scale(blk, 2 * rp + 1);
#pragma unroll
            for (int j = 0; j < SG_MAX; ++j) {
                if (j >= m) break;
                float *t = tb + (j * rows + rgl * 4 + 2 * rp) * L + b;
                t[0] = __fmul_rn(static_cast<float>(S[j][0] - 4 * bs[j]), __fmul_rn(d0, da[j]));
                t[L] = __fmul_rn(static_cast<float>(S[j][1] - 4 * bs[j]), __fmul_rn(d1, da[j]));
            }
            __syncwarp();
            // the slot is read: refill it with the unit SG_SLOTS ahead
            if (k + SG_SLOTS < my) {
                fence_proxy_async_smem();
                issue(k + SG_SLOTS, s);
            }
            const int urow0 = (first + k * SG_WARPS) * rows;  // first matrix row of the unit
            for (int t = lane; t < m * rows; t += 32) {
                const float *row = tb + t * L;
                float v[SG_UNIT];
#pragma unroll
                for (int bb = 0; bb < SG_UNIT; ++bb) v[bb] = bb < L ? row[bb] : 0.0f;
                float acc = 0.0f;  // the blocks in order
#pragma unroll
                for (int bb = 0; bb < SG_UNIT; ++bb)
                    if (bb < L) acc = __fadd_rn(acc, v[bb]);
                const int j = t / rows;
                Y[static_cast<int64_t>(pb + j) * N + urow0 + (t - j * rows)] = acc;
            }
            __syncwarp();
            if (++s == SG_SLOTS) {
                s = 0;
                ph ^= 1;
            }
        }
    }
}

}  // namespace

namespace {

SgJob sg_job(const GroupedArgs &a, bool down) {
    SgJob J{};
    if (down) {
        J.mat[0] = J.mat[1] = a.down;
        J.mat_bytes = a.mb_d;
        J.y[0] = J.y[1] = a.o;
        J.n_mat = 1;
        J.N = a.H;
        J.K = a.I;
    } else {
        J.mat[0] = a.gate;
        J.mat[1] = a.up;
        J.mat_bytes = a.mb_gu;
        J.y[0] = a.g;
        J.y[1] = a.u;
        J.n_mat = 2;
        J.N = a.I;
        J.K = a.H;
    }
    J.down = down ? 1 : 0;
    return J;
}

int sg_smem(int K) { return sg_act_bytes(K) + SG_WARPS * sg_warp_bytes() + SG_LIST * 4; }

// A unit must be whole row groups (L divides 16, the rows a multiple of
// the unit's), its copies 16-byte aligned, the shared memory within bounds.
bool sg_fits(const SgJob &J) {
    if (J.K % QK != 0 || SG_UNIT % (J.K / QK) != 0) return false;
    const int unit_rg = SG_UNIT / (J.K / QK);
    if (J.N % 4 != 0 || (J.N / 4) % unit_rg != 0) return false;
    if (J.mat_bytes % 16 != 0) return false;
    for (int i = 0; i < J.n_mat; ++i)
        if (reinterpret_cast<uintptr_t>(J.mat[i]) % 16 != 0) return false;
    return sg_smem(J.K) + 256 <= max_smem_optin();  // with the static shared memory
}

}  // namespace

int small_groups_max(const GroupedArgs &a) {
    if (a.max_chunks > SG_LIST) return 0;
    return (sg_fits(sg_job(a, false)) && sg_fits(sg_job(a, true))) ? SG_MAX : 0;
}

cudaError_t launch_small_groups(const GroupedArgs &a, bool down, cudaStream_t st) {
    const SgJob J = sg_job(a, down);
    if (!sg_fits(J)) return cudaErrorInvalidValue;
    static unsigned char set[64];
    cudaError_t e = allow_max_smem(reinterpret_cast<const void *>(small_groups_kernel), set);
    if (e != cudaSuccess) return e;
    small_groups_kernel<<<num_sms(), SG_WARPS * 32, sg_smem(J.K), st>>>(a, J);
    return cudaGetLastError();
}

}  // namespace tq
