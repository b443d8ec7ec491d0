// tqfx4_pack and tqfx4_quantize_act kernels (Tied Trit-Planes, Sec. 2.1 and
// 2.2): writing 520-byte tq2_0_fx4 blocks from trit planes or fp32 weights
// (round-to-nearest, or the tied alternating solver), and per-256-block int8
// activation quantization.
#include "tq_common.cuh"
#include "tq_launch.h"

namespace tq {

// One warp per (row group, block): four rows of 256 elements become one
// 520-byte block. Lane l handles elements 8l .. 8l+7 of each row; lanes
// 0..15 own the low nibbles (elements 0..127) and receive the high nibbles
// (elements 128..255) from lanes 16..31.
template <int SRC>
__global__ void __launch_bounds__(256) pack_kernel(const void *a, const int8_t *t2, const uint16_t *scales,
                                                   int64_t n_rg, int nb, int64_t k, uint8_t *blocks,
                                                   int *status) {
    const int lane = threadIdx.x & 31;
    const int64_t unit = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (unit >= n_rg * nb) return;
    const int64_t rg = unit / nb;
    const int b = static_cast<int>(unit - rg * nb);
    uint8_t *blk = blocks + unit * BLOCK_BYTES;
    uint16_t dbits[4];
    bool bad = false;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int64_t row = rg * 4 + r;
        const int64_t e0 = row * k + static_cast<int64_t>(b) * QK + 8 * lane;
        uint32_t u[2] = {0u, 0u};
        if (SRC == TQFX4_SRC_F32_RTN || SRC == TQFX4_SRC_F32_TIED) {
            const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(a) + e0);
            const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
            const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            bool finite = true;
            float amax = 0.0f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                finite &= isfinite(v[i]);
                amax = fmaxf(amax, fabsf(v[i]));
            }
#pragma unroll
            for (int s = 16; s > 0; s >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, s));
            bad |= !__all_sync(0xffffffffu, finite);
            __half d = __float2half_rn(__fdiv_rn(amax, 4.0f));
            uint16_t db = __half_as_ushort(d);
            if ((db & 0x7c00u) == 0x7c00u) db = 0x7bffu;  // saturate at 65504
            float cf[8];
            auto codes = [&](uint16_t bits) {
                const float dq = __half2float(__ushort_as_half(bits));
                const float id = (dq != 0.0f) ? __fdiv_rn(1.0f, dq) : 0.0f;
#pragma unroll
                for (int i = 0; i < 8; ++i) cf[i] = fminf(fmaxf(roundf(__fmul_rn(v[i], id)), -4.0f), 4.0f);
            };
            codes(db);
            if (SRC == TQFX4_SRC_F32_TIED && __all_sync(0xffffffffu, finite)) {
                // the tied alternating solver: least-squares scale of the
                // codes, rounded to f16, then the nearest codes to it, until
                // the scale repeats. <w, c>: each lane sums its 8 products in
                // index order, then partners at XOR 16, 8, 4, 2, 1 add (every
                // lane ends with the same value); <c, c> is exact.
                for (int it = 0; it < TQFX4_TIED_MAX_ITER; ++it) {
                    float pw = 0.0f, pc = 0.0f;
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        pw = __fadd_rn(pw, __fmul_rn(v[i], cf[i]));
                        pc = __fadd_rn(pc, __fmul_rn(cf[i], cf[i]));
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) {
                        pw = __fadd_rn(pw, __shfl_xor_sync(0xffffffffu, pw, o));
                        pc = __fadd_rn(pc, __shfl_xor_sync(0xffffffffu, pc, o));
                    }
                    if (pc == 0.0f) break;  // all codes zero (absmax = 0)
                    uint16_t nbits = __half_as_ushort(__float2half_rn(__fdiv_rn(pw, pc)));
                    if ((nbits & 0x7c00u) == 0x7c00u) nbits = 0x7bffu;
                    if (nbits == db) break;  // a fixed point
                    db = nbits;
                    codes(db);
                }
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint32_t uu = finite ? static_cast<uint32_t>(static_cast<int>(cf[i]) + 4) : 4u;
                u[i >> 2] |= uu << (8 * (i & 3));
            }
            dbits[r] = db;
        } else {
            const uint2 a8 = __ldg(reinterpret_cast<const uint2 *>(static_cast<const int8_t *>(a) + e0));
            const uint2 b8 = __ldg(reinterpret_cast<const uint2 *>(t2 + e0));
            bool ok = true;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint32_t wa = (i < 4) ? a8.x : a8.y, wb = (i < 4) ? b8.x : b8.y;
                const int t1v = static_cast<int8_t>((wa >> (8 * (i & 3))) & 0xffu);
                const int t2v = static_cast<int8_t>((wb >> (8 * (i & 3))) & 0xffu);
                ok &= (t1v >= -1 && t1v <= 1 && t2v >= -1 && t2v <= 1);
                const int c = 3 * t1v + t2v;
                const uint32_t uu = (t1v >= -1 && t1v <= 1 && t2v >= -1 && t2v <= 1)
                                        ? static_cast<uint32_t>(c + 4) : 4u;
                u[i >> 2] |= uu << (8 * (i & 3));
            }
            bad |= !__all_sync(0xffffffffu, ok);
            dbits[r] = __ldg(scales + row * nb + b);
        }
        // combine: lane l < 16 keeps elements 8l.. (low nibble) and takes
        // elements 128 + 8l.. (high nibble) from lane l + 16
        const uint32_t h0 = __shfl_down_sync(0xffffffffu, u[0], 16);
        const uint32_t h1 = __shfl_down_sync(0xffffffffu, u[1], 16);
        if (lane < 16) {
            uint2 *dst = reinterpret_cast<uint2 *>(blk + CODE_OFS + r * ROW_BYTES + 8 * lane);
            *dst = make_uint2(u[0] | (h0 << 4), u[1] | (h1 << 4));
        }
    }
    if (lane == 0) {
        *reinterpret_cast<uint2 *>(blk) =
            make_uint2(static_cast<uint32_t>(dbits[0]) | (static_cast<uint32_t>(dbits[1]) << 16),
                       static_cast<uint32_t>(dbits[2]) | (static_cast<uint32_t>(dbits[3]) << 16));
        if (bad) report(status, TQFX4_EDATA, K_PACK, static_cast<int>(unit));
    }
}

// One warp per (row, block) of the activations.
__global__ void __launch_bounds__(256) quantize_kernel(const float *x, int64_t units, int nb, int64_t k,
                                                       int8_t *q, float *da, int32_t *bsum, int *status) {
    grid_dependency_wait();  // x may come from the previous kernel
    grid_dependents_launch();
    const int lane = threadIdx.x & 31;
    const int64_t unit = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (unit >= units) return;
    const int64_t m = unit / nb;
    const int b = static_cast<int>(unit - m * nb);
    const int64_t e0 = m * k + static_cast<int64_t>(b) * QK + 8 * lane;
    const float4 *src = reinterpret_cast<const float4 *>(x + e0);
    const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
    const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
    uint2 packed;
    float d;
    int s;
    const bool ok = quant_block_warp(v, packed, d, s);
    *reinterpret_cast<uint2 *>(q + e0) = packed;
    if (lane == 0) {
        da[unit] = d;
        bsum[unit] = s;
        if (!ok) report(status, TQFX4_EDATA, K_QUANT, static_cast<int>(unit));
    }
}

cudaError_t launch_pack(int src, const void *a, const int8_t *t2, const uint16_t *scales, int64_t n, int64_t k,
                        void *blocks, int *status, cudaStream_t st) {
    const int64_t n_rg = n / 4;
    const int nb = static_cast<int>(k / QK);
    const int64_t units = n_rg * nb;
    if (units == 0) return cudaSuccess;
    const int64_t grid = (units * 32 + 255) / 256;
    if (src == TQFX4_SRC_F32_RTN)
        pack_kernel<TQFX4_SRC_F32_RTN><<<static_cast<unsigned>(grid), 256, 0, st>>>(
            a, t2, scales, n_rg, nb, k, static_cast<uint8_t *>(blocks), status);
    else if (src == TQFX4_SRC_F32_TIED)
        pack_kernel<TQFX4_SRC_F32_TIED><<<static_cast<unsigned>(grid), 256, 0, st>>>(
            a, t2, scales, n_rg, nb, k, static_cast<uint8_t *>(blocks), status);
    else
        pack_kernel<TQFX4_SRC_TRITS><<<static_cast<unsigned>(grid), 256, 0, st>>>(
            a, t2, scales, n_rg, nb, k, static_cast<uint8_t *>(blocks), status);
    return cudaGetLastError();
}

// One warp per block of the matrix: its 512 code bytes (16 a lane, four
// 32-bit words at 4-byte alignment) must hold nibbles 0..8, and lanes 0-3
// check the four f16 row scales are finite. A bad block records TQFX4_EDATA
// with its index.
__global__ void __launch_bounds__(256) validate_kernel(const uint8_t *__restrict__ blocks, int64_t nblocks,
                                                       int *status) {
    const int64_t blk = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (blk >= nblocks) return;  // whole warps
    const uint8_t *b = blocks + blk * BLOCK_BYTES;
    const uint32_t *w = reinterpret_cast<const uint32_t *>(b + CODE_OFS + 16 * lane);
    uint32_t bad = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        // per byte, u + 0x77 reaches bit 7 exactly when the nibble u is 9..15
        const uint32_t x = __ldg(w + i);
        bad |= ((x & 0x0f0f0f0fu) + 0x77777777u | ((x >> 4) & 0x0f0f0f0fu) + 0x77777777u) & 0x80808080u;
    }
    if (lane < ROWS) {  // f16 exponent all ones: infinity or NaN
        const uint16_t h = __ldg(reinterpret_cast<const unsigned short *>(b) + lane);
        bad |= (h & 0x7C00u) == 0x7C00u;
    }
    if (__any_sync(0xffffffffu, bad != 0) && lane == 0)
        report(status, TQFX4_EDATA, K_VALIDATE, static_cast<int>(imin64(blk, 0x7fffffff)));
}

cudaError_t launch_validate(const void *blocks, int64_t n, int64_t k, int *status, cudaStream_t st) {
    const int64_t nblocks = (n / ROWS) * (k / QK);
    if (nblocks == 0) return cudaSuccess;
    const int64_t grid = (nblocks * 32 + 255) / 256;
    validate_kernel<<<static_cast<unsigned>(grid), 256, 0, st>>>(static_cast<const uint8_t *>(blocks), nblocks, status);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const float *x, int64_t m, int64_t k, int8_t *q, float *da, int32_t *bsum,
                            int *status, cudaStream_t st) {
    const int nb = static_cast<int>(k / QK);
    const int64_t units = m * nb;
    if (units == 0) return cudaSuccess;
    const int64_t grid = (units * 32 + 255) / 256;
    return launch_dependent(quantize_kernel, dim3(static_cast<unsigned>(grid)), dim3(256), 0, st, x, units, nb, k, q,
                            da, bsum, status);
}

}  // namespace tq
