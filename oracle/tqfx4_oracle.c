/*
 * tqfx4 oracle: a plain, slow, single-threaded CPU restatement of the
 * tied trit-plane (tq2_0_fx4) integer dot pass and of the mixture-of-experts
 * decode math built on it.
 *
 * THIS IS TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load it. The product path (the CUDA library)
 * neither links nor calls it, and shares no header, table or helper with it.
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off -fPIC -shared (no intrinsics,
 * no SIMD, no OpenMP). Every float operation is a single IEEE binary32
 * operation with round-to-nearest-even; no fused multiply-add is allowed, so
 * the results are identical on x86-64 and aarch64.
 *
 * Paper references are to "Tied Trit-Planes" (arXiv 2608.08910):
 *   Sec. 2.1  the tie alpha = (3s, s): W_hat = s * c, c = 3 t1 + t2 in {-4..4}
 *   Sec. 2.2  the persistent folded format: a 520-byte block covers four
 *             columns x 256 elements, 512 code bytes (two codes per byte) plus
 *             four f16 column scales, 4.0625 bits/weight; codes decode by
 *             arithmetic; integer dot against block-quantized activations;
 *             one float multiply-add per block; a shared float schedule.
 * Readings where the paper is silent (byte order inside the block, nibble
 * encoding, activation block size and scale type, the router and SwiGLU
 * arithmetic) are stated at each function.
 *
 * Parity status: every function here is pinned by the CPU test suite
 * (closed forms, brute force, library routines); none is "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define QK 256          /* elements per block along K (Sec. 2.2) */
#define ROWS 4          /* output rows ("columns") per block (Sec. 2.2) */
#define BLOCK_BYTES 520 /* 8 scale bytes + 512 code bytes (Sec. 2.2) */
#define CODE_OFS 8      /* reading: the four f16 scales come first */
#define ROW_CODE_BYTES 128

/* ------------------------------------------------------------------ */
/* Sec. 2.1: the fold. c = 3 t1 + t2, t1, t2 in {-1, 0, 1}.            */
/* ------------------------------------------------------------------ */

/* Returns c in -4..4, or -100 if a trit is outside {-1, 0, 1}. */
int tqo_fold(int t1, int t2) {
    if (t1 < -1 || t1 > 1 || t2 < -1 || t2 > 1) return -100;
    return 3 * t1 + t2;
}

/* Inverse of the fold (balanced ternary, two digits): t2 is the balanced
 * residue of c modulo 3, t1 the remaining digit. Returns 0, or -1 if c is
 * outside -4..4. */
int tqo_unfold(int c, int *t1, int *t2) {
    if (c < -4 || c > 4) return -1;
    int r = ((c % 3) + 3) % 3;   /* 0, 1, 2 */
    int d2 = (r == 2) ? -1 : r;  /* balanced digit -1, 0, 1 */
    *t2 = d2;
    *t1 = (c - d2) / 3;
    return 0;
}

/* ------------------------------------------------------------------ */
/* IEEE 754 binary16, written out from the format definition.           */
/* ------------------------------------------------------------------ */

/* float -> binary16, round to nearest, ties to even; overflow gives inf. */
uint16_t tqo_f32_to_f16(float f) {
    uint32_t x;
    memcpy(&x, &f, 4);
    uint32_t sign = (x >> 16) & 0x8000u;
    uint32_t ex = (x >> 23) & 0xffu;
    uint32_t man = x & 0x7fffffu;
    if (ex == 0xffu) return (uint16_t)(sign | 0x7c00u | (man ? 0x200u : 0u));
    int e = (int)ex - 127 + 15;
    if (e >= 31) return (uint16_t)(sign | 0x7c00u);
    if (e <= 0) {
        if (e < -10) return (uint16_t)sign;
        uint32_t m = man | 0x800000u;
        int shift = 14 - e;
        uint32_t h = m >> shift;
        uint32_t rem = m & ((1u << shift) - 1u);
        uint32_t half = 1u << (shift - 1);
        if (rem > half || (rem == half && (h & 1u))) h++;
        return (uint16_t)(sign | h);
    }
    uint32_t h = ((uint32_t)e << 10) | (man >> 13);
    uint32_t rem = man & 0x1fffu;
    if (rem > 0x1000u || (rem == 0x1000u && (h & 1u))) h++;
    return (uint16_t)(sign | h);
}

float tqo_f16_to_f32(uint16_t h) {
    int sign = (h >> 15) & 1;
    int ex = (h >> 10) & 0x1f;
    int man = h & 0x3ff;
    double v;
    if (ex == 0) v = ldexp((double)man, -24);
    else if (ex == 31) v = man ? NAN : INFINITY;
    else v = ldexp((double)(1024 + man), ex - 25);
    return (float)(sign ? -v : v);
}

/* ------------------------------------------------------------------ */
/* Sec. 2.2: the 520-byte block.                                        */
/* Reading of the byte order (the paper names the parts but not their   */
/* order): bytes 0..7 hold the four f16 scales d[r] of rows r = 0..3    */
/* (little endian); bytes 8 + 128 r .. 8 + 128 r + 127 hold row r's 256  */
/* codes, byte j carrying element j in its low nibble and element       */
/* j + 128 in its high nibble. A nibble stores u = c + 4 in 0..8          */
/* (values 9..15 are invalid). Blocks of a matrix W[N][K] are ordered    */
/* [N/4 row groups][K/256 blocks].                                       */
/* ------------------------------------------------------------------ */

int64_t tqo_matrix_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || n % ROWS || k % QK) return -1;
    return (n / ROWS) * (k / QK) * BLOCK_BYTES;
}

static uint8_t *block_at(uint8_t *blocks, int64_t k, int64_t n, int64_t kk) {
    int64_t nb = k / QK;
    return blocks + ((n / ROWS) * nb + kk / QK) * BLOCK_BYTES;
}

static const uint8_t *cblock_at(const uint8_t *blocks, int64_t k, int64_t n, int64_t kk) {
    int64_t nb = k / QK;
    return blocks + ((n / ROWS) * nb + kk / QK) * BLOCK_BYTES;
}

static void put_scale(uint8_t *blk, int r, uint16_t d) {
    blk[2 * r] = (uint8_t)(d & 0xff);
    blk[2 * r + 1] = (uint8_t)(d >> 8);
}

static uint16_t get_scale(const uint8_t *blk, int r) {
    return (uint16_t)(blk[2 * r] | (blk[2 * r + 1] << 8));
}

static void put_code(uint8_t *blk, int r, int j, int c) {
    uint8_t *p = blk + CODE_OFS + ROW_CODE_BYTES * r + (j % ROW_CODE_BYTES);
    uint8_t u = (uint8_t)(c + 4);
    if (j < ROW_CODE_BYTES) *p = (uint8_t)((*p & 0xf0) | u);
    else *p = (uint8_t)((*p & 0x0f) | (u << 4));
}

/* Returns the nibble u (0..15); the caller maps it to c = u - 4. */
static int get_nibble(const uint8_t *blk, int r, int j) {
    const uint8_t *p = blk + CODE_OFS + ROW_CODE_BYTES * r + (j % ROW_CODE_BYTES);
    return (j < ROW_CODE_BYTES) ? (*p & 0x0f) : (*p >> 4);
}

/* Fold two trit planes into blocks (Sec. 2.1 and 2.2): c = 3 t1 + t2 with the
 * given f16 scale per (row, 256-block). t1, t2: int8 [n][k]; d: [n][k/256].
 * Returns 0, -1 on a bad shape, -2 on a trit outside {-1, 0, 1}. */
int tqo_pack_trits(const int8_t *t1, const int8_t *t2, const uint16_t *d,
                   int64_t n, int64_t k, uint8_t *out) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    memset(out, 0, (size_t)tqo_matrix_bytes(n, k));
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            uint8_t *blk = block_at(out, k, row, b * QK);
            put_scale(blk, (int)(row % ROWS), d[row * nb + b]);
            for (int j = 0; j < QK; j++) {
                int64_t i = row * k + b * QK + j;
                int c = tqo_fold(t1[i], t2[i]);
                if (c == -100) return -2;
                put_code(blk, (int)(row % ROWS), j, c);
            }
        }
    }
    return 0;
}

/* Round-to-nearest codes from fp32 weights. Per (row, 256-block):
 *   d  = f16(absmax / 4)           (saturated to the largest finite f16)
 *   dq = float(d)                   (codes use the stored, f16-rounded scale)
 *   c  = clamp(round(w * (1/dq)), -4, 4), round = half away from zero,
 * with dq = 0 giving every code 0. W_hat = dq * c is the tied quantizer of
 * Sec. 2.1 fitted in one step. Returns 0, -1 on a bad shape, -3 on a
 * non-finite weight. */
int tqo_pack_rtn(const float *w, int64_t n, int64_t k, uint8_t *out) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    memset(out, 0, (size_t)tqo_matrix_bytes(n, k));
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            const float *src = w + row * k + b * QK;
            float amax = 0.0f;
            for (int j = 0; j < QK; j++) {
                if (!isfinite(src[j])) return -3;
                float a = fabsf(src[j]);
                if (a > amax) amax = a;
            }
            uint16_t d = tqo_f32_to_f16(amax / 4.0f);
            if ((d & 0x7c00u) == 0x7c00u) d = 0x7bffu; /* saturate */
            float dq = tqo_f16_to_f32(d);
            float id = (dq != 0.0f) ? 1.0f / dq : 0.0f;
            uint8_t *blk = block_at(out, k, row, b * QK);
            put_scale(blk, (int)(row % ROWS), d);
            for (int j = 0; j < QK; j++) {
                float v = roundf(src[j] * id);
                if (v > 4.0f) v = 4.0f;
                if (v < -4.0f) v = -4.0f;
                put_code(blk, (int)(row % ROWS), j, (int)v);
            }
        }
    }
    return 0;
}

/* The tied alternating solver (Sec. 2.1: the solver alternates plane
 * updates against the single scale s, which is the same as fitting the
 * uniform quantizer W_hat = s * c, c in -4..4; scales serialize to f16).
 * Readings where the paper gives no details (initialisation, iteration
 * count, the group, the arithmetic): per (row, 256-block),
 *   start:  the round-to-nearest fit (tqo_pack_rtn): s = f16(absmax / 4),
 *           c = clamp(round(w * (1/s)), -4, 4);
 *   repeat: s' = f16(<w, c> / <c, c>)   (least-squares scale of the codes,
 *                                        rounded to the nearest f16);
 *           stop if s' == s (a fixed point) or after max_iter updates;
 *           s = s', c = clamp(round(w * (1/s)), -4, 4).
 * Each step minimises the block's squared error over its own variable (the
 * nearest level for each weight; and, the error being a parabola in s, the
 * f16 value nearest the least-squares optimum is the best f16 value for the
 * codes), so the error never exceeds the round-to-nearest fit's, and the
 * stored block is a pair (s, c) whose codes are nearest to their own scale.
 * Arithmetic: binary32, no fused operations. <c, c> is an exact integer;
 * <w, c> is summed in one fixed order: 32 groups of 8 consecutive elements,
 * each summed in index order, then the 32 partial sums combined pairwise
 * with the partner whose index differs in bit 4, 3, 2, 1, 0 in turn (every
 * partial of a level becomes p[l] + p[l ^ o]). iters (nullable, [n][k/256])
 * receives the number of scale updates, negated when max_iter stopped the
 * block before a fixed point. Returns 0, -1 on a bad shape or max_iter < 0,
 * -3 on a non-finite weight. */
static float tied_dot_wc(const float *w, const float *c) {
    float p[32], q[32];
    for (int l = 0; l < 32; l++) {
        float a = 0.0f;
        for (int i = 0; i < 8; i++) a = a + w[8 * l + i] * c[8 * l + i];
        p[l] = a;
    }
    for (int o = 16; o > 0; o >>= 1) {
        for (int l = 0; l < 32; l++) q[l] = p[l] + p[l ^ o];
        memcpy(p, q, sizeof(p));
    }
    return p[0];
}

static void tied_codes(const float *w, float dq, float *c) {
    float id = (dq != 0.0f) ? 1.0f / dq : 0.0f;
    for (int j = 0; j < QK; j++) {
        float v = roundf(w[j] * id);
        if (v > 4.0f) v = 4.0f;
        if (v < -4.0f) v = -4.0f;
        c[j] = v;
    }
}

int tqo_pack_tied(const float *w, int64_t n, int64_t k, int max_iter, uint8_t *out, int32_t *iters) {
    if (tqo_matrix_bytes(n, k) < 0 || max_iter < 0) return -1;
    int64_t nb = k / QK;
    memset(out, 0, (size_t)tqo_matrix_bytes(n, k));
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            const float *src = w + row * k + b * QK;
            float amax = 0.0f;
            for (int j = 0; j < QK; j++) {
                if (!isfinite(src[j])) return -3;
                float a = fabsf(src[j]);
                if (a > amax) amax = a;
            }
            uint16_t d = tqo_f32_to_f16(amax / 4.0f);
            if ((d & 0x7c00u) == 0x7c00u) d = 0x7bffu; /* saturate */
            float c[QK];
            tied_codes(src, tqo_f16_to_f32(d), c);
            int updates = 0, fixed = 0;
            while (!fixed && updates < max_iter) {
                float cc = 0.0f;
                for (int j = 0; j < QK; j++) cc = cc + c[j] * c[j];
                if (cc == 0.0f) { fixed = 1; break; } /* all codes zero: absmax = 0 */
                uint16_t d2 = tqo_f32_to_f16(tied_dot_wc(src, c) / cc);
                if ((d2 & 0x7c00u) == 0x7c00u) d2 = 0x7bffu;
                if (d2 == d) { fixed = 1; break; }
                d = d2;
                tied_codes(src, tqo_f16_to_f32(d), c);
                updates++;
            }
            if (iters) iters[row * nb + b] = fixed ? updates : -updates;
            uint8_t *blk = block_at(out, k, row, b * QK);
            put_scale(blk, (int)(row % ROWS), d);
            for (int j = 0; j < QK; j++) put_code(blk, (int)(row % ROWS), j, (int)c[j]);
        }
    }
    return 0;
}

/* Decode blocks back to codes c[n][k] (c = u - 4, "by arithmetic") and
 * scales d[n][k/256]. Returns 0, -1 on a bad shape, -4 on a nibble > 8. */
int tqo_unpack(const uint8_t *blocks, int64_t n, int64_t k, int8_t *c, uint16_t *d) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            const uint8_t *blk = cblock_at(blocks, k, row, b * QK);
            if (d) d[row * nb + b] = get_scale(blk, (int)(row % ROWS));
            for (int j = 0; j < QK; j++) {
                int u = get_nibble(blk, (int)(row % ROWS), j);
                if (u > 8) return -4;
                c[row * k + b * QK + j] = (int8_t)(u - 4);
            }
        }
    }
    return 0;
}

/* Dequantized weights W_hat = s * c (Sec. 2.1), in fp64. */
int tqo_dequant(const uint8_t *blocks, int64_t n, int64_t k, double *w_hat) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            const uint8_t *blk = cblock_at(blocks, k, row, b * QK);
            double s = (double)tqo_f16_to_f32(get_scale(blk, (int)(row % ROWS)));
            for (int j = 0; j < QK; j++) {
                int u = get_nibble(blk, (int)(row % ROWS), j);
                if (u > 8) return -4;
                w_hat[row * k + b * QK + j] = s * (double)(u - 4);
            }
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Sec. 2.2: block-quantized activations. Reading: 256-element blocks    */
/* aligned with the weight blocks, symmetric int8 in -127..127, one fp32 */
/* scale per block:                                                      */
/*   da = absmax / 127, q = clamp(round(x * (1/da)), -127, 127),          */
/*   bsum = sum(q) (the offset-binary dot needs it).                      */
/* x: [m][k]; q: [m][k]; da, bsum: [m][k/256].                          */
/* Returns 0, -1 on a bad shape, -3 on a non-finite input.               */
/* ------------------------------------------------------------------ */
int tqo_quantize_act(const float *x, int64_t m, int64_t k, int8_t *q, float *da, int32_t *bsum) {
    if (m < 0 || k < 0 || k % QK) return -1;
    int64_t nb = k / QK;
    for (int64_t t = 0; t < m; t++) {
        for (int64_t b = 0; b < nb; b++) {
            const float *src = x + t * k + b * QK;
            float amax = 0.0f;
            for (int j = 0; j < QK; j++) {
                if (!isfinite(src[j])) return -3;
                float a = fabsf(src[j]);
                if (a > amax) amax = a;
            }
            float s = amax / 127.0f;
            float id = (s != 0.0f) ? 1.0f / s : 0.0f;
            int32_t sum = 0;
            for (int j = 0; j < QK; j++) {
                float v = roundf(src[j] * id);
                if (v > 127.0f) v = 127.0f;
                if (v < -127.0f) v = -127.0f;
                q[t * k + b * QK + j] = (int8_t)v;
                sum += (int32_t)v;
            }
            da[t * nb + b] = s;
            bsum[t * nb + b] = sum;
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Sec. 2.2: the integer dot pass.                                       */
/*   S[n][b] = sum_{j<256} c[n][256 b + j] * q[256 b + j]   (exact int)   */
/*   y[n]    = sum over b ascending of float(S) * (d[n][b] * da[b])       */
/* The float schedule is fixed: acc starts at +0.0f and, for b = 0, 1,    */
/* ..., acc = acc + float(S) * (dq * da) with each operation rounded to   */
/* binary32 (no fused multiply-add). Returns 0, -1 on a bad shape, -4 on  */
/* an invalid nibble.                                                     */
/* ------------------------------------------------------------------ */
int tqo_block_sums(const uint8_t *blocks, int64_t n, int64_t k, const int8_t *q, int32_t *S) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    for (int64_t row = 0; row < n; row++) {
        for (int64_t b = 0; b < nb; b++) {
            const uint8_t *blk = cblock_at(blocks, k, row, b * QK);
            int32_t s = 0;
            for (int j = 0; j < QK; j++) {
                int u = get_nibble(blk, (int)(row % ROWS), j);
                if (u > 8) return -4;
                s += (int32_t)(u - 4) * (int32_t)q[b * QK + j];
            }
            S[row * nb + b] = s;
        }
    }
    return 0;
}

int tqo_gemv(const uint8_t *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
             float *y, int32_t *S_out) {
    if (tqo_matrix_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    int32_t *S = S_out ? S_out : (int32_t *)malloc(sizeof(int32_t) * (size_t)(n * nb + 1));
    if (!S) return -5;
    int rc = tqo_block_sums(blocks, n, k, q, S);
    if (rc == 0) {
        for (int64_t row = 0; row < n; row++) {
            float acc = 0.0f;
            for (int64_t b = 0; b < nb; b++) {
                const uint8_t *blk = cblock_at(blocks, k, row, b * QK);
                float dq = tqo_f16_to_f32(get_scale(blk, (int)(row % ROWS)));
                float sc = dq * da[b];
                float t = (float)S[row * nb + b] * sc;
                acc = acc + t;
            }
            y[row] = acc;
        }
    }
    if (!S_out) free(S);
    return rc;
}

/* ------------------------------------------------------------------ */
/* The MXFP4 arm (Sec. 2.3: the released expert bytes, served         */
/* directly): OCP microscaling blocks of 32 elements, one e8m0          */
/* scale byte E (2^(E-127); E = 255 is NaN) and 32 e2m1 values (sign,    */
/* two exponent bits, one mantissa bit: 0, 0.5, 1, 1.5, 2, 3, 4, 6), 17 */
/* bytes per block, 4.25 bits/weight. Readings: the block stores E in    */
/* byte 0 and the codes in bytes 1..16, element j (< 16) in the low      */
/* nibble of byte 1 + j and element 16 + j in the high nibble (the       */
/* interchange order of the released files); rows of k/32 blocks are     */
/* contiguous. The dot pass uses the doubled codes c = 2 * e2m1 (the     */
/* integers 0, 1, 2, 3, 4, 6, 8, 12 with a sign), so a block's sum       */
/* S = sum c q is an exact int32 and the block's value is 2^(E-128) * S. */
/* ------------------------------------------------------------------ */
#define MX_K 32
#define MX_BYTES 17

int64_t tqo_mxfp4_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || k % MX_K) return -1;
    return n * (k / MX_K) * MX_BYTES;
}

/* Doubled e2m1 code of a nibble: magnitudes 0, 1, 2, 3, 4, 6, 8, 12. */
static int mx_code(int nib) {
    static const int mag[8] = {0, 1, 2, 3, 4, 6, 8, 12};
    int m = mag[nib & 7];
    return (nib & 8) ? -m : m;
}

static int mx_nibble(const uint8_t *blk, int j) {
    const uint8_t b = blk[1 + (j % 16)];
    return (j < 16) ? (b & 0x0f) : (b >> 4);
}

/* Dequantized weights (fp64) W[n][k] = 2^(E-128) * c. Returns 0, -1 on a bad
 * shape, -4 on a NaN scale (E = 255). */
int tqo_mxfp4_dequant(const uint8_t *blocks, int64_t n, int64_t k, double *w) {
    if (tqo_mxfp4_bytes(n, k) < 0) return -1;
    int64_t nb = k / MX_K;
    for (int64_t row = 0; row < n; row++)
        for (int64_t b = 0; b < nb; b++) {
            const uint8_t *blk = blocks + (row * nb + b) * MX_BYTES;
            if (blk[0] == 255) return -4;
            double sc = ldexp(1.0, (int)blk[0] - 128);
            for (int j = 0; j < MX_K; j++) w[row * k + b * MX_K + j] = sc * mx_code(mx_nibble(blk, j));
        }
    return 0;
}

/* GEMV of MXFP4 blocks against per-256-block int8 activations (q, da as
 * tqo_quantize_act writes them): per 32-block the exact sum S = sum c q and
 * its value t = (float)S * 2^(E-128) (exact: an integer below 2^16 times a
 * power of two that binary32 holds, subnormals included; inf past the
 * range). The float schedule follows the activation's scale unit: per
 * 256-element block g (eight 32-blocks, one da[g]) G = G + t over its
 * 32-blocks in ascending order, then acc = acc + G * da[g] over g in
 * ascending order (each product and sum rounded once). S_out (nullable)
 * receives S [n][k/32]. Returns 0, -1 on a bad shape or k not a multiple of
 * 256, -4 on a NaN scale, -5 on allocation failure. */
int tqo_mxfp4_gemv(const uint8_t *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                   int32_t *S_out) {
    if (tqo_mxfp4_bytes(n, k) < 0 || k % QK) return -1;
    int64_t nb = k / MX_K;
    const int per_g = QK / MX_K;
    for (int64_t row = 0; row < n; row++) {
        float acc = 0.0f;
        for (int64_t g = 0; g < k / QK; g++) {
            float G = 0.0f;
            for (int64_t b = g * per_g; b < (g + 1) * per_g; b++) {
                const uint8_t *blk = blocks + (row * nb + b) * MX_BYTES;
                if (blk[0] == 255) return -4;
                int32_t s = 0;
                for (int j = 0; j < MX_K; j++)
                    s += (int32_t)mx_code(mx_nibble(blk, j)) * (int32_t)q[b * MX_K + j];
                if (S_out) S_out[row * nb + b] = s;
                G = G + (float)s * ldexpf(1.0f, (int)blk[0] - 128);
            }
            acc = acc + G * da[g];
        }
        y[row] = acc;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* The free-scale two-plane format (Table 1's free-scale K=2 row, 4.125   */
/* bits/weight: the pair with two independent scales does not fold, so   */
/* the two trit planes are stored apart): W = a1 t1 + a2 t2 per row and   */
/* 256 columns, t1, t2 in {-1, 0, 1}, a1, a2 f16. Reading of the bytes     */
/* (the paper gives only the size): blocks of 4 rows x 256 columns, 528   */
/* bytes, ordered [N/4 row groups][K/256 blocks] like the 520-byte block; */
/* bytes 0..7 hold a1 of rows 0..3 and bytes 8..15 a2 (f16, little        */
/* endian); bytes 16 + 128 r .. + 63 hold row r's plane t1 and the next 64 */
/* bytes its plane t2, element j in bits 2 (j % 4) of byte j / 4 as       */
/* u = t + 1 in 0..2 (3 is invalid).                                      */
/* ------------------------------------------------------------------ */
#define FREE_BLOCK_BYTES 528
#define FREE_PLANE_OFS 16
#define FREE_ROW_BYTES 128

int64_t tqo_free_bytes(int64_t n, int64_t k) {
    if (n < 0 || k < 0 || n % ROWS || k % QK) return -1;
    return (n / ROWS) * (k / QK) * FREE_BLOCK_BYTES;
}

static const uint8_t *free_block(const uint8_t *blocks, int64_t k, int64_t row, int64_t b) {
    return blocks + ((row / ROWS) * (k / QK) + b) * FREE_BLOCK_BYTES;
}

/* Trit of plane p (0: t1, 1: t2) of row r, element j of a block; -9 if invalid. */
static int free_trit(const uint8_t *blk, int r, int p, int j) {
    const uint8_t byte = blk[FREE_PLANE_OFS + FREE_ROW_BYTES * r + 64 * p + j / 4];
    const int u = (byte >> (2 * (j % 4))) & 3;
    return u == 3 ? -9 : u - 1;
}

/* Pack two trit planes with their scales. t1, t2: int8 [n][k]; a1, a2: f16
 * bits [n][k/256]. Returns 0, -1 on a bad shape, -2 on a trit outside
 * {-1, 0, 1}. */
int tqo_pack_free(const int8_t *t1, const int8_t *t2, const uint16_t *a1, const uint16_t *a2,
                  int64_t n, int64_t k, uint8_t *out) {
    if (tqo_free_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    memset(out, 0, (size_t)tqo_free_bytes(n, k));
    for (int64_t row = 0; row < n; row++)
        for (int64_t b = 0; b < nb; b++) {
            uint8_t *blk = out + ((row / ROWS) * nb + b) * FREE_BLOCK_BYTES;
            const int r = (int)(row % ROWS);
            const uint16_t s1 = a1[row * nb + b], s2 = a2[row * nb + b];
            blk[2 * r] = (uint8_t)(s1 & 0xff);
            blk[2 * r + 1] = (uint8_t)(s1 >> 8);
            blk[8 + 2 * r] = (uint8_t)(s2 & 0xff);
            blk[8 + 2 * r + 1] = (uint8_t)(s2 >> 8);
            for (int j = 0; j < QK; j++)
                for (int p = 0; p < 2; p++) {
                    const int t = (p ? t2 : t1)[row * k + b * QK + j];
                    if (t < -1 || t > 1) return -2;
                    blk[FREE_PLANE_OFS + FREE_ROW_BYTES * r + 64 * p + j / 4] |= (uint8_t)((t + 1) << (2 * (j % 4)));
                }
        }
    return 0;
}

/* W = a1 t1 + a2 t2 in fp64. Returns 0, -1 on a bad shape, -3 on an
 * invalid trit. */
int tqo_free_dequant(const uint8_t *blocks, int64_t n, int64_t k, double *w) {
    if (tqo_free_bytes(n, k) < 0) return -1;
    for (int64_t row = 0; row < n; row++)
        for (int64_t b = 0; b < k / QK; b++) {
            const uint8_t *blk = free_block(blocks, k, row, b);
            const int r = (int)(row % ROWS);
            const double s1 = tqo_f16_to_f32((uint16_t)(blk[2 * r] | (blk[2 * r + 1] << 8)));
            const double s2 = tqo_f16_to_f32((uint16_t)(blk[8 + 2 * r] | (blk[8 + 2 * r + 1] << 8)));
            for (int j = 0; j < QK; j++) {
                const int x1 = free_trit(blk, r, 0, j), x2 = free_trit(blk, r, 1, j);
                if (x1 < -1 || x2 < -1) return -3;
                w[row * k + b * QK + j] = s1 * x1 + s2 * x2;
            }
        }
    return 0;
}

/* The two-plane dot pass: per (row, 256-block) the exact int32 sums
 * S1 = sum t1 q and S2 = sum t2 q, then the fixed float schedule
 * acc = acc + (float(S1) * (a1 * da) + float(S2) * (a2 * da)), blocks in
 * ascending order, every product and sum rounded once. S1, S2 (nullable):
 * [n][k/256]. Returns 0, -1 on a bad shape, -3 on an invalid trit. */
int tqo_free_gemv(const uint8_t *blocks, int64_t n, int64_t k, const int8_t *q, const float *da, float *y,
                  int32_t *S1_out, int32_t *S2_out) {
    if (tqo_free_bytes(n, k) < 0) return -1;
    int64_t nb = k / QK;
    for (int64_t row = 0; row < n; row++) {
        float acc = 0.0f;
        for (int64_t b = 0; b < nb; b++) {
            const uint8_t *blk = free_block(blocks, k, row, b);
            const int r = (int)(row % ROWS);
            int32_t s1 = 0, s2 = 0;
            for (int j = 0; j < QK; j++) {
                const int x1 = free_trit(blk, r, 0, j), x2 = free_trit(blk, r, 1, j);
                if (x1 < -1 || x2 < -1) return -3;
                s1 += x1 * (int32_t)q[b * QK + j];
                s2 += x2 * (int32_t)q[b * QK + j];
            }
            if (S1_out) S1_out[row * nb + b] = s1;
            if (S2_out) S2_out[row * nb + b] = s2;
            const float a1 = tqo_f16_to_f32((uint16_t)(blk[2 * r] | (blk[2 * r + 1] << 8)));
            const float a2 = tqo_f16_to_f32((uint16_t)(blk[8 + 2 * r] | (blk[8 + 2 * r + 1] << 8)));
            const float p1 = (float)s1 * (a1 * da[b]);
            const float p2 = (float)s2 * (a2 * da[b]);
            const float t = p1 + p2;
            acc = acc + t;
        }
        y[row] = acc;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* exp in binary32 (used by SwiGLU). The paper does not fix how SwiGLU   */
/* is evaluated; because its output is re-quantized to int8 (a rounding  */
/* decision), both this oracle and the kernel evaluate it with the same  */
/* fully specified binary32 method, each from its own source:            */
/* Cody-Waite range reduction z = n ln2 + r with ln2 split into          */
/* 0.693359375 + (-2.12194440e-4) (the Cephes split), |r| <= ln2/2, then */
/* the degree-7 Taylor polynomial of e^r in Horner form, scaled by 2^n.  */
/* Inputs are clamped to [-87, 88] so the result stays a normal number.  */
/* ------------------------------------------------------------------ */
float tqo_expf(float z) {
    if (z != z) return z;
    if (z > 88.0f) z = 88.0f;
    if (z < -87.0f) z = -87.0f;
    float t = z * 1.44269502f; /* log2(e) rounded to binary32 */
    float nf = rintf(t);
    float r = z - nf * 0.693359375f;
    r = r - nf * -2.12194440e-4f;
    float p = 1.98412698e-4f;        /* 1/7! */
    p = p * r + 1.38888889e-3f;      /* 1/6! */
    p = p * r + 8.33333333e-3f;      /* 1/5! */
    p = p * r + 4.16666667e-2f;      /* 1/4! */
    p = p * r + 1.66666667e-1f;      /* 1/3! */
    p = p * r + 0.5f;                /* 1/2! */
    p = p * r + 1.0f;
    p = p * r + 1.0f;
    return ldexpf(p, (int)nf);
}

/* SwiGLU: h = silu(g) * u with silu(g) = g / (1 + exp(-g)), binary32. */
void tqo_swiglu(const float *g, const float *u, int64_t n, float *h) {
    for (int64_t i = 0; i < n; i++) {
        float e = tqo_expf(-g[i]);
        float den = 1.0f + e;
        float s = g[i] / den;
        h[i] = s * u[i];
    }
}

/* ------------------------------------------------------------------ */
/* One routed expert (gate/up/down SwiGLU FFN, the projections the paper */
/* stores in tq2_0_fx4): x [hidden] -> out [hidden].                       */
/*   qx = quant(x); g = gemv(gate, qx); u = gemv(up, qx);                  */
/*   h = swiglu(g, u); qh = quant(h); out = gemv(down, qh).                */
/* gate, up: [inter][hidden]; down: [hidden][inter]. Optional debug        */
/* outputs (nullable): g, u, h [inter]; qh [inter]; dh, bh [inter/256].    */
/* ------------------------------------------------------------------ */
/* The dot pass of the expert's weight format: 0 = tq2_0_fx4 blocks,
 * 1 = MXFP4 blocks (the expert-lossless arm of Sec. 2.3). */
static int gemv_fmt(int fmt, const uint8_t *blocks, int64_t n, int64_t k, const int8_t *q, const float *da,
                    float *y) {
    return fmt ? tqo_mxfp4_gemv(blocks, n, k, q, da, y, NULL) : tqo_gemv(blocks, n, k, q, da, y, NULL);
}

static int expert_ffn_fmt(int fmt, const uint8_t *gate, const uint8_t *up, const uint8_t *down,
                          int64_t hidden, int64_t inter, const float *x, float *out,
                          float *g_dbg, float *u_dbg, float *h_dbg, int8_t *qh_dbg,
                          float *dh_dbg, int32_t *bh_dbg) {
    if (hidden % QK || inter % QK || hidden <= 0 || inter <= 0) return -1;
    int64_t nbh = hidden / QK, nbi = inter / QK;
    int8_t *qx = (int8_t *)malloc((size_t)hidden);
    float *dx = (float *)malloc(sizeof(float) * (size_t)nbh);
    int32_t *bx = (int32_t *)malloc(sizeof(int32_t) * (size_t)nbh);
    float *g = (float *)malloc(sizeof(float) * (size_t)inter);
    float *u = (float *)malloc(sizeof(float) * (size_t)inter);
    float *h = (float *)malloc(sizeof(float) * (size_t)inter);
    int8_t *qh = (int8_t *)malloc((size_t)inter);
    float *dh = (float *)malloc(sizeof(float) * (size_t)nbi);
    int32_t *bh = (int32_t *)malloc(sizeof(int32_t) * (size_t)nbi);
    int rc = -5;
    if (qx && dx && bx && g && u && h && qh && dh && bh) {
        rc = tqo_quantize_act(x, 1, hidden, qx, dx, bx);
        if (!rc) rc = gemv_fmt(fmt, gate, inter, hidden, qx, dx, g);
        if (!rc) rc = gemv_fmt(fmt, up, inter, hidden, qx, dx, u);
        if (!rc) {
            tqo_swiglu(g, u, inter, h);
            rc = tqo_quantize_act(h, 1, inter, qh, dh, bh);
        }
        if (!rc) rc = gemv_fmt(fmt, down, hidden, inter, qh, dh, out);
        if (!rc) {
            if (g_dbg) memcpy(g_dbg, g, sizeof(float) * (size_t)inter);
            if (u_dbg) memcpy(u_dbg, u, sizeof(float) * (size_t)inter);
            if (h_dbg) memcpy(h_dbg, h, sizeof(float) * (size_t)inter);
            if (qh_dbg) memcpy(qh_dbg, qh, (size_t)inter);
            if (dh_dbg) memcpy(dh_dbg, dh, sizeof(float) * (size_t)nbi);
            if (bh_dbg) memcpy(bh_dbg, bh, sizeof(int32_t) * (size_t)nbi);
        }
    }
    free(qx); free(dx); free(bx); free(g); free(u); free(h); free(qh); free(dh); free(bh);
    return rc;
}

int tqo_expert_ffn(const uint8_t *gate, const uint8_t *up, const uint8_t *down,
                   int64_t hidden, int64_t inter, const float *x, float *out,
                   float *g_dbg, float *u_dbg, float *h_dbg, int8_t *qh_dbg,
                   float *dh_dbg, int32_t *bh_dbg) {
    return expert_ffn_fmt(0, gate, up, down, hidden, inter, x, out, g_dbg, u_dbg, h_dbg, qh_dbg, dh_dbg, bh_dbg);
}

/* The same expert with MXFP4 gate, up and down matrices. */
int tqo_expert_ffn_mxfp4(const uint8_t *gate, const uint8_t *up, const uint8_t *down,
                         int64_t hidden, int64_t inter, const float *x, float *out,
                         float *g_dbg, float *u_dbg, float *h_dbg, int8_t *qh_dbg,
                         float *dh_dbg, int32_t *bh_dbg) {
    return expert_ffn_fmt(1, gate, up, down, hidden, inter, x, out, g_dbg, u_dbg, h_dbg, qh_dbg, dh_dbg, bh_dbg);
}

/* ------------------------------------------------------------------ */
/* Router (the paper does not describe it; this is the standard MoE      */
/* router that the workload names): logits in fp64,                       */
/*   l[e] = sum_k W_r[e][k] x[k] + bias[e],                               */
/* the top_k experts by logit (ties to the lower index), in rank order,   */
/* and w_j = exp(l_j - l_0) / sum_i exp(l_i - l_0) over the selected ones */
/* (equal to renormalizing the top-k of a full softmax), rounded to fp32. */
/* W_r: [E][H]; bias nullable [E]; logits (nullable) [E]; idx, w [top_k]. */
/* ------------------------------------------------------------------ */
int tqo_router(const float *Wr, const float *bias, int64_t E, int64_t H, const float *x,
               int top_k, double *logits_out, int32_t *idx, float *w) {
    if (E <= 0 || H <= 0 || top_k <= 0 || top_k > E) return -1;
    double *l = (double *)malloc(sizeof(double) * (size_t)E);
    char *taken = (char *)calloc((size_t)E, 1);
    if (!l || !taken) { free(l); free(taken); return -5; }
    for (int64_t e = 0; e < E; e++) {
        double acc = 0.0;
        for (int64_t kk = 0; kk < H; kk++) acc += (double)Wr[e * H + kk] * (double)x[kk];
        if (bias) acc += (double)bias[e];
        l[e] = acc;
    }
    for (int j = 0; j < top_k; j++) {
        int64_t best = -1;
        for (int64_t e = 0; e < E; e++) {
            if (taken[e]) continue;
            if (best < 0 || l[e] > l[best]) best = e; /* strict: ties keep the lower index */
        }
        taken[best] = 1;
        idx[j] = (int32_t)best;
    }
    double m = l[idx[0]], sum = 0.0;
    for (int j = 0; j < top_k; j++) sum += exp(l[idx[j]] - m);
    for (int j = 0; j < top_k; j++) w[j] = (float)(exp(l[idx[j]] - m) / sum);
    if (logits_out) memcpy(logits_out, l, sizeof(double) * (size_t)E);
    free(l); free(taken);
    return 0;
}

/* ------------------------------------------------------------------ */
/* MoE layer for one token: route, run each selected expert, combine in  */
/* rank order: out[n] = sum over j = 0..top_k-1 of w_j * o_j[n], fp32,    */
/* acc starting at +0.0f, acc = acc + w_j * o_j[n] (no fused multiply-add).*/
/* Experts are given as per-expert pointer arrays; an entry may be NULL   */
/* for an expert the token does not select (returns -6 if it does).       */
/* ------------------------------------------------------------------ */
static int moe_token_fmt(int fmt, const uint8_t *const *gate, const uint8_t *const *up,
                         const uint8_t *const *down, int64_t E, int64_t hidden, int64_t inter,
                         const float *Wr, const float *bias, int top_k, const float *x, float *out,
                         int32_t *idx, float *w) {
    int rc = tqo_router(Wr, bias, E, hidden, x, top_k, NULL, idx, w);
    if (rc) return rc;
    float *o = (float *)malloc(sizeof(float) * (size_t)hidden);
    if (!o) return -5;
    for (int64_t n = 0; n < hidden; n++) out[n] = 0.0f;
    for (int j = 0; j < top_k; j++) {
        int32_t e = idx[j];
        if (!gate[e] || !up[e] || !down[e]) { free(o); return -6; }
        rc = expert_ffn_fmt(fmt, gate[e], up[e], down[e], hidden, inter, x, o,
                            NULL, NULL, NULL, NULL, NULL, NULL);
        if (rc) { free(o); return rc; }
        for (int64_t n = 0; n < hidden; n++) {
            float t = w[j] * o[n];
            out[n] = out[n] + t;
        }
    }
    free(o);
    return 0;
}

int tqo_moe_token(const uint8_t *const *gate, const uint8_t *const *up, const uint8_t *const *down,
                  int64_t E, int64_t hidden, int64_t inter, const float *Wr, const float *bias,
                  int top_k, const float *x, float *out, int32_t *idx, float *w) {
    return moe_token_fmt(0, gate, up, down, E, hidden, inter, Wr, bias, top_k, x, out, idx, w);
}

/* Batched MoE: by definition, each of the T tokens independently through
 * the one-token layer. X, OUT: [T][hidden]; idx, w: [T][top_k]. fmt: the
 * experts' weight format (0 tq2_0_fx4, 1 MXFP4). */
int tqo_moe_tokens_fmt(int fmt, const uint8_t *const *gate, const uint8_t *const *up,
                       const uint8_t *const *down, int64_t E, int64_t hidden, int64_t inter,
                       const float *Wr, const float *bias, int top_k, const float *X, int64_t T,
                       float *OUT, int32_t *idx, float *w) {
    if (fmt != 0 && fmt != 1) return -1;
    for (int64_t t = 0; t < T; t++) {
        int rc = moe_token_fmt(fmt, gate, up, down, E, hidden, inter, Wr, bias, top_k,
                               X + t * hidden, OUT + t * hidden, idx + t * top_k, w + t * top_k);
        if (rc) return rc;
    }
    return 0;
}

int tqo_moe_tokens(const uint8_t *const *gate, const uint8_t *const *up, const uint8_t *const *down,
                   int64_t E, int64_t hidden, int64_t inter, const float *Wr, const float *bias,
                   int top_k, const float *X, int64_t T, float *OUT, int32_t *idx, float *w) {
    return tqo_moe_tokens_fmt(0, gate, up, down, E, hidden, inter, Wr, bias, top_k, X, T, OUT, idx, w);
}

/* Token gather per expert (the grouping step of batched decode/prefill):
 * counts[e] = number of (token, slot) pairs routed to e; offsets = exclusive
 * prefix sum of counts; pairs are listed expert by expert, and within an
 * expert by ascending token (then slot). pair_token, pair_slot: [T*top_k];
 * offsets: [E+1]. Returns 0, or -1 on an index outside 0..E-1. */
int tqo_group_by_expert(const int32_t *idx, int64_t T, int top_k, int64_t E,
                        int32_t *counts, int32_t *offsets, int32_t *pair_token, int32_t *pair_slot) {
    for (int64_t e = 0; e < E; e++) counts[e] = 0;
    for (int64_t i = 0; i < T * top_k; i++) {
        if (idx[i] < 0 || idx[i] >= E) return -1;
        counts[idx[i]]++;
    }
    offsets[0] = 0;
    for (int64_t e = 0; e < E; e++) offsets[e + 1] = offsets[e] + counts[e];
    int64_t p = 0;
    for (int64_t e = 0; e < E; e++)
        for (int64_t t = 0; t < T; t++)
            for (int j = 0; j < top_k; j++)
                if (idx[t * top_k + j] == e) {
                    pair_token[p] = (int32_t)t;
                    pair_slot[p] = j;
                    p++;
                }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Array helpers for the test harness (element-wise, no new arithmetic). */
/* ------------------------------------------------------------------ */
void tqo_f32_to_f16_n(const float *x, int64_t n, uint16_t *h) {
    for (int64_t i = 0; i < n; i++) h[i] = tqo_f32_to_f16(x[i]);
}

void tqo_f16_to_f32_n(const uint16_t *h, int64_t n, float *x) {
    for (int64_t i = 0; i < n; i++) x[i] = tqo_f16_to_f32(h[i]);
}

void tqo_expf_n(const float *z, int64_t n, float *y) {
    for (int64_t i = 0; i < n; i++) y[i] = tqo_expf(z[i]);
}
