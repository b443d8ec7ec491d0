/*
 * tqfx4.h -- C ABI of libtqfx4, the GB300 (sm_103a) implementation of the
 * tq2_0_fx4 integer dot pass and of the mixture-of-experts layers built on it.
 *
 * Paper: "Tied Trit-Planes: Constraining PTQTP to a Uniform Nine-Level
 * Quantizer, with a Persistent Folded Format for Disk-Streamed
 * Mixture-of-Experts Serving" (arXiv 2608.08910).
 *
 *   Sec. 2.1  Tying the two PTQTP scales at alpha = (3s, s) turns the pair of
 *             trit planes t1, t2 in {-1, 0, 1} into one uniform nine-level
 *             code c = 3 t1 + t2 in {-4, ..., 4}, with W_hat = s * c.
 *   Sec. 2.2  tq2_0_fx4 stores c directly: one 520-byte block covers four
 *             columns x 256 elements (512 code bytes, two codes per byte, plus
 *             four f16 column scales), 4.0625 bits/weight. Codes decode by
 *             arithmetic, are dotted against block-quantized activations with
 *             integer arithmetic, and get one float multiply-add per block.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - W is a logical [N][K] fp32 weight (out x in, row-major); y = W x.
 *    N must be a multiple of 4 (TQFX4_ROWS), K a multiple of 256 (TQFX4_QK).
 *  - Block layout (the paper names the parts, not their order; this is the
 *    library's reading): bytes 0..7 are the f16 scales d[0..3] of the block's
 *    four rows, little endian; bytes 8 + 128 r .. 8 + 128 r + 127 hold row r's
 *    codes, byte j carrying element j in its low nibble and element j + 128
 *    in its high nibble. A nibble holds u = c + 4 in 0..8 (9..15 invalid).
 *    A matrix is [N/4 row groups][K/256 blocks] of such blocks, contiguous.
 *  - Activations are quantized per 256-element block: da = absmax / 127,
 *    q = clamp(round(x / da), -127, 127) (x times the binary32 reciprocal of
 *    da, rounded half away from zero), bsum = sum(q).
 *  - The dot pass computes, per row n and block b, the exact integer
 *    S[n][b] = sum_j c[n][256 b + j] q[256 b + j], then
 *    y[n] = sum over b ascending of float(S) * (d[n][b] * da[b]) in binary32
 *    with no fused multiply-add (a fixed float schedule).
 *  - Memory: every pointer argument named as device memory must be device
 *    memory (cudaMalloc or equivalent) owned by the caller. The library
 *    allocates no device memory and keeps no state between calls. Host
 *    structs passed by pointer (tqfx4_experts, tqfx4_router) are read during
 *    the call only.
 *  - Alignment: block arrays 16 bytes; fp32/int32 arrays 4 bytes; int8
 *    activation arrays 16 bytes; the workspace 256 bytes.
 *  - Streams: `stream` is a cudaStream_t (NULL = the legacy default stream).
 *    Every call enqueues its kernels asynchronously on that stream and
 *    returns. Argument errors are detected on the host before anything is
 *    enqueued. Errors found by a kernel (invalid data, a bounded wait that
 *    ran out) are recorded in the status word at the start of the workspace
 *    `ws`; tqfx4_check() synchronizes the stream and reports them.
 *  - Workspace: each call takes `ws`/`ws_bytes`, device memory of at least
 *    the size its *_workspace_bytes query returns (TQFX4_STATUS_BYTES at
 *    least). Zero it once (cudaMemset) before its first use; the library
 *    keeps the status word and its counters consistent after that. Calls
 *    that share a workspace must be ordered on one stream.
 *  - Determinism: no output is produced with atomics; repeated calls on the
 *    same inputs give bit-identical outputs, wherever the data sits in
 *    memory (the "same bytes, same result" property of Sec. 2.2).
 */
#ifndef TQFX4_H
#define TQFX4_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum tqfx4_status {
    TQFX4_OK = 0,
    TQFX4_EINVAL = 1,     /* null pointer, unknown enum value, negative size */
    TQFX4_ESHAPE = 2,     /* N % 4, K % 256, top_k or expert count out of range */
    TQFX4_EALIGN = 3,     /* a pointer violates its alignment rule */
    TQFX4_EWORKSPACE = 4, /* ws smaller than the size query returned */
    TQFX4_ECUDA = 5,      /* a CUDA runtime call or launch failed */
    TQFX4_ETIMEOUT = 6,   /* a kernel's bounded wait ran out (from tqfx4_check) */
    TQFX4_EDATA = 7       /* invalid data seen by a kernel: a trit outside
                             {-1,0,1}, a non-finite weight or activation */
} tqfx4_status;

#define TQFX4_QK 256           /* elements per block along K (Sec. 2.2) */
#define TQFX4_ROWS 4           /* rows ("columns") per block (Sec. 2.2) */
#define TQFX4_BLOCK_BYTES 520  /* 8 scale bytes + 512 code bytes (Sec. 2.2) */
#define TQFX4_STATUS_BYTES 256 /* status area at the start of every workspace */
#define TQFX4_MAX_K 16384      /* largest K (hidden or intermediate size) */
#define TQFX4_MAX_EXPERTS 1024
#define TQFX4_MAX_TOP_K 16

/* Sources for tqfx4_pack. */
#define TQFX4_SRC_TRITS 0   /* fold two trit planes with given f16 scales */
#define TQFX4_SRC_F32_RTN 1 /* round-to-nearest codes from fp32 weights */
#define TQFX4_SRC_F32_TIED 2 /* the tied alternating solver from fp32 weights */
#define TQFX4_TIED_MAX_ITER 64 /* scale updates per block of the tied solver, at most */

/* Paths for tqfx4_moe_grouped. */
#define TQFX4_PATH_AUTO 0    /* the library's choice: PREFILL (measured faster at every batch size) */
#define TQFX4_PATH_DECODE 1  /* per-expert grouped GEMM on integer MMA (weights read once) */
#define TQFX4_PATH_PREFILL 2 /* per-expert grouped GEMM on tensor cores (tcgen05); chunks of at most
                                4 pairs stream through an integer (dp4a) pass instead; results
                                are the same bit for bit on every path */

/* Bytes of one N x K matrix: (N/4) * (K/256) * 520 (Sec. 2.2: 4.0625
 * bits/weight). Returns -1 if N % 4 or K % 256 or a size is negative. */
int64_t tqfx4_matrix_bytes(int64_t n, int64_t k);

/* Workspace bytes for tqfx4_pack, tqfx4_quantize_act and tqfx4_gemv
 * (the status area only). */
size_t tqfx4_basic_workspace_bytes(void);

/*
 * tqfx4_pack -- write blocks for an N x K matrix (Sec. 2.1 fold, Sec. 2.2
 * layout).
 *   src == TQFX4_SRC_TRITS: a = t1 (int8 [n][k], device), t2 = int8 [n][k]
 *     (device), scales_f16 = f16 bit patterns [n][k/256] (device). Each code
 *     is c = 3 t1 + t2. A trit outside {-1, 0, 1} sets TQFX4_EDATA.
 *   src == TQFX4_SRC_F32_RTN: a = W (fp32 [n][k], device); t2 and
 *     scales_f16 must be NULL. Per (row, block): d = f16(absmax / 4)
 *     (round to nearest even, saturated at 65504), c = clamp(round(w /
 *     float(d)), -4, 4) computed as w times the binary32 reciprocal of the
 *     f16-rounded scale, rounded half away from zero; d = 0 gives c = 0. A
 *     non-finite weight sets TQFX4_EDATA.
 *   src == TQFX4_SRC_F32_TIED: a = W as for F32_RTN (t2, scales_f16 NULL).
 *     The tied alternating solver of Sec. 2.1 (the two planes fitted against
 *     one scale s, i.e. W_hat = s * c): per (row, block), starting from the
 *     F32_RTN fit, the scale becomes f16(<w, c> / <c, c>) (binary32; <w, c>
 *     summed as 32 groups of 8 consecutive elements in index order, then the
 *     partials combined pairwise by index XOR 16, 8, 4, 2, 1) and the codes
 *     are recomputed against it as in F32_RTN, until the scale repeats (a
 *     fixed point: the codes are nearest to their own scale, the scale is
 *     the best f16 value for the codes) or TQFX4_TIED_MAX_ITER updates. The
 *     squared error of every block is at most the F32_RTN fit's.
 *   blocks: device, tqfx4_matrix_bytes(n, k) bytes, 16-byte aligned, written
 *     completely. n == 0 or k == 0 writes nothing.
 */
tqfx4_status tqfx4_pack(int src, const void *a, const int8_t *t2, const uint16_t *scales_f16,
                        int64_t n, int64_t k, void *blocks,
                        void *ws, size_t ws_bytes, void *stream);

/*
 * tqfx4_quantize_act -- per-256-block int8 activation quantization (Sec. 2.2,
 * "block-quantized activations"). x: fp32 [m][k] (device). Outputs (device):
 * q int8 [m][k] (16-byte aligned), da fp32 [m][k/256], bsum int32
 * [m][k/256]. A non-finite input sets TQFX4_EDATA.
 */
tqfx4_status tqfx4_quantize_act(const float *x, int64_t m, int64_t k,
                                int8_t *q, float *da, int32_t *bsum,
                                void *ws, size_t ws_bytes, void *stream);

/*
 * tqfx4_validate_blocks -- checks an N x K tq2_0_fx4 matrix against the
 * format (Sec. 2.2): every code nibble u is 0..8 (the nine levels c = u - 4)
 * and every f16 row scale is finite. A violation records TQFX4_EDATA in the
 * status word (tqfx4_check; the detail names a bad block), so a matrix from
 * an outside source can be checked before it is served. The debug build
 * (libtqfx4_debug.so, compiled with TQFX4_DEBUG) runs this check on every
 * matrix the dot-pass entry points read, and checks data-dependent indices
 * inside the kernels. blocks: device, 16-byte aligned.
 */
tqfx4_status tqfx4_validate_blocks(const void *blocks, int64_t n, int64_t k, void *ws, size_t ws_bytes,
                                   void *stream);

/*
 * tqfx4_gemv -- the integer dot pass (Sec. 2.2): y = W x for one activation
 * vector already quantized by tqfx4_quantize_act.
 *   blocks: device, the N x K matrix. q, da, bsum: device, one vector
 *   (k, k/256, k/256 entries). y: fp32 [n] (device).
 *   block_sums: nullable; if given, int32 [n][k/256] (device) receives the
 *   exact integer block sums S[n][b].
 *   k == 0 gives y = 0; n == 0 does nothing.
 */
tqfx4_status tqfx4_gemv(const void *blocks, int64_t n, int64_t k,
                        const int8_t *q, const float *da, const int32_t *bsum,
                        float *y, int32_t *block_sums,
                        void *ws, size_t ws_bytes, void *stream);

/*
 * tqfx4_gemv_x -- tqfx4_quantize_act and tqfx4_gemv in one launch (Sec. 2.2):
 * y = W x for one fp32 vector x, quantized per 256-block inside the kernel
 * with the quantizer of tqfx4_quantize_act, then dotted as tqfx4_gemv does;
 * q, da, bsum and y are the two calls' results bit for bit.
 *   blocks: device, the N x K matrix (16-byte aligned). x: fp32 [k]
 *   (device, 16-byte aligned). y: fp32 [n] (device).
 *   q, da, bsum: all NULL, or device outputs for the quantized vector (k
 *   bytes 16-byte aligned, k/256 and k/256 entries).
 *   k must be a positive multiple of 512 up to TQFX4_MAX_K (the chunked
 *   pass), else TQFX4_ESHAPE; n == 0 does nothing. A non-finite x sets
 *   TQFX4_EDATA.
 */
tqfx4_status tqfx4_gemv_x(const void *blocks, int64_t n, int64_t k, const float *x, float *y,
                          int8_t *q, float *da, int32_t *bsum,
                          void *ws, size_t ws_bytes, void *stream);

/* Workspace bytes for tqfx4_gemv_x_host: the status word, then staging for x
 * and y. 0 for shapes tqfx4_gemv_x refuses. */
size_t tqfx4_gemv_x_host_workspace_bytes(int64_t n, int64_t k);

/*
 * tqfx4_gemv_x_host -- tqfx4_gemv_x with x (fp32 [k]) and y (fp32 [n]) in
 * host memory, ordered on `stream` (Sec. 2.2). Page-locked buffers (x 16-byte
 * and y 4-byte aligned) are used in place through their device addresses:
 * the kernel reads x and writes y directly. Pageable or unaligned ones go
 * through the workspace's staging with one cudaMemcpyAsync each. Returns once
 * enqueued; y is complete after the stream has passed the call. y equals
 * tqfx4_gemv_x's bit for bit. Errors: as tqfx4_gemv_x.
 */
tqfx4_status tqfx4_gemv_x_host(const void *blocks, int64_t n, int64_t k, const float *x_host, float *y_host,
                               void *ws, size_t ws_bytes, void *stream);

/*
 * The free-scale two-plane format (Table 1's free-scale K=2 row, 4.125
 * bits/weight; the ablation of the tie of Sec. 2.1): W = a1 t1 + a2 t2 per
 * row and 256 columns, t1, t2 in {-1, 0, 1}, two independent f16 scales.
 * The pair does not fold, so both trit planes are stored: blocks of 4 rows x
 * 256 columns, 528 bytes, ordered [N/4 row groups][K/256 blocks] like the
 * 520-byte block. Bytes 0..7: a1 of rows 0..3; bytes 8..15: a2 (f16, little
 * endian); row r's plane t1 at bytes 16 + 128 r .. + 63 and plane t2 at the
 * next 64 bytes, element j in bits 2 (j % 4) of byte j / 4 as u = t + 1
 * (u = 3 is invalid). (The paper gives the size, not the byte order.)
 *   tqfx4_free_bytes: (n/4)(k/256) * 528, or -1 unless n % 4 == 0 and
 *     k % 256 == 0.
 *   tqfx4_pack_free: t1, t2 int8 [n][k] (device, 16-byte aligned), a1, a2
 *     f16 bits [n][k/256] (device) -> blocks (device, 16-byte aligned,
 *     caller-allocated). A trit outside {-1, 0, 1} sets TQFX4_EDATA.
 *   tqfx4_gemv_free: y = W x for x quantized by tqfx4_quantize_act (q, da,
 *     bsum). Per (row, 256-block) the exact int32 sums S1 = sum t1 q and
 *     S2 = sum t2 q; y[n] = the binary32 sum in ascending block order of
 *     float(S1) * (a1 * da) + float(S2) * (a2 * da) (each product and sum
 *     rounded once). S1, S2: both NULL or both int32 [n][k/256] (device).
 *     k <= TQFX4_MAX_K.
 */
int64_t tqfx4_free_bytes(int64_t n, int64_t k);
tqfx4_status tqfx4_pack_free(const int8_t *t1, const int8_t *t2, const uint16_t *a1_f16,
                             const uint16_t *a2_f16, int64_t n, int64_t k, void *blocks,
                             void *ws, size_t ws_bytes, void *stream);
tqfx4_status tqfx4_gemv_free(const void *blocks, int64_t n, int64_t k, const int8_t *q,
                             const float *da, const int32_t *bsum, float *y, int32_t *S1,
                             int32_t *S2, void *ws, size_t ws_bytes, void *stream);

/*
 * The MXFP4 arm (Sec. 2.3, the expert-lossless arm): the released expert
 * bytes (4.25 bits/weight in Table 1), served by the integer dot pass with no
 * transcode. Format (OCP microscaling): blocks of 32 consecutive elements of
 * a row, 17 bytes each: byte 0 the e8m0 scale E (2^(E-127); E = 255 is NaN),
 * bytes 1..16 the e2m1 codes (sign, two exponent bits, one mantissa bit:
 * 0, 0.5, 1, 1.5, 2, 3, 4, 6), element j < 16 in the low nibble of byte
 * 1 + j and element 16 + j in the high nibble. A row is k/32 consecutive
 * blocks; rows are consecutive.
 *   tqfx4_mxfp4_bytes: n * (k/32) * 17, or -1 if k is not a multiple of 32.
 *   tqfx4_gemv_mxfp4: y = W x for such a matrix and x quantized by
 *     tqfx4_quantize_act (q int8 [k], da fp32 [k/256]). Per 32-block the
 *     exact int32 sum S = sum c q of the doubled codes c = 2 e2m1 (the
 *     integers 0..12 with a sign) and q, and its exact value
 *     t = float(S) * 2^(E-128) (subnormals kept, inf past the range). Float
 *     schedule, by the activation's 256-element scale unit g: G_g = the
 *     binary32 sum of t over g's eight blocks in ascending order, then y[n]
 *     = the binary32 sum of G_g * da[g] over g ascending (each product and
 *     sum rounded once).
 *     block_sums: nullable int32 [n][k/32] (device) receives S. k must be a
 *     multiple of 512 (rows 16-byte aligned), <= TQFX4_MAX_K; blocks and q
 *     16-byte aligned. A NaN scale sets TQFX4_EDATA.
 */
int64_t tqfx4_mxfp4_bytes(int64_t n, int64_t k);
tqfx4_status tqfx4_gemv_mxfp4(const void *blocks, int64_t n, int64_t k,
                              const int8_t *q, const float *da,
                              float *y, int32_t *block_sums,
                              void *ws, size_t ws_bytes, void *stream);

/*
 * Routed experts: gate and up are [n_experts] stacked matrices of shape
 * inter x hidden, down is [n_experts] stacked matrices of shape hidden x
 * inter, each expert's matrix at base + e * tqfx4_matrix_bytes(...) (one
 * expert-projection is one contiguous byte range, Sec. 1 and 2.2). Device
 * pointers, 16-byte aligned.
 */
typedef struct tqfx4_experts {
    const void *gate;
    const void *up;
    const void *down;
    int64_t n_experts; /* 1 .. TQFX4_MAX_EXPERTS */
    int64_t hidden;    /* multiple of 256, <= TQFX4_MAX_K */
    int64_t inter;     /* multiple of 256, <= TQFX4_MAX_K */
} tqfx4_experts;

/*
 * Router: logits = W_r x + bias, evaluated with a compensated binary32 dot
 * product (Ogita-Rump-Oishi Dot2) and kept as double-binary32 pairs (about
 * 44 significant bits); the top_k experts by logit (ties go to the lower
 * expert index) in descending order; weights = softmax over the selected
 * logits (the renormalized top-k of the full softmax), evaluated in
 * double-binary32 and rounded once to binary32, so they agree with a binary64
 * evaluation. The paper does not describe the router; this is the standard
 * top-k router.
 */
typedef struct tqfx4_router {
    const float *weight; /* [n_experts][hidden] fp32, device */
    const float *bias;   /* nullable [n_experts] fp32, device; added before selection */
    int32_t top_k;       /* 1 .. min(n_experts, TQFX4_MAX_TOP_K) */
} tqfx4_router;

/* Workspace bytes for tqfx4_moe_ffn (tokens == 1, path ignored) or
 * tqfx4_moe_grouped with `tokens` tokens on `path`. Returns 0 if the shapes
 * are invalid. */
size_t tqfx4_moe_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt,
                                 int64_t tokens, int path);

/*
 * tqfx4_moe_ffn -- one token through a routed-expert MoE layer:
 *   route x (fp32 logits, top-k, renormalized weights); quantize x once;
 *   for each selected expert j: g = gate_j x, u = up_j x (dot pass),
 *   h = silu(g) * u, quantize h, o_j = down_j h (dot pass);
 *   out = sum over j in rank order of w_j * o_j (binary32, fixed order).
 * SwiGLU is evaluated in binary32 as g / (1 + exp(-g)) * u with exp computed
 * by Cody-Waite reduction and a degree-7 Taylor polynomial, so that the int8
 * re-quantization of h is reproducible bit for bit.
 * Only the selected experts' blocks are read.
 *   x, out: fp32 [hidden] (device). sel_idx int32 [top_k], sel_w fp32
 *   [top_k] (device) receive the routing decision.
 */
tqfx4_status tqfx4_moe_ffn(const tqfx4_experts *ex, const tqfx4_router *rt,
                           const float *x, float *out, int32_t *sel_idx, float *sel_w,
                           void *ws, size_t ws_bytes, void *stream);

/* Workspace bytes for tqfx4_moe_ffn_host: tqfx4_moe_ffn's layout followed by
 * device staging for x, out and the selection. 0 if the shapes are invalid. */
size_t tqfx4_moe_ffn_host_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt);

/*
 * tqfx4_moe_ffn_host -- tqfx4_moe_ffn for a token in host memory (Sec. 2.2,
 * the serving call with its transfers): x_host (fp32 [hidden]) reaches the
 * workspace's staging, the layer runs, and out (fp32 [hidden]) and, when
 * their pointers are not NULL, sel_idx (int32 [top_k]) and sel_w (fp32
 * [top_k]) reach host memory, all ordered on `stream`. Page-locked host
 * buffers (16-byte aligned x, 4-byte aligned outputs) are used in place
 * through their device addresses: a small kernel reads x and the layer
 * writes out and the selection directly, with no copy-engine transfer.
 * Pageable or unaligned ones go through the staging with one
 * cudaMemcpyAsync each (which makes the call wait for them). The call
 * returns once the work is enqueued: the host buffers must stay valid, and
 * the outputs are complete only after the stream has passed them
 * (synchronize before reading). The results equal tqfx4_moe_ffn's bit for
 * bit. Workspace: tqfx4_moe_ffn_host_workspace_bytes.
 * Errors: as tqfx4_moe_ffn, and TQFX4_EINVAL for a NULL x_host or out_host.
 */
tqfx4_status tqfx4_moe_ffn_host(const tqfx4_experts *ex, const tqfx4_router *rt, const float *x_host,
                                float *out_host, int32_t *sel_idx_host, float *sel_w_host, void *ws,
                                size_t ws_bytes, void *stream);

/*
 * tqfx4_moe_ffn_mxfp4 -- tqfx4_moe_ffn with MXFP4 experts (the
 * expert-lossless arm, Sec. 2.3: the released expert bytes served by the
 * same engine): ex->gate, up and down hold the stacked experts in the MXFP4
 * layout of tqfx4_gemv_mxfp4, each expert projection
 * tqfx4_mxfp4_bytes(rows, cols) contiguous bytes at base + e * that size.
 * Routing, the activation quantizer, SwiGLU and the rank-order combine are
 * tqfx4_moe_ffn's; each projection is tqfx4_gemv_mxfp4's dot pass. hidden
 * and inter must be multiples of 512. Workspace: tqfx4_moe_workspace_bytes
 * with tokens == 1. A NaN scale in a selected expert sets TQFX4_EDATA.
 */
tqfx4_status tqfx4_moe_ffn_mxfp4(const tqfx4_experts *ex, const tqfx4_router *rt,
                                 const float *x, float *out, int32_t *sel_idx, float *sel_w,
                                 void *ws, size_t ws_bytes, void *stream);
/* The same, recording events[0..4] around its stages (router, gate_up,
 * down with SwiGLU and the quantization of h in its prologue, combine:
 * tqfx4_moe_stage_count(2, 0) == 4 and tqfx4_moe_stage_name(2, 0, i)); the
 * stages then run without programmatic dependent launch. */
tqfx4_status tqfx4_moe_ffn_mxfp4_traced(const tqfx4_experts *ex, const tqfx4_router *rt,
                                        const float *x, float *out, int32_t *sel_idx, float *sel_w,
                                        void *ws, size_t ws_bytes, void *stream, void *const *events);

/*
 * tqfx4_moe_route and tqfx4_moe_experts -- tqfx4_moe_ffn in two calls, for
 * callers that place the selected experts' blocks themselves between the
 * routing decision and the expert projections: an expert tier that keeps
 * experts in host memory and copies a missing expert projection, one
 * contiguous range of bytes, into a device slot (the GPU counterpart of the
 * paper's streamed expert store, Sec. 2.2: the same bytes and the same
 * kernels wherever an expert is cached, so the outputs are bitwise the same).
 *   tqfx4_moe_route: routes x as tqfx4_moe_ffn does and writes sel_idx and
 *     sel_w (device, [top_k]); ex->gate/up/down are not read. It also
 *     quantizes x into the workspace for the next call.
 *   tqfx4_moe_experts: the rest of tqfx4_moe_ffn for the token last routed
 *     on this workspace (the two calls must be ordered on one stream, with
 *     no other MoE call on the workspace between them). ptrs: device array
 *     of 3 x top_k device pointers, the gate blocks of the selected experts
 *     in rank order, then their up blocks, then their down blocks, each
 *     16-byte aligned and holding one expert projection
 *     (tqfx4_matrix_bytes of its shape); ex->gate/up/down are not read.
 *   Workspace and out: as for tqfx4_moe_ffn (tqfx4_moe_workspace_bytes with
 *   tokens == 1). The results equal tqfx4_moe_ffn's bit for bit when ptrs
 *   point at bytes equal to the selected experts' blocks.
 */
tqfx4_status tqfx4_moe_route(const tqfx4_experts *ex, const tqfx4_router *rt,
                             const float *x, int32_t *sel_idx, float *sel_w,
                             void *ws, size_t ws_bytes, void *stream);
tqfx4_status tqfx4_moe_experts(const tqfx4_experts *ex, const tqfx4_router *rt,
                               const void *const *ptrs, float *out,
                               void *ws, size_t ws_bytes, void *stream);

/*
 * tqfx4_moe_grouped -- T tokens through the same MoE layer, grouped by
 * expert: route all tokens, count (token, slot) pairs per expert, exclusive
 * scan, stable gather (ascending token order within each expert), run each
 * touched expert once over all of its tokens (its weights are read once),
 * then combine each token's expert outputs in rank order. Results equal
 * tqfx4_moe_ffn applied to each token.
 *   X, OUT: fp32 [T][hidden] (device, 16-byte aligned). sel_idx int32
 *   [T][top_k], sel_w fp32 [T][top_k] (device). T == 0 does nothing. hidden
 *   and inter must be multiples of 512 on this path.
 */
tqfx4_status tqfx4_moe_grouped(const tqfx4_experts *ex, const tqfx4_router *rt,
                               const float *X, int64_t T, float *OUT,
                               int32_t *sel_idx, float *sel_w, int path,
                               void *ws, size_t ws_bytes, void *stream);

/* Workspace bytes for tqfx4_moe_grouped_host with `tokens` tokens on `path`:
 * tqfx4_moe_grouped's layout followed by staging for X, OUT and the
 * selection. 0 if the shapes are invalid or tokens < 1. */
size_t tqfx4_moe_grouped_host_workspace_bytes(const tqfx4_experts *ex, const tqfx4_router *rt, int64_t tokens,
                                              int path);

/*
 * tqfx4_moe_grouped_host -- tqfx4_moe_grouped with X, OUT (fp32 [T][hidden])
 * and, when their pointers are not NULL, sel_idx (int32 [T][top_k]) and
 * sel_w (fp32 [T][top_k]) in host memory, ordered on `stream`. Page-locked
 * buffers (X and OUT 16-byte aligned, the selection 4-byte aligned) are used
 * in place: a copy kernel reads X into the workspace's staging, and the
 * combine and the top-k write OUT and the selection straight into host
 * memory; pageable or unaligned buffers go through the staging with one
 * cudaMemcpyAsync each. Returns once enqueued; the outputs are complete after
 * the stream has passed the call. Results equal tqfx4_moe_grouped's bit for
 * bit. Workspace: tqfx4_moe_grouped_host_workspace_bytes. T == 0 does
 * nothing.
 */
tqfx4_status tqfx4_moe_grouped_host(const tqfx4_experts *ex, const tqfx4_router *rt, const float *X_host,
                                    int64_t T, float *OUT_host, int32_t *sel_idx_host, float *sel_w_host, int path,
                                    void *ws, size_t ws_bytes, void *stream);

/*
 * tqfx4_moe_ffn_noalloc -- tqfx4_moe_ffn without a caller workspace, for
 * callers that cannot allocate device memory: for example a plug-in whose
 * host application owns all device memory through its own allocator and
 * hands it no workspace, or a real-time serving loop in which an allocation
 * (which may block and synchronize the device) is not allowed. The paper
 * has no counterpart; it is a convenience of this library.
 *   Inputs, outputs and their rules are those of tqfx4_moe_ffn. The scratch
 *   is a device array of TQFX4_NOALLOC_SCRATCH_BYTES (1 MiB) inside the
 *   library, which every GPU that loads the library keeps until the process
 *   exits. Shapes whose one-token workspace (the layout tqfx4_moe_ffn uses)
 *   exceeds that size are rejected with TQFX4_EWORKSPACE before anything is
 *   enqueued (the 256-expert, hidden 4096, intermediate 2048, top-8 layer
 *   needs 361 472 bytes, about 0.35 MiB). The call allocates nothing: no
 *   cudaMalloc, no cudaFree.
 *   Every call looks up the scratch's device address in the current context
 *   (cudaGetSymbolAddress; nothing is cached, so a device reset or a
 *   non-primary context is followed). The first call on a device may load
 *   the library's device code there: make it before any stream capture.
 *   Each call clears the scratch's status word and counters on `stream`
 *   before its kernels; device-side error reports therefore are not kept
 *   between calls (use tqfx4_moe_ffn with a workspace and tqfx4_check to
 *   read them).
 *   All calls share the one scratch array, which keeps the last call's
 *   contents: calls whose work overlaps on the GPU (different streams, or
 *   different host threads without ordering) race on it and must not be
 *   issued.
 */
#define TQFX4_NOALLOC_SCRATCH_BYTES (1 << 20)
tqfx4_status tqfx4_moe_ffn_noalloc(const tqfx4_experts *ex, const tqfx4_router *rt,
                                   const float *x, float *out, int32_t *sel_idx, float *sel_w,
                                   void *stream);

/*
 * tqfx4_expert_ffn -- one expert's SwiGLU FFN for one token (Sec. 1 and
 * 2.2; the expert FFN of tqfx4_moe_ffn, without a router): g = W_gate x and
 * u = W_up x through the integer dot pass with x quantized per 256-block,
 * h = silu(g) u quantized per 256-block, out = W_down h. The output, and
 * the intermediates left in the workspace, are bit for bit those of
 * tqfx4_moe_ffn on a one-expert layer (whose routing weight is 1).
 *   gate, up: inter x hidden matrices; down: hidden x inter (device,
 *   16-byte aligned, tqfx4_matrix_bytes each). x: fp32 [hidden] (device,
 *   16-byte aligned); out: fp32 [hidden] (device).
 *   ws: at least tqfx4_expert_ffn_workspace_bytes(hidden, inter) bytes,
 *   zeroed once before its first use (0 for invalid shapes: hidden and
 *   inter positive multiples of 256 up to TQFX4_MAX_K), and zeroed again
 *   after a call that reported TQFX4_ETIMEOUT. A non-finite x or h sets
 *   TQFX4_EDATA.
 *   Launches (tqfx4_expert_ffn_launches tells which): one cooperative
 *   launch of one CTA per SM where the expert fits the SMs' shared memory
 *   and hidden and inter are multiples of 512 (the 4096 x 2048 expert does):
 *   each CTA copies its share of all three matrices on chip at its start,
 *   forms its g, u and h rows, meets the others at a grid-wide barrier
 *   (bounded wait, TQFX4_ETIMEOUT when it runs out), quantizes h and forms
 *   its down rows. Otherwise two launches: gate/up with the quantization
 *   of x inside, then down. tqfx4_expert_ffn_traced records events[0..2]
 *   before, between and after the two (stages "gate_up", "down"); around
 *   the one launch it records events[0] before and events[1] and events[2]
 *   after it.
 */
size_t tqfx4_expert_ffn_workspace_bytes(int64_t hidden, int64_t inter);

/* Kernel launches tqfx4_expert_ffn makes for these shapes on the current
 * device: 1 (the cooperative one-launch kernel) or 2; 0 for invalid shapes. */
int tqfx4_expert_ffn_launches(int64_t hidden, int64_t inter);
tqfx4_status tqfx4_expert_ffn(const void *gate, const void *up, const void *down,
                              int64_t hidden, int64_t inter, const float *x, float *out,
                              void *ws, size_t ws_bytes, void *stream);

/* Workspace bytes for tqfx4_expert_ffn_host: tqfx4_expert_ffn's, then
 * staging for x and out. 0 if the shapes are invalid. */
size_t tqfx4_expert_ffn_host_workspace_bytes(int64_t hidden, int64_t inter);

/*
 * tqfx4_expert_ffn_host -- tqfx4_expert_ffn with x and out (fp32 [hidden])
 * in host memory, ordered on `stream`. A page-locked x (16-byte aligned) is
 * read into the staging by a small kernel and a page-locked out (4-byte
 * aligned) is written in place by the kernel that forms the down rows (the
 * one-launch kernel, or the down kernel of the two); pageable or unaligned
 * buffers go through the staging with one cudaMemcpyAsync each. Returns once
 * enqueued; out is complete after the stream has passed the call. out equals
 * tqfx4_expert_ffn's bit for bit. Errors: as tqfx4_expert_ffn.
 */
tqfx4_status tqfx4_expert_ffn_host(const void *gate, const void *up, const void *down, int64_t hidden,
                                   int64_t inter, const float *x_host, float *out_host, void *ws, size_t ws_bytes,
                                   void *stream);
tqfx4_status tqfx4_expert_ffn_traced(const void *gate, const void *up, const void *down,
                                     int64_t hidden, int64_t inter, const float *x, float *out,
                                     void *ws, size_t ws_bytes, void *stream, void *const *events);

/*
 * Profiling variants: identical to the calls above, and additionally record
 * `events[i]` (cudaEvent_t, created by the caller) on the stream before
 * stage i, and events[n_stages] after the last stage, where n_stages is
 * given by tqfx4_moe_stage_count. Stage names come from
 * tqfx4_moe_stage_name.
 */
int tqfx4_moe_stage_count(int grouped, int path);
const char *tqfx4_moe_stage_name(int grouped, int path, int stage);
tqfx4_status tqfx4_moe_ffn_traced(const tqfx4_experts *ex, const tqfx4_router *rt,
                                  const float *x, float *out, int32_t *sel_idx, float *sel_w,
                                  void *ws, size_t ws_bytes, void *stream, void *const *events);
tqfx4_status tqfx4_moe_grouped_traced(const tqfx4_experts *ex, const tqfx4_router *rt,
                                      const float *X, int64_t T, float *OUT,
                                      int32_t *sel_idx, float *sel_w, int path,
                                      void *ws, size_t ws_bytes, void *stream,
                                      void *const *events);

/*
 * Byte offsets, from the start of the workspace, of the intermediates a MoE
 * call leaves there (for inspection and tests; valid after the call's
 * stream work completes). Entries that a path does not produce are
 * SIZE_MAX. P = T * top_k (token, slot) pairs; pairs are ordered by expert
 * then token for the grouped call, by rank for tqfx4_moe_ffn.
 */
typedef struct tqfx4_moe_views {
    size_t logits;     /* fp32 [T][n_experts]: high part of each logit */
    size_t logits_lo;  /* fp32 [T][n_experts]: low part (logit = hi + lo exactly) */
    size_t qx;         /* int8 [T][hidden] */
    size_t dx;         /* fp32 [T][hidden/256] */
    size_t bx;         /* int32 [T][hidden/256] */
    size_t g;          /* fp32 [P][inter] */
    size_t u;          /* fp32 [P][inter] */
    size_t h;          /* fp32 [P][inter] */
    size_t qh;         /* int8 [P][inter] */
    size_t dh;         /* fp32 [P][inter/256] */
    size_t bh;         /* int32 [P][inter/256] */
    size_t o;          /* fp32 [P][hidden]: each pair's expert output */
    size_t counts;     /* int32 [n_experts] (grouped only) */
    size_t offsets;    /* int32 [n_experts + 1] (grouped only) */
    size_t pair_token; /* int32 [P] (grouped only) */
    size_t pair_slot;  /* int32 [P] (grouped only) */
    size_t pair_of;    /* int32 [T][top_k]: position of each (token, slot) pair (grouped only) */
} tqfx4_moe_views;

tqfx4_status tqfx4_moe_workspace_views(const tqfx4_experts *ex, const tqfx4_router *rt,
                                       int64_t tokens, int grouped, int path,
                                       tqfx4_moe_views *views);

/*
 * tqfx4_check -- synchronize `stream`, read the status word in `ws` and
 * clear it. Returns TQFX4_OK, the first device-side error recorded since
 * the last check (TQFX4_EDATA, TQFX4_ETIMEOUT), or TQFX4_ECUDA if the
 * stream reports a CUDA error.
 */
tqfx4_status tqfx4_check(void *ws, void *stream);

/*
 * tqfx4_selftest_wait_timeout -- a check of the library's failure detection
 * that faults nothing: one warp runs the streaming engine's consume loop
 * (the loop under the GEMV and MoE kernels) on a ring whose copies were
 * never issued, with a wait budget of 10^6 cycles instead of the production
 * limit of about two seconds. Its wait gives up, the warp records
 * TQFX4_ETIMEOUT in the status word of `ws` (kernel "selftest") and the
 * kernel returns; no copy is in flight, so the context stays usable.
 * tqfx4_check(ws, stream) then returns TQFX4_ETIMEOUT and clears the word.
 * ws: device, at least TQFX4_STATUS_BYTES. Not part of the paper's method.
 */
tqfx4_status tqfx4_selftest_wait_timeout(void *ws, size_t ws_bytes, void *stream);

/* Message for the last error returned on the calling host thread. */
const char *tqfx4_last_error(void);
const char *tqfx4_status_string(tqfx4_status s);

#ifdef __cplusplus
}
#endif

#endif /* TQFX4_H */
