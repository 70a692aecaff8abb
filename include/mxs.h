/*
 * mxs.h -- C ABI of libmxs, the MXINT mixed-precision linear layer of MXSens
 * (arxiv 2607.17733) for NVIDIA GB300 (sm_103a).
 *
 * The layer computes y = x W^T where the activations x [M,K] (bf16) and the
 * weights W [N,K] (bf16) are both quantized to MXINT: every block of 32
 * consecutive values along K shares one power-of-two scale and holds fixed-point
 * integer mantissas of 4, 6 or 8 bits (Sec. 2, Sec. 4.1).  The width of each
 * K-block comes from a per-layer map (the paper's Alg. 3 allocation, produced
 * offline).  The quantization rules the paper leaves open are read from the OCP
 * MX MXINT definition it cites:
 *   scale byte S = clamp(floor(log2 max|x|), -127, 127) + 127 (E8M0);
 *   element m = clamp(round(x * 2^(b-2-E)), -(2^(b-1)-1), 2^(b-1)-1),
 *   value = m * 2^(E-(b-2)); rounding ties-to-even (MXS_RNE) or away from
 *   zero (MXS_RHAZ); a block with a NaN/Inf gets S = 255 and zero codes.
 * The GEMM returns fp32 y[m,n] = sum_blocks 2^(Ea'+Ew') * (exact integer dot
 * of the two blocks), E' = E-(b-2), accumulated in fp32.
 *
 * Conventions (all entry points):
 *   - Return MXS_OK (0) or a positive MXS_ERR_* code; never abort, never print.
 *     mxs_last_error() gives a thread-local message for the last failure.
 *   - Sizes are int64_t; K must be a positive multiple of 32 and at most
 *     MXS_MAX_K; M, N >= 1 (M = 0 is accepted and does nothing).
 *   - `bits` is a HOST array of K/32 bytes, each 4, 6 or 8, read during the
 *     call.  Blocks are stored grouped by width: slot s < n4 holds the s-th
 *     4-bit block, then the 6-bit blocks, then the 8-bit ones, each group in
 *     increasing block order.
 *   - Every other pointer is DEVICE memory owned by the caller; the library
 *     allocates nothing.  Buffers must be 16-byte aligned unless stated.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued asynchronously; device pointers must stay
 *     valid until the stream reaches it.  Errors raised while the kernels run
 *     surface at the caller's next synchronisation.
 *   - Outputs are overwritten in full, padding rows and slots included; only
 *     the alignment gaps between the sections of an activation planes buffer
 *     and the scale-tile bytes of its rows beyond M (which no GEMM reads) are
 *     left unwritten.
 *   - Kernels use programmatic dependent launch: mxs_quantize_act and
 *     mxs_linear_decode may start before the preceding work on `stream` has
 *     finished and wait for it before they touch their inputs and outputs.
 *     The one exception is stated at mxs_linear_decode (its weights).
 *   - Only sm_103a devices are supported (MXS_ERR_UNSUPPORTED otherwise).
 *
 * Storage format (the "packed" layouts; byte offsets are exact):
 *   Activation codes, per row m (row_bytes = 16*n4 + 32*(n6+n8)):
 *     4-bit slot s: bytes [16s, 16s+16), element i in byte i/2 (low nibble for
 *     even i), two's complement; 6/8-bit slot s: bytes [16*n4 + 32(s-n4), +32),
 *     one int8 per element.  Activation scales: uint8 [M, K/32] by slot.
 *   Weight buffer (layout MXS_W_COMPACT): codes are sign-magnitude, a 4-bit
 *     code as (sign<<3)|m and a 6/8-bit code as (sign<<7)|m (the symmetric
 *     clamp never yields -2^(b-1)); rows are padded to a multiple of 128 and
 *     cut into groups of 128 rows; group g is GB = 2176*n4 + 4224*(n6+n8)
 *     contiguous bytes at g*GB, so any K range of a group is one copy:
 *       4-bit slot s at 2176*s: 128 rows x 16 code bytes (row r at 16r; byte
 *         4i+j holds element 8i+j in the low nibble, 8i+4+j in the high
 *         nibble), then the rows' 128 scale bytes;
 *       6/8-bit slot n4+j at 2176*n4 + 4224*j: 128 rows x 32 code bytes
 *         (row r at 32r, byte e = element e), then 128 scale bytes.
 *     Compact size = align256(G*GB); scale bytes of padding rows are 0.
 *   MMA planes (layout MXS_W_COMPACT_AND_PLANES for weights, the `planes`
 *     output of mxs_quantize_act for activations), Kp = 128*(ceil(n4/4) +
 *     ceil((n6+n8)/2)):
 *       P [rows, Kp]: 4-bit slot s at bytes [32s, +32) = e4m3 m/4; padding
 *       to a multiple of 4 slots is zero; 6/8-bit slot j at 64 bytes from
 *       128*ceil(n4/4)+64j: element i at +2i is the bf16 value
 *       m*2^(S-127-(b-2)) (exact), 0x7FC0 (NaN) in a block with S = 255
 *       (for weights and activations of every M: the operand of both GEMMs).
 *       SF at align256(P + rows*Kp): per 128-row tile and 128-byte K' stage,
 *       512 B ordered [i<32][w<4][q<4] = S of row 128*tile+32w+i, slot 4*st+q
 *       (4-bit stages) or 2*(st-ceil(n4/4))+q for q<2 (6/8-bit stages); every
 *       other byte 0 (for activations: every other byte of the rows < M).
 *     For weights P and SF follow the compact part inside the same buffer.
 */
#ifndef MXS_H_
#define MXS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define MXS_API __attribute__((visibility("default")))
#else
#define MXS_API
#endif

#define MXS_VERSION 3
#define MXS_MAX_K 65536 /* K/32 <= 2048 blocks */

enum mxs_status {
    MXS_OK = 0,
    MXS_ERR_INVALID_ARG = 1, /* NULL pointer, bad enum, bad leading dimension */
    MXS_ERR_SHAPE = 2,       /* K not a positive multiple of 32, K > MXS_MAX_K, M/N < 0 */
    MXS_ERR_BITS = 3,        /* a map entry outside {4, 6, 8} */
    MXS_ERR_ALIGN = 4,       /* a device pointer not 16-byte aligned */
    MXS_ERR_BUFFER = 5,      /* a caller buffer smaller than required */
    MXS_ERR_CUDA = 6,        /* a CUDA runtime call failed (message has the name) */
    MXS_ERR_TIMEOUT = 7,     /* a kernel gave up waiting (see mxs_device_status) */
    MXS_ERR_UNSUPPORTED = 8  /* not an sm_103a device, or a feature not built */
};

enum mxs_rounding { MXS_RNE = 0, MXS_RHAZ = 1 };
enum mxs_weight_layout { MXS_W_COMPACT = 0, MXS_W_COMPACT_AND_PLANES = 1 };

/* Thread-local description of the last failure of a call on this thread. */
MXS_API const char *mxs_last_error(void);
/* MXS_VERSION of the built library. */
MXS_API int mxs_version(void);

/* ---------------------------------------------------------------- sizes
 * Bytes the caller must provide.  They touch no device and return a negative
 * mxs_status (e.g. -MXS_ERR_BITS) for invalid arguments.  The storage they
 * count is the paper's: b bits per element for a b-bit block (one width per
 * 32-element block, Sec. 4.1) plus one 8-bit shared exponent per block, i.e.
 * +0.25 bit per element (Sec. 5.1), laid out as the format above.
 *   mxs_act_row_bytes    code bytes of one activation row: 16*n4 + 32*(n6+n8)
 *   mxs_act_codes_bytes  M rows of codes (the scales are a separate [M, K/32])
 *   mxs_act_planes_bytes activation MMA planes + scale tiles, one buffer with
 *                        the tiles at align256(M*Kp)
 *   mxs_weight_bytes     the weight buffer of mxs_pack_weight for `layout`
 *   mxs_gemm_workspace_bytes  scratch of mxs_gemm / mxs_gemm_decode (0 for
 *                        the current kernels; kept so callers need not change
 *                        if a kernel ever needs one) */
MXS_API int64_t mxs_act_row_bytes(int64_t K, const uint8_t *bits);
MXS_API int64_t mxs_act_codes_bytes(int64_t M, int64_t K, const uint8_t *bits);
MXS_API int64_t mxs_act_planes_bytes(int64_t M, int64_t K, const uint8_t *bits);
/* Workspace of mxs_linear_decode (and of each problem of
 * mxs_linear_decode_group) for M tokens, K columns, N output rows: for M = 1
 * the CUDA-core path's arrival counters (8 bytes per 128 rows) and partial
 * sums (256 KiB); otherwise mxs_act_planes_bytes(M, K, bits).  Negative
 * error code on bad arguments. */
MXS_API int64_t mxs_linear_decode_workspace_bytes(int64_t M, int64_t K, int64_t N, const uint8_t *bits);
MXS_API int64_t mxs_weight_bytes(int64_t N, int64_t K, const uint8_t *bits, int layout);
MXS_API int64_t mxs_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K, const uint8_t *bits);

/* ---------------------------------------------------------------- A1: activation quantization
 * Quantizes x (bf16 [M,K], row stride ld_x elements, ld_x >= K and a multiple
 * of 8) block by block with widths `bits` (Sec. 4.1 one width per block;
 * Appendix A.2 activations quantized on the fly) and writes
 *   codes  [M, mxs_act_row_bytes]  packed codes (may be NULL)
 *   scales [M, K/32]               scale bytes by slot (NULL iff codes NULL)
 *   planes mxs_act_planes_bytes    MMA planes + scale tiles (may be NULL)
 * At least one of codes / planes must be non-NULL. */
MXS_API int mxs_quantize_act(const void *x_bf16, int64_t M, int64_t K, int64_t ld_x,
                     const uint8_t *bits, int rounding,
                     void *codes, uint8_t *scales, void *planes, void *stream);

/* ---------------------------------------------------------------- A2: weight packing (offline)
 * The paper quantizes the weights of every linear layer with the same MXINT
 * rule as the activations (Appendix A.2), under the layer's one width map
 * (Sec. 4.1), and stores each block at its width plus the 8-bit exponent
 * (Sec. 5.1).  Quantizes W (bf16 [N,K] row stride ld_w >= K, a multiple of 8;
 * the nn.Linear convention) with those rules and writes the weight buffer
 * (mxs_weight_bytes(N,K,bits,layout) bytes, caller-allocated device memory,
 * fully overwritten).  Run once per layer, offline.  Errors: MXS_ERR_SHAPE,
 * MXS_ERR_BITS, MXS_ERR_INVALID_ARG (NULL, rounding, layout, ld_w),
 * MXS_ERR_ALIGN (w, packed), MXS_ERR_CUDA. */
MXS_API int mxs_pack_weight(const void *w_bf16, int64_t N, int64_t K, int64_t ld_w,
                    const uint8_t *bits, int rounding, int layout,
                    void *packed, void *stream);

/* ---------------------------------------------------------------- A3/A4: GEMM
 * The MXINT product (Sec. 2): within a block the integer mantissas multiply
 * and add exactly under the two shared scales, and the blocks' terms
 * 2^(Ea'+Ew') * D add up to y; the widths come one per block (Sec. 4.1).
 * y [M,N] fp32 (row stride ld_y >= N, elements) = x W^T over the quantized
 * operands.  act_bits must equal w_bits: the paper's Alg. 3 returns one
 * column allocation per linear layer, derived from one Hessian diagonal that
 * serves both operands (Sec. 3.1), so one map applies to W and A; maps that
 * differ return MXS_ERR_UNSUPPORTED.  `w_layout` is the layout W was packed
 * with.
 * mxs_gemm picks the decode kernel for M <= 16 (over act_planes when given,
 * else over codes/scales) and the tensor-core prefill kernel otherwise (needs
 * act_planes and a weight packed with MXS_W_COMPACT_AND_PLANES).  workspace may be NULL when
 * mxs_gemm_workspace_bytes() is 0. */
MXS_API int mxs_gemm(const void *act_codes, const uint8_t *act_scales, const void *act_planes,
             const uint8_t *act_bits, const void *packed_w, int w_layout, const uint8_t *w_bits,
             int64_t M, int64_t N, int64_t K, float *y, int64_t ld_y,
             void *workspace, size_t ws_bytes, void *stream);

/* Decode path only (M <= 16): weights streamed once from the compact layout by
 * bulk copies into shared memory, converted there to exact e4m3 values
 * (4-bit blocks, on the block-scaled FP8 MMA) or bf16 values (6/8-bit blocks,
 * on the bf16 MMA) and multiplied on the tensor cores (tcgen05, fp32
 * accumulation in tensor memory); when K is split over a thread-block cluster the partial
 * tiles are added in rank order.  The activations are given EITHER as packed
 * codes + scales (act_planes NULL) OR as the MMA planes written by
 * mxs_quantize_act (codes and scales NULL; faster: the operand is loaded by
 * TMA instead of being rebuilt by every CTA).  Needs no workspace (ws may be
 * NULL).  Waits inside the kernel are bounded like the prefill kernel's. */
MXS_API int mxs_gemm_decode(const void *act_codes, const uint8_t *act_scales, const void *act_planes,
                    const uint8_t *bits, const void *packed_w, int64_t M, int64_t N, int64_t K,
                    float *y, int64_t ld_y, void *workspace, size_t ws_bytes, void *stream);

/* A1 + A4 for one linear layer at decode (M <= 16): y [M,N] fp32 = x W^T
 * like mxs_gemm_decode, x bf16 [M,K] (row stride ld_x elements) quantized
 * on the fly with `bits` and `rounding` (Appendix A.2: activations are
 * quantized on the fly).  `workspace`: device, 16-byte aligned, at least
 * mxs_linear_decode_workspace_bytes(M, K, N, bits) bytes, any prior contents.
 *   M = 1: one kernel.  Its prologue quantizes x (the rule of
 *     mxs_quantize_act) and its CUDA cores form the integer block dots from
 *     the packed codes.  Every CTA streams an equal share of the weight bytes;
 *     the CTAs that share a 128-row group leave their partial sums and a
 *     tagged arrival count in the workspace, and the last to arrive adds the
 *     partials in a fixed order (results do not depend on timing).
 *   M > 1: the quantizer writes the activations' MMA planes into the
 *     workspace (the planes mxs_quantize_act writes), then the tensor-core
 *     GEMM reads them.
 * The GEMM is launched as a programmatic dependent of the kernel before it,
 * so its weight stream starts while the activations are produced -- in a
 * chain of such calls, while the previous layer finishes.  Hence packed_w
 * must not be written by work that is still in flight on `stream` when the
 * call is made (weights are static; pack them, then synchronise, before the
 * first use).  x, y and the workspace have the ordinary stream semantics; the
 * workspace may be reused by the next call on the same stream (two calls in
 * flight at once on one workspace race).  After MXS_ERR_TIMEOUT
 * (mxs_device_status) a workspace may hold a partial count of the failed
 * call: rewrite it (e.g. zero it) before it serves a CUDA graph that replays
 * the failed call. */
MXS_API int mxs_linear_decode(const void *x_bf16, int64_t M, int64_t K, int64_t ld_x, const uint8_t *bits,
                              int rounding, const void *packed_w, int64_t N, float *y, int64_t ld_y,
                              void *workspace, size_t ws_bytes, void *stream);

/* mxs_linear_decode for callers that cannot allocate device memory (an
 * allocator-free runtime that owns all device memory, a plug-in whose host
 * forbids allocation on its hot path, a real-time loop that must not block in
 * the allocator).  The paper has no counterpart.  Same arguments, results
 * and launches as mxs_linear_decode, but the activation planes live in a
 * fixed 2 MiB array inside the library (a __device__ variable every GPU that
 * loads the library holds until exit) instead of a caller workspace; the call
 * allocates nothing.  Sizes whose workspace exceeds 2 MiB
 * (mxs_linear_decode_workspace_bytes(M, K, N, bits) > 2 MiB; M <= 16 fits
 * for K <= 49152 with any map, M = 1 for N up to about 29 million) return
 * MXS_ERR_BUFFER.  The first call on each device looks
 * up the array's device address (cudaGetSymbolAddress, current device) and
 * keeps it for the life of the process: make that first call before any
 * stream capture, and do not reset the device (cudaDeviceReset, or anything
 * else that destroys its primary context) after it, since the kept address
 * would then be stale.  All calls share the one
 * array and leave their planes in it: calls ordered on one stream are safe
 * (each waits for the one before it as mxs_linear_decode does), calls that
 * overlap on the GPU (other streams, other host threads) race and give wrong
 * results.  Nothing in the array has to start at zero: every byte the GEMM
 * reads is written by the same call (the one-token path's arrival counts are
 * tagged per call). */
MXS_API int mxs_linear_decode_noalloc(const void *x_bf16, int64_t M, int64_t K, int64_t ld_x, const uint8_t *bits,
                                      int rounding, const void *packed_w, int64_t N, float *y, int64_t ld_y,
                                      void *stream);

/* Prefill path only (M > 16; MXS_ERR_SHAPE for 1 <= M <= 16, whose planes
 * hold the decode form): the tensor-core kernel over the MMA planes of the
 * activations (mxs_quantize_act `planes`) and of the weights (packed with
 * MXS_W_COMPACT_AND_PLANES).  The mixed widths run on fixed-width tensor
 * cores in exact forms accumulated into one fp32 accumulator: 4-bit blocks as
 * e4m3 m/4 on the block-scaled FP8 MMA (UE8M0 scale per 32 elements, one MMA
 * per block), 6/8-bit blocks as their bf16 values on the bf16 MMA (two K=16
 * MMAs per block).  Waits inside the kernel are bounded (about 2 s); on
 * expiry it records MXS_ERR_TIMEOUT (see mxs_device_status). */
MXS_API int mxs_gemm_prefill(const void *act_planes, const uint8_t *bits, const void *packed_w,
                             int64_t M, int64_t N, int64_t K, float *y, int64_t ld_y, void *stream);

/* ---------------------------------------------------------------- status
 * Kernels that wait on barriers give up after a bounded number of polls and
 * record MXS_ERR_TIMEOUT in a per-device status word instead of hanging.
 * Reads that word for the current device after synchronising `stream`;
 * clears it when reset != 0. */
MXS_API int mxs_device_status(int *status, int reset, void *stream);

/* Test hook for the bounded waits: mxs_gemm_prefill, except that the
 * producer never loads K' stage `stage` (1-based), so the MMA warp's wait for
 * it runs out; the kernel then records MXS_ERR_TIMEOUT, drains what it issued,
 * frees its tensor memory and returns (y is left partly unwritten).  No
 * device fault or hang is involved; the context stays usable. */
MXS_API int mxs_test_prefill_starve(const void *act_planes, const uint8_t *bits, const void *packed_w,
                                    int64_t M, int64_t N, int64_t K, float *y, int64_t ld_y, int stage,
                                    void *stream);

/* Test hook for the decode kernel's bounded waits (failure handling of this
 * library; the paper has no counterpart): mxs_gemm_decode over
 * activation planes (M in 1..16), except that every CTA skips the weight copy
 * of its copy chunk `chunk` (1-based, in the CTA's streaming order), so the
 * converter warps' wait for it runs out.  Each CTA then records
 * MXS_ERR_TIMEOUT, stops its quads, waits (bounded) for what it issued and for
 * any slices its cluster partners sent it, frees its tensor memory and
 * returns; y is left partly unwritten.  No device fault or hang is involved;
 * the context stays usable.  Errors as mxs_gemm_decode, MXS_ERR_INVALID_ARG
 * for chunk < 1. */
MXS_API int mxs_test_decode_starve(const void *act_planes, const uint8_t *bits, const void *packed_w, int64_t M,
                                   int64_t N, int64_t K, float *y, int64_t ld_y, int chunk, void *stream);

/* Test hook for the bounded waits of the two kernels mxs_linear_decode(_group)
 * runs (failure handling of this library; the paper has no counterpart):
 * arms the next launch of kernel 1 (the one-token CUDA-core GEMM, M = 1) or
 * kernel 2 (the tensor-core GEMM for 2..16 tokens) so that every CTA skips
 * the weight copy of its stage `stage` (1-based, in the CTA's streaming
 * order; 0 disarms).  The consumers' wait for that stage runs out after ~2 s;
 * each such CTA records MXS_ERR_TIMEOUT (mxs_device_status), stops its
 * arithmetic, waits (bounded) for the copies it issued, frees its tensor
 * memory and returns; y is left partly unwritten.  CTAs with fewer stages
 * finish normally.  The arming is process-wide and taken by that one launch.
 * No device fault or hang is involved; the context stays usable.
 * MXS_ERR_INVALID_ARG for another kernel number or stage < 0. */
MXS_API int mxs_test_decode_arm_starve(int kernel, int stage);

/* Test hook: the one-token decode kernel's ring of weight stages.  stages =
 * 2 or 3 caps it at that many stages for the calls that follow in this
 * process (the kernel drops to fewer than four by itself only when a CTA's
 * token codes need the shared memory: long K over several row groups);
 * 0 restores the choice by size.  MXS_ERR_INVALID_ARG for other values. */
MXS_API int mxs_test_gemv_ring(int stages);

/* Test hook (host only, no device): the one-token decode path's work split
 * for `count` (1..3) problems of K[i] columns, width map bits[i] and N[i]
 * rows on `sms` SMs.  Writes each problem's CTA count to ncta[i] and, for
 * every CTA in launch order, four ints to spans (room for 4 * 256): its first
 * 128-row group, the first slot (32-element block, in the plan's slot order)
 * it takes there, its last group, and the slot where it stops there (the
 * group's block count when it takes the group to its end).  The ranges are
 * balanced by weight: a 6/8-bit slot weighs its 4224 bytes, a 4-bit slot
 * 2176 bytes times the build's weight (mxs_test_dtc_split_weight).  Returns
 * the number of CTAs, or minus an error code. */
MXS_API int mxs_test_gemv_split(const int64_t *K, const uint8_t *const *bits, const int64_t *N, int count, int sms,
                                int32_t *ncta, int32_t *spans);

/* Test hook (host only, no device): the same for the tensor-core decode path
 * (2..16 tokens), whose ranges are cut at plane-stage boundaries (four 4-bit
 * slots, two 6/8-bit slots, the end of the 4-bit run, the group's end) and
 * balanced by weight: a 4-bit slot weighs its 2176 bytes, a 6/8-bit slot
 * 4224 bytes times the build's weight (mxs_test_dtc_split_weight). */
MXS_API int mxs_test_dtc_split(const int64_t *K, const uint8_t *const *bits, const int64_t *N, int count, int sms,
                               int32_t *ncta, int32_t *spans);

/* The split weights of this build, in percent: a 6/8-bit slot's in the
 * tensor-core decode split (returned) and a 4-bit slot's in the one-token
 * split (*cost4, if not NULL). */
MXS_API int mxs_test_dtc_split_weight(int *cost4);

/* mxs_quantize_act_permuted / mxs_pack_weight_permuted -- the layer's
 * columns in the order of the allocation (Alg. 3 returns column lists, and the
 * 32 most sensitive columns form one 8-bit block only once they are placed
 * together, Sec. 4.1): mxs_quantize_act and mxs_pack_weight of x[:, perm] and
 * w[:, perm], i.e. position p of the quantized row holds source column
 * perm[p].  perm: device int32 [K], 16-byte aligned, a permutation of
 * 0..K-1 (mxs_allocate_layer writes one); values outside [0, K) give
 * unspecified results (they are clamped, never read outside the row).  The
 * GEMMs then run unchanged on the outputs: y = x W^T does not depend on the
 * order of the K terms.  Other arguments, layouts and errors as in
 * mxs_quantize_act / mxs_pack_weight (plus MXS_ERR_INVALID_ARG for a NULL
 * perm, MXS_ERR_ALIGN for an unaligned one).  The gather reads 2 bytes per
 * element (the rows are read through the L1/L2 caches). */
MXS_API int mxs_quantize_act_permuted(const void *x_bf16, int64_t M, int64_t K, int64_t ld_x, const int32_t *perm,
                                      const uint8_t *act_bits, int rounding, void *codes, uint8_t *scales,
                                      void *planes_or_null, void *stream);
MXS_API int mxs_pack_weight_permuted(const void *w_bf16, int64_t N, int64_t K, int64_t ld_w, const int32_t *perm,
                                     const uint8_t *w_bits, int rounding, int layout, void *packed, void *stream);

/* mxs_linear_decode_group -- up to three decode layers in one launch: the
 * projections of a decoder layer that share an input (q, k and v; gate and
 * up) each run exactly as mxs_linear_decode (own activations, width map,
 * weights, output and planes workspace), but their GEMMs are one kernel
 * launch: the set-up, the wait for the activations and the teardown are paid
 * once, and the CTAs are shared out among the problems by their weight bytes.
 * The activations of all problems are quantized first, in one quantizer
 * launch, then the grouped GEMM runs as its programmatic dependent.
 * Same operands, layouts and contract as mxs_linear_decode (weights static;
 * 1 <= count <= 3; M <= 16, the same for every problem); every problem needs
 * its own workspace (mxs_linear_decode_workspace_bytes(M, K, N, bits) bytes).  The K split of
 * a problem may differ from its single launch, so results agree with
 * mxs_linear_decode to fp32 rounding, not bit for bit.  Errors as
 * mxs_linear_decode, per problem (the message names it). */
typedef struct mxs_decode_problem {
    const void *x;         /* device, bf16 [M, K], row stride ld_x */
    int64_t K, ld_x;
    const uint8_t *bits;   /* host, K/32 widths */
    const void *packed_w;  /* device, compact layout (mxs_pack_weight) */
    int64_t N;
    float *y;              /* device, fp32 [M, N], row stride ld_y */
    int64_t ld_y;
    void *workspace;       /* device, the activation planes of this problem */
    size_t ws_bytes;
} mxs_decode_problem;
MXS_API int mxs_linear_decode_group(const mxs_decode_problem *probs, int count, int64_t M, int rounding, void *stream);
/* mxs_quantize_act_group -- A1 (the activations of every linear layer are
 * quantized on the fly, Appendix A.2; one width per 32-element block, Sec.
 * 4.1) for up to three activations with M rows each (the inputs of linear
 * layers that read the same hidden state: q, k and v; gate and up), each with
 * its own width map, in one kernel launch: byte for byte what
 * mxs_quantize_act(x_i, M, K_i, ld_i, bits_i, rounding, NULL, NULL, planes_i)
 * writes, one link in the launch chain instead of one per layer.
 * planes_i: device, at least mxs_act_planes_bytes(M, K_i, bits_i) bytes
 * (planes_bytes_i says how many the caller has), 16-byte aligned, distinct
 * buffers.  1 <= count <= 3.  Asynchronous on `stream`
 * (programmatic dependent launch as mxs_quantize_act); allocates nothing.
 * Errors as mxs_quantize_act, per problem (the message names it). */
typedef struct mxs_quant_problem {
    const void *x;         /* device, bf16 [M, K], row stride ld_x (>= K, a multiple of 8) */
    int64_t K, ld_x;
    const uint8_t *bits;   /* host, K/32 widths */
    void *planes;          /* device, the MMA planes + scale tiles */
    size_t planes_bytes;   /* size of `planes`; MXS_ERR_BUFFER below mxs_act_planes_bytes(M, K, bits) */
} mxs_quant_problem;
MXS_API int mxs_quantize_act_group(const mxs_quant_problem *probs, int count, int64_t M, int rounding, void *stream);

/* ---------------------------------------------------------------- KV cache
 * The paper quantizes the KV cache too, with a 4-8 bit configuration
 * (Appendix A.2).  A cache is two code buffers in the activation layout of
 * mxs_quantize_act: row t holds token t's K (or V) values of all KV heads,
 * H_kv * D of them, quantized along the row with that cache's width map
 * (codes [T_max, mxs_act_row_bytes(H_kv * D, bits)], scales [T_max, H_kv*D/32]).
 * Appending token t is one mxs_quantize_act call of M = 1 row into row t.
 *
 * mxs_attention_decode_batch -- one decode step of B sequences: sequence b
 * owns cache rows [b * T_cap, b * T_cap + T_b) and has one query token; for
 * its query head h (reading KV head h / (H / H_kv)),
 *   out[b][h] = sum_t softmax_t(scale * <q[b][h], k_t>) * v_t,   t < T_b,
 * with k_t, v_t the MXINT element values of the cache (code * 2^(S-127-(b-2))).
 *   q        device, bf16 [B, H, D], row-major
 *   k_*, v_* device code rows and scales as above, B * T_cap rows each (code
 *            buffers 16-byte aligned); k_bits, v_bits host width maps of
 *            H_kv * D / 32 entries
 *   lengths  device int32 [B] (4-byte aligned): T_b, clamped to [0, T_cap];
 *            NULL means every sequence has T_cap tokens.  A sequence of
 *            length 0 gets zeros.
 *   out      device, fp32 [B, H, D], 16-byte aligned
 *   workspace device, mxs_attention_decode_batch_workspace_bytes(B, T_cap, H, D)
 *            bytes, 16-byte aligned.  Its first bytes hold arrival counters
 *            that must be zero when the call starts and are zero again when
 *            its kernel ends: zero the workspace once after allocating it
 *            (and again before using it with other sizes).  The rest holds
 *            per-split partial sums, overwritten.
 * D is 64 or 128, H a multiple of H_kv with H / H_kv <= 8, H_kv * D <= 8192,
 * 1 <= B <= 65535, 1 <= T_cap < 2^31.  Scores and weighted sums run on the
 * tensor cores in bf16 with fp32 accumulation: the cache elements are exact in
 * bf16, so every score product is exact; the softmax weights enter as a sum
 * of two bf16 terms (relative error <= 2^-18).  Splits of a sequence and the
 * warps within a split are combined in a fixed order: deterministic for given
 * sizes on a given GPU.  A cache block with scale 255 (NaN/Inf when written)
 * makes the heads that read it NaN.  Asynchronous on `stream`; allocates
 * nothing.  Errors: MXS_ERR_UNSUPPORTED (D), MXS_ERR_SHAPE, MXS_ERR_BITS,
 * MXS_ERR_INVALID_ARG, MXS_ERR_ALIGN, MXS_ERR_BUFFER, MXS_ERR_CUDA.
 *
 * mxs_attention_decode -- the same for one sequence of T tokens (B = 1,
 * T_cap = T, no lengths); q bf16 [H, D], out fp32 [H, D], workspace of
 * mxs_attention_decode_workspace_bytes(T, H, D) bytes with the same rule. */
MXS_API int64_t mxs_attention_decode_workspace_bytes(int64_t T, int64_t H, int64_t D);
MXS_API int mxs_attention_decode(const void *q_bf16, int64_t H, int64_t H_kv, int64_t D, const void *k_codes,
                                 const uint8_t *k_scales, const uint8_t *k_bits, const void *v_codes,
                                 const uint8_t *v_scales, const uint8_t *v_bits, int64_t T, float scale, float *out,
                                 void *workspace, size_t ws_bytes, void *stream);
MXS_API int64_t mxs_attention_decode_batch_workspace_bytes(int64_t B, int64_t T_cap, int64_t H, int64_t D);
MXS_API int mxs_attention_decode_batch(const void *q_bf16, int64_t B, int64_t H, int64_t H_kv, int64_t D,
                                       const void *k_codes, const uint8_t *k_scales, const uint8_t *k_bits,
                                       const void *v_codes, const uint8_t *v_scales, const uint8_t *v_bits,
                                       const int32_t *lengths, int64_t T_cap, float scale, float *out,
                                       void *workspace, size_t ws_bytes, void *stream);

/* ---------------------------------------------------------------- tensor-core rate probes
 * Measurement only (not on the layer's path; the paper has no counterpart):
 * the denominators of the GEMMs' rooflines, and the cost of the small MMAs
 * the decode GEMM issues.  One CTA per SM; thread 0 of each issues `iters`
 * MMAs back to back into one tensor-memory accumulator over all-zero
 * operands, commits them and waits (bounded) for completion:
 *   kind 0  tcgen05.mma kind::mxf8f6f4 block_scale (e4m3, UE8M0 per 32),
 *           M = 128, N = n, K = 32, A and B in shared memory (the prefill
 *           GEMM's 4-bit instruction);
 *   kind 1  the same with A in tensor memory (the decode GEMM's instruction);
 *   kind 2  tcgen05.mma kind::f16 (bf16 -> fp32), M = 128, N = n, K = 16;
 *   kind 3  legacy warp MMA mma.sync m16n8k32 s8 -> s32 on four warps per
 *           CTA (n ignored): the INT8 tensor rate of this part.
 * n: a multiple of 16 in [16, 256].  *flop receives the launch's operations
 * (2*M*N*K per MMA); time the launch with events on `stream`.  cycles
 * (device int64 [SM count], 8-byte aligned, or NULL) receives each CTA's
 * clock cycles from its first MMA to its wait's end (kinds 0-2) or its
 * loop (kind 3).  Asynchronous.  Errors: MXS_ERR_INVALID_ARG (kind 0..3, n,
 * iters outside [1, 2^32], flop NULL), MXS_ERR_ALIGN, MXS_ERR_CUDA.
 * mxs_probe_status synchronises the device and reads (reset != 0: clears)
 * the probes' status word: MXS_ERR_TIMEOUT if a wait ran out. */
MXS_API int mxs_probe_mma(int kind, int n, int64_t iters, int64_t *cycles, double *flop, void *stream);
MXS_API int mxs_probe_status(int *status, int reset);
/* Issue-rate probe for the decode GEMMs' MMAs (measurement only; the paper
 * has no counterpart): on every SM, `issuers` warps (1, 2 or 4), one thread
 * each, issue `iters` (a multiple of 4) MMAs back to back into four
 * accumulators of their own: M = 128, N = 16, A in tensor memory, the A
 * column and scale byte varying as in the decode kernels; kind 0 block-scaled
 * e4m3 (kind::mxf8f6f4), 1 bf16 (kind::f16), 2 kind 0 with two scale-tile
 * copies (tcgen05.cp) per four MMAs.  cycles (device int64 [SM count],
 * 8-byte aligned, or NULL) receives issuer 0's clock cycles from its first
 * MMA to its commit's completion; cycles / iters is the cost per MMA of one
 * issuing thread.  Asynchronous.  Errors: MXS_ERR_INVALID_ARG, MXS_ERR_ALIGN,
 * MXS_ERR_CUDA; status as mxs_probe_mma. */
MXS_API int mxs_probe_mma_issue(int kind, int issuers, int64_t iters, int64_t *cycles, void *stream);

/* ---------------------------------------------------------------- offline allocation
 * Calibration that produces the width maps (Alg. 1, Alg. 3, Theorem 1).  Not
 * on the inference path; run once per model over calibration activations.
 *
 * mxs_column_sensitivity -- Alg. 1 (Sec. 3.1): the column sensitivity of a
 * linear layer is the diagonal of H = X^T X summed over the calibration
 * samples, s[j] = sum_k X[k][j]^2.  One call adds one batch:
 *   x        device, bf16 [T, K] row-major with row stride ld_x elements
 *            (ld_x >= K, a multiple of 8; x 16-byte aligned); T >= 0 rows
 *   K        a positive multiple of 32 (the layer's input dimension)
 *   s        device, fp64 [K], 8-byte aligned: s[j] = (accumulate ? s[j] : 0)
 *            + sum of x[k][j]^2 over the T rows
 * Deterministic: the result depends on x, T and K only.  Each square of a bf16
 * is exact; runs of 8 rows are added in fp32 (relative error <= 2^-21 of the
 * run) unless a run leaves [2^-100, 2^100), in which case it is added in fp64;
 * the runs are added in fp64.  NaN or Inf in a column makes its s NaN or Inf.
 * Asynchronous on `stream`; allocates nothing.  Errors: MXS_ERR_SHAPE (T < 0,
 * K), MXS_ERR_INVALID_ARG (NULL, ld_x), MXS_ERR_ALIGN, MXS_ERR_CUDA. */
MXS_API int mxs_column_sensitivity(const void *x_bf16, int64_t T, int64_t K, int64_t ld_x, double *s, int accumulate,
                                   void *stream);

/* mxs_allocation_r -- Theorem 1 (Appendix A): the control parameter R that
 * makes the triplet allocation average B bits per column over n layers (32
 * columns per layer at 8 bits, R * S_i * (d_i - 32) at 6, the rest at 4),
 * before any flooring:
 *   R = ((B - 4) * sum_i d_i - 4 * 32 * n) / sum_i 2 * S_i * (d_i - 32).
 * Host only (all arguments host memory): d_in[n] positive multiples of 32,
 * s_layer[n] the layer sensitivities of Alg. 2 in [0, 1] (an input here).
 * Errors: MXS_ERR_SHAPE (n, d_in), MXS_ERR_INVALID_ARG (NULL, S outside
 * [0, 1], no layer with S > 0 and d > 32, or B below the 8-bit floor: R < 0). */
MXS_API int mxs_allocation_r(int64_t n, const int64_t *d_in, const double *s_layer, double B, double *R);

/* mxs_allocate_layer -- Alg. 3 for one layer with K = d_in columns:
 *   s      device, fp64 [K] column sensitivities (mxs_column_sensitivity);
 *          NaN keys give an unspecified order
 *   perm   device, int32 [K] out: perm[p] = the original column at position p
 *          of the descending order of s (equal values by column index)
 *   bits   host, uint8 [K/32] out, written before the call returns: the width
 *          of each 32-column block of that order -- block 0: 8 bits (the 32
 *          most sensitive columns), then floor(N6 / 32) blocks of 6 bits (the
 *          6-bit columns in whole blocks, Sec. 4.1), the rest 4 bits
 *   n6     host out (may be NULL): N6 = floor(R * s_layer * (K - 32)) clamped
 *          to [0, K - 32]
 * K a multiple of 32 in [32, MXS_MAX_K]; R >= 0; s_layer in [0, 1].  The order
 * is computed on the GPU, asynchronously on `stream` (O(K^2) comparisons).
 * Applying the order (permuting the layer's weight columns and, upstream, its
 * input channels) is the caller's.  Errors: MXS_ERR_SHAPE, MXS_ERR_INVALID_ARG,
 * MXS_ERR_ALIGN (s 8-byte, perm 4-byte aligned), MXS_ERR_CUDA. */
MXS_API int mxs_allocate_layer(const double *s, int64_t K, double R, double s_layer, int32_t *perm, uint8_t *bits,
                               int64_t *n6, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* MXS_H_ */
