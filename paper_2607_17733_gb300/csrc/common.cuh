// common.cuh -- shared pieces of libmxs: the grouping plan, the block
// quantizer, launch helpers.  Device code here is sm_103a only.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/mxs.h"

namespace mxs {

constexpr int kBlock = 32;
constexpr int kMaxNb = MXS_MAX_K / kBlock;

// Width grouping of a map (step A0).  slot -> original block index, stable
// inside each width group; passed by value to kernels (__grid_constant__).
struct Plan {
    int nb, n4, n6, n8, n68;
    int st4;  // ceil(n4/4): 128-byte K' stages of 4-bit slots in the plane layout
    int nst;  // st4 + ceil(n68/2)
    int64_t row_bytes;  // packed activation row
    int64_t kp;         // plane row bytes = 128*nst
    uint16_t slot_block[kMaxNb];
};

template <class P>
__host__ __device__ inline int slot_width(const P &p, int s) {
    return s < p.n4 ? 4 : (s < p.n4 + p.n6 ? 6 : 8);
}

__host__ __device__ inline int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

// Packed weights: group g (128 rows) is GB = 2176*n4 + 4224*n68 contiguous
// bytes; a 4-bit slot is 128 x 16 code bytes + 128 scale bytes, a 6/8-bit
// slot 128 x 32 + 128.
struct WeightOffsets {
    int64_t G, Np, GB, compact, planes, sf, total;
};

template <class P>
__host__ __device__ inline int64_t slot_offset(const P &p, int s) {
    return s < p.n4 ? 2176 * (int64_t)s : 2176 * (int64_t)p.n4 + 4224 * (int64_t)(s - p.n4);
}

__host__ __device__ inline WeightOffsets weight_offsets(const Plan &p, int64_t N, bool with_planes) {
    WeightOffsets w;
    w.G = (N + 127) / 128;
    w.Np = w.G * 128;
    w.GB = 2176 * (int64_t)p.n4 + 4224 * (int64_t)p.n68;
    w.compact = align256(w.G * w.GB);
    w.planes = w.compact;
    w.sf = align256(w.planes + N * p.kp);
    w.total = with_planes ? align256(w.sf + (N + 127) / 128 * p.nst * 512) : w.compact;
    return w;
}

// ------------------------------------------------------------ quantizer
// Integer form of the MXINT rule on bf16 bit patterns: the scale byte is the
// bf16 exponent field of the block's largest magnitude (floor(log2) of a
// normal number, 0 for zero/subnormal maxima, 255 for Inf/NaN), and an element
// with significand sig and exponent field e is sig * 2^-sh in units of the
// grid step, sh = S - max(e,1) + 9 - b >= 0.  Rounding is done on the bits
// that shift out, then the magnitude is clamped to 2^(b-1)-1.
__device__ __forceinline__ int quant_elem(uint32_t h, int S, int b, int rhaz) {
    const int e = (h >> 7) & 0xFF;
    const int sig = e ? (int)((h & 0x7F) | 0x80) : (int)(h & 0x7F);
    int sh = S - (e ? e : 1) + 9 - b;
    sh = sh > 10 ? 10 : sh;  // beyond 9 the magnitude is below 1/4 step: 0
    int q;
    if (sh == 0) {
        q = sig;
    } else {
        q = sig >> sh;
        const int rem = sig & ((1 << sh) - 1);
        const int half = 1 << (sh - 1);
        q += (rem > half) | ((rem == half) & (rhaz | (q & 1)));
    }
    const int Q = (1 << (b - 1)) - 1;
    q = q > Q ? Q : q;
    return (h & 0x8000) ? -q : q;
}

// e4m3 byte of an exactly representable value (hardware conversion).
__device__ __forceinline__ uint16_t e4m3x2(float lo, float hi) {
    uint16_t r;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
    return r;
}

// bf16 pair of two exactly representable values (lo in the low half)
__device__ __forceinline__ uint32_t bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// 2^e as fp32 for e in [-149, 127] (subnormal below -126), exact.
__device__ __forceinline__ float pow2f(int e) {
    return e >= -126 ? __int_as_float((e + 127) << 23) : __int_as_float(1 << (e + 149 < 0 ? 0 : e + 149));
}

}  // namespace mxs

// ------------------------------------------------------------ host side
namespace mxs {
void set_error(const char *fmt, ...);
int fail(int code, const char *fmt, ...);
int build_plan(const uint8_t *bits, int64_t K, Plan *p);
int check_device();
int cuda_fail(cudaError_t e, const char *what);

// kernel launchers (one translation unit each)
int quantize_act_impl(const void *x, int64_t M, int64_t K, int64_t ld_x, const int32_t *perm, const uint8_t *bits,
                      int rounding, void *codes, uint8_t *scales, void *planes, void *stream);
int pack_weight_impl(const void *w, int64_t N, int64_t K, int64_t ld_w, const int32_t *perm, const uint8_t *bits,
                     int rounding, int layout, void *packed, void *stream);
int launch_quantize(const Plan &p, const void *x, int64_t M, int64_t ld, int rounding, void *codes,
                    uint8_t *scales, void *planes, cudaStream_t st, const int32_t *perm = nullptr);
// the activations of up to three decode problems to MMA planes in one launch
int launch_quantize_group(const Plan *const *plans, const void *const *x, const int64_t *ld, int64_t M, int rounding,
                          void *const *planes, int count, cudaStream_t st);
int launch_pack_weight(const Plan &p, const void *w, int64_t N, int64_t ld, int rounding, bool planes,
                       void *packed, cudaStream_t st, const int32_t *perm = nullptr);
int64_t decode_workspace_bytes(const Plan &p, int64_t M, int64_t N);
// decode GEMM over packed codes + scales (act_planes NULL) or over the
// activation MMA planes (codes/scales NULL); pdl: the launch may overlap the
// tail of the previous kernel on the stream (programmatic dependent launch)
// starve > 0 (test hook): every CTA skips the weight copy of its chunk starve-1
int launch_gemm_decode(const Plan &p, const void *codes, const uint8_t *scales, const void *act_planes,
                       const void *packed, int64_t M, int64_t N, float *y, int64_t ld_y, bool pdl, cudaStream_t st,
                       int starve = 0);
// up to three decode GEMMs (planes mode) in one launch; returns -1, with no
// error recorded, when no cluster size fits every problem
int launch_gemm_decode_group(const Plan *const *plans, const void *const *act_planes, const void *const *packed,
                             const int64_t *N, float *const *y, const int64_t *ld_y, int count, int64_t M, bool pdl,
                             cudaStream_t st);
int decode_status(int *status, int reset);
int gemv_status(int *status, int reset);
// Decode shapes of at most kGemvMaxM tokens: the activations' quantization
// fused into a CUDA-core GEMM (dp4a integer dots, fp32 fold), up to three
// problems that read x_i (bf16 [M, K_i], row stride ld_x_i) in one launch.
// The kernel takes 1 <= M <= 4; the library routes M = 1 to it by default
// (beyond one token the tensor-core path is faster, as measured on GB300).
#ifndef MXS_GEMV_MAX_M
#define MXS_GEMV_MAX_M 1
#endif
constexpr int kGemvMaxM = MXS_GEMV_MAX_M;
// ws_i: device workspace of at least gemv_workspace_bytes(M, N_i) bytes
// (arrival counters and partial sums; any prior contents).
int launch_gemv_decode(const Plan *const *plans, const void *const *x, const int64_t *ld_x, const void *const *packed,
                       const int64_t *N, float *const *y, const int64_t *ld_y, void *const *ws,
                       const size_t *ws_bytes, int count, int64_t M, int rounding, bool pdl, cudaStream_t st);
int64_t gemv_workspace_bytes(int64_t M, int64_t N);
// test hook: the next launch of that kernel has every CTA skip the weight copy
// of its stage `stage` (1-based; 0 disarms)
void gemv_arm_starve(int stage);
int gemv_split_cost4();  // the split's weight of a 4-bit slot, percent of its bytes
// Decode shapes of kGemvMaxM < M <= 16 tokens through mxs_linear_decode(_group):
// the quantizer writes the planes into ws_i, then the tensor-core kernel of
// decode_tc.cu (an equal share of the weight bytes per CTA) runs as its
// programmatic dependent.  ws_i: [planes][arrival counters][partial sums],
// dtc_workspace_bytes(plan, M, N) bytes for the most CTAs (fewer fit a smaller one).
#ifndef MXS_DECODE_TC
#define MXS_DECODE_TC 1
#endif
int launch_decode_tc(const Plan *const *plans, void *const *ws, const size_t *ws_bytes, const void *const *packed,
                     const int64_t *N, float *const *y, const int64_t *ld_y, int count, int64_t M, bool pdl,
                     cudaStream_t st);
int64_t dtc_workspace_bytes(const Plan &p, int64_t M, int64_t N);
int dtc_status(int *status, int reset);
void dtc_arm_starve(int stage);  // as gemv_arm_starve
int dtc_split_cost8();           // the split's weight of a 6/8-bit slot, percent of its bytes
int launch_gemm_prefill(const Plan &p, const void *act_planes, const void *packed_w, int64_t M, int64_t N,
                        float *y, int64_t ld_y, int starve, cudaStream_t st);
int prefill_status(int *status, int reset, cudaStream_t st);
// 2-D TMA map over an e4m3 plane matrix [rows, kp] (row stride kp bytes):
// boxes of 128 bytes x box_rows rows, 128-byte swizzle, zero fill outside
int make_plane_map(CUtensorMap *map, const void *base, int64_t rows, int64_t kp, int box_rows);
// 2-D TMA map over an fp32 output y [rows, cols] (row stride ld elements, a
// multiple of 4; base 16-byte aligned): boxes of 32 rows x 16 columns
int make_f32_out_map(CUtensorMap *map, float *base, int64_t rows, int64_t cols, int64_t ld);
}  // namespace mxs
