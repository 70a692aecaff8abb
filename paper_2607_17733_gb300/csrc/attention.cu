// attention.cu -- decode attention over an MXINT-quantized KV cache.
//
// The paper quantizes the KV cache with a 4-8 bit configuration (Appendix
// A.2) and keeps Softmax in FP16.  The cache rows are written by
// mxs_quantize_act (one token's H_kv * D values per row, quantized along the
// row with the row's width map), so appending a token is one quantizer call
// into row t; this file reads the cache.  One query token per sequence, a
// batch of B sequences of their own lengths, grouped-query heads (query head
// h reads KV head h / G):
//     s_t = scale * <q_h, k_t>,  out_h = sum_t softmax(s)_t * v_t.
//
// One launch.  A CTA owns (sequence, KV head, split): a contiguous run of the
// sequence's tokens, in tiles of 64 that a cp.async ring stages in shared
// memory (codes by 16-byte copies, the tile's scale bytes through registers).
// Each of the four warps takes 16 tokens of a tile and keeps its own running
// softmax (max, sum, weighted sums) for the G query heads:
//   * a cache element c * 2^(S - 127 - (b - 2)) is exact in bf16 (|c| <= 127),
//     so the codes are expanded to bf16 pairs by integer operations that put
//     the code in the mantissa of a bf16 whose exponent carries the block
//     scale, and one exact subtraction removes the offset (for 6/8-bit codes
//     the high and low nibbles are placed apart and added exactly); blocks
//     with S outside [8, 247] (tiny, huge, NaN) take an fp32 route;
//   * scores: mma.sync m16n8k16 bf16 -> fp32 with A = the query heads (rows,
//     padded to 16) and B = the dequantized keys (8 tokens per n-tile): every
//     product is exact and the sums are fp32;
//   * weighted sums: A = the softmax weights p split as p_hi + p_lo (two bf16
//     rows per head, |p - p_hi - p_lo| <= 2^-18 p), B = the dequantized values
//     (16 tokens x 8 dimensions per n-tile), fp32 accumulators;
//   * the warps' states merge in warp order, the splits of a (sequence, KV
//     head) in split order in the CTA that arrives last (a counter per
//     (sequence, KV head) in the workspace, reset by that CTA): deterministic.
// HBM-bound: every cache byte of the batch is read once per step.
#include <cuda_bf16.h>

#include <cmath>

#include "common.cuh"

namespace mxs {
namespace {

#ifndef MXS_ATT_MIN_CTAS
#define MXS_ATT_MIN_CTAS 3
#endif
constexpr int kTile = 64;          // tokens per ring stage (16 per warp)
constexpr int kWarps = 4;
constexpr int kThreads = 32 * kWarps;
constexpr int kStages = 4;         // ring depth
constexpr int kMaxG = 8;           // query heads per KV head (the MMA's 8 rows)
constexpr int kMaxKvBlocks = 256;  // H_kv * D / 32 (H_kv * D <= 8192)
constexpr int kMaxSplits = 64;     // splits of one sequence
constexpr uint32_t kOne = 0x3F803F80u;  // bf16x2 (1, 1)

struct AttnArgs {
    const uint16_t *q;                 // [B, H, D] bf16
    const uint8_t *kc, *ks, *vc, *vs;  // codes [B * T_cap, row bytes], scales [B * T_cap, nb]
    const int32_t *lengths;            // [B] device, or null: every sequence has T_cap tokens
    float *part;                       // [B][H_kv][S][G][D]: weighted sums of each split
    float *stat;                       // [B][H_kv][S][G][2]: its max and sum
    uint32_t *count;                   // [B * H_kv] arrivals; zero before and after a launch
    float *out;                        // [B, H, D] fp32
    int64_t k_row, v_row, T_cap;
    int nb, H, H_kv, G, S;
    float sl2;                         // scale * log2(e)
    // per block of a row: byte offset of its codes in a code row, width, scale slot
    uint16_t k_off[kMaxKvBlocks], v_off[kMaxKvBlocks];
    uint8_t k_b[kMaxKvBlocks], v_b[kMaxKvBlocks];
    uint8_t k_slot[kMaxKvBlocks], v_slot[kMaxKvBlocks];
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
// a + c in bf16x2 (as a * 1 + c): used only where the sum is representable, so exact
__device__ __forceinline__ uint32_t bf2_add(uint32_t a, uint32_t c) {
    uint32_t d;
    asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(kOne), "r"(c));
    return d;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&v);
}
// 2^x by the SFU (relative error about 2^-22; 2^-inf = 0, NaN stays NaN)
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// transpose of an 8x8 matrix of 16-bit elements held one row pair per lane
// (lane 4r + c: row r, columns 2c, 2c+1) into the same layout
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
    return y;
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 2^(S - 127 - (b - 2)) in fp32 (NaN for S = 255): the fp32 route's factor
__device__ __forceinline__ float block_factor(int S, int b) {
    return S == 255 ? __int_as_float(0x7FC00000) : ldexpf(1.0f, S - 125 - b);
}
__device__ __forceinline__ bool fast_scale(int S) { return S >= 8 && S <= 247; }

// Two cache elements as a bf16 pair, from `y` holding their codes in its low
// and high half (a 4-bit code in bits 0-3 of each half; an int8 code in bits
// 0-7), each half with its own block scale S in [8, 247].
// 4-bit: x = bf16 with exponent field S + 5 and mantissa (c ^ 8) is
// 2^(S-122) * (1 + (c + 8)/128), and x - 2^(S-122) * (1 + 8/128) = c * 2^(S-129).
// 6/8-bit, c = 16h + l: xh = bf16(exponent field Eh = S + 13 - b, mantissa
// h ^ 8), t = xh - 2^(Eh-127) * 1.125 = (h - 8) * 2^(Eh-134), and
// xl = bf16(exponent field Eh - 4, mantissa l) = 2^(Eh-131) + l * 2^(Eh-138),
// so xl + t = (16h + l) * 2^(Eh-138) = c * 2^(S-125-b).  Every step is exact.
__device__ __forceinline__ uint32_t e4(int SA, int SB) {
    return (((uint32_t)(SA + 5) << 7) | 8u) | ((((uint32_t)(SB + 5) << 7) | 8u) << 16);
}
__device__ __forceinline__ uint32_t deq4_pair(uint32_t y, uint32_t xe) {
    return bf2_add((y & 0x000F000Fu) ^ xe, xe ^ 0x80008000u);
}
struct Deq8 {
    uint32_t xh, xl, c1n;
};
__device__ __forceinline__ Deq8 e8(int SA, int SB, int b) {
    const uint32_t ea = (uint32_t)(SA + 13 - b), eb = (uint32_t)(SB + 13 - b);
    Deq8 d;
    d.xh = ((ea << 7) | 8u) | (((eb << 7) | 8u) << 16);
    d.xl = ((ea - 4) << 7) | (((eb - 4) << 7) << 16);
    d.c1n = (((ea << 7) | 16u) | (((eb << 7) | 16u) << 16)) ^ 0x80008000u;
    return d;
}
__device__ __forceinline__ uint32_t deq8_pair(uint32_t y, const Deq8 &c) {
    const uint32_t xh = ((y >> 4) & 0x000F000Fu) ^ c.xh;
    const uint32_t xl = (y & 0x000F000Fu) | c.xl;
    return bf2_add(xl, bf2_add(xh, c.c1n));
}
// code of element e of a segment held in words w (width b)
__device__ __forceinline__ int seg_code(const uint32_t *w, int b, int e) {
    if (b == 4) return (int)(w[e >> 3] << (28 - 4 * (e & 7))) >> 28;
    return (int)(w[e >> 2] << (24 - 8 * (e & 3))) >> 24;
}

// The K segment of lane q is dimensions [q * D/4, (q+1) * D/4) of the head:
// one block (D = 128) or half a block (D = 64).  Its bf16 pairs in the order
// the score MMA consumes them (pair 2s -> k-slots 2q, 2q+1 of k-step s, pair
// 2s+1 -> k-slots 2q+8, 2q+9): 4-bit pair r = dims (8(r/4) + r%4, that + 4);
// 6/8-bit pair r = dims (4(r/2) + r%2, that + 2).  The query uses the same order.
__device__ __forceinline__ int kpair_dim(int b, int r, int hi) {
    return b == 4 ? 8 * (r >> 2) + (r & 3) + 4 * hi : 4 * (r >> 1) + (r & 1) + 2 * hi;
}

template <int D>
__global__ void __launch_bounds__(kThreads, MXS_ATT_MIN_CTAS) attention_decode_kernel(const __grid_constant__ AttnArgs a) {
    constexpr int NBH = D / 32;      // blocks per head
    constexpr int KSTEPS = D / 16;   // k-steps of the score MMA
    constexpr int NT = D / 8;        // n-tiles of the weighted-sum MMA (= dims of a V segment)
    constexpr int SEGK = D / 4;      // dims of a lane's K segment
    constexpr int KW = SEGK / 4;     // words of a K segment at 8 bits (half at 4 bits)
    constexpr int VW = NT / 4;       // words of a V segment at 8 bits (half at 4 bits)
    // A staged token row keeps 32 bytes per block whatever its width (a 4-bit
    // block fills the first 16), so every shared-memory offset is a constant;
    // V rows carry 16 more bytes, which spreads four-token reads over the banks.
    constexpr int KS = D, VS = D + 16;
    constexpr int STAGE = kTile * (KS + VS + 2 * NBH);
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ int sh_last;
    const int split = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int gi = lane >> 2, q = lane & 3;  // MMA group (row / column index), lane in the group
    const int G = a.G;
    uint8_t *const ring = smem;

    // lane q reads the K segment of block jq, lane group gi the V segment of block jv
    const int jq = (q * SEGK) / 32, jv = (gi * NT) / 32;
    int kbq = 4, vbv = 4;
#pragma unroll
    for (int j = 0; j < NBH; ++j) {
        if (j == jq) kbq = a.k_b[hk * NBH + j];
        if (j == jv) vbv = a.v_b[hk * NBH + j];
    }

    // this CTA's tokens [t0, t1) of sequence b
    int len = (int)a.T_cap;
    if (a.lengths) len = min(max(__ldg(a.lengths + b), 0), (int)a.T_cap);
    const int per = ((len + a.S - 1) / a.S + kTile - 1) / kTile * kTile;
    const int t0 = min(len, split * per), t1 = min(len, t0 + per);
    const int ntile = (t1 - t0 + kTile - 1) / kTile;
    const int64_t row0 = (int64_t)b * a.T_cap;

    // ---- each warp stages its own 16 tokens of every tile (and only reads
    // those): lane l copies token l/2 of the warp's slice, K (even l) or V (odd)
    const int ptok = 16 * warp + (lane >> 1), pv = lane & 1;
    const uint8_t *const pcode = pv ? a.vc : a.kc;
    const uint8_t *const pscale = pv ? a.vs : a.ks;
    const int64_t prow = pv ? a.v_row : a.k_row;
    int poff[NBH], pwide[NBH], pslot[NBH];
#pragma unroll
    for (int j = 0; j < NBH; ++j) {
        const int kb = hk * NBH + j;
        poff[j] = pv ? a.v_off[kb] : a.k_off[kb];
        pwide[j] = (pv ? a.v_b[kb] : a.k_b[kb]) != 4;
        pslot[j] = pv ? a.v_slot[kb] : a.k_slot[kb];
    }
    const uint32_t pdst = smem_u32(ring) + (pv ? kTile * KS + ptok * VS : ptok * KS);
    auto issue = [&](int tile, uint32_t &scales) {
        const int t = t0 + tile * kTile + ptok;
        const uint32_t dst = pdst + (uint32_t)((tile & (kStages - 1)) * STAGE);
        scales = 0x7F7F7F7Fu;  // tokens past the end: a plain scale (their weights are zero)
        if (t < t1) {
            const uint8_t *src = pcode + (row0 + t) * prow;
#pragma unroll
            for (int j = 0; j < NBH; ++j) {
                cp_async16(dst + 32 * j, src + poff[j]);
                if (pwide[j]) cp_async16(dst + 32 * j + 16, src + poff[j] + 16);
            }
            const uint8_t *srow = pscale + (row0 + t) * a.nb;
            uint32_t sb = 0;
#pragma unroll
            for (int j = 0; j < NBH; ++j) sb |= (uint32_t)__ldg(srow + pslot[j]) << (8 * j);
            scales = sb;
        }
    };
    auto put_scales = [&](int tile, uint32_t scales) {
        uint8_t *d = ring + (tile & (kStages - 1)) * STAGE + kTile * (KS + VS) + (pv ? kTile * NBH : 0) + ptok * NBH;
        if (NBH == 4)
            *reinterpret_cast<uint32_t *>(d) = scales;
        else
            *reinterpret_cast<uint16_t *>(d) = (uint16_t)scales;
    };

    // ---- the query as the score MMA's B operand: column gi = query head gi
    //      (zero for gi >= G), k-slots of lane q's K segment in pair order
    const int kseg_byte = kbq == 4 ? ((q * SEGK) % 32) / 2 : (q * SEGK) % 32;
    uint32_t qb[KSTEPS][2];
    {
        const bool real = gi < G;
        const uint16_t *qrow = a.q + ((int64_t)b * a.H + hk * G + (real ? gi : 0)) * D + q * SEGK;
#pragma unroll
        for (int s = 0; s < KSTEPS; ++s)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int r = 2 * s + h;
                const uint32_t lo = real ? __ldg(qrow + kpair_dim(kbq, r, 0)) : 0u;
                const uint32_t hi = real ? __ldg(qrow + kpair_dim(kbq, r, 1)) : 0u;
                qb[s][h] = lo | (hi << 16);
            }
    }
    const int vseg_byte = vbv == 4 ? ((gi * NT) % 32) / 2 : (gi * NT) % 32;
    // per-lane offsets in a stage: K rows of tokens gi and gi + 8 of the warp's
    // 16; V rows of tokens 2q, 2q+1, 2q+8, 2q+9; their scale bytes
    const int koff = (16 * warp + gi) * KS + 32 * jq + kseg_byte;
    const int voff = kTile * KS + (16 * warp + 2 * q) * VS + 32 * jv + vseg_byte;
    const int ksof = kTile * (KS + VS) + (16 * warp + gi) * NBH + jq;
    const int vsof = kTile * (KS + VS + NBH) + (16 * warp + 2 * q) * NBH + jv;

    // running softmax: maxima (log2 units) and this lane's part of the sums of
    // heads 2q, 2q+1; weighted sums of head gi (MMA rows gi: p_hi, gi + 8: p_lo)
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.0f, l1 = 0.0f;
    float acc[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.0f;

    // ---- ring prologue: tiles 0 .. kStages-2.  The scale bytes travel through
    // registers: loaded when their tile's copies are issued, stored to shared
    // memory in the iteration before the tile is used (two iterations later).
    // No barrier across warps: each warp waits for its own copies only.
    static_assert(kStages == 4, "the scale pipeline below holds two tiles");
    uint32_t pend1 = 0x7F7F7F7Fu, pend2 = 0x7F7F7F7Fu;  // scales of tiles tile+1, tile+2
    {
        uint32_t s0 = 0x7F7F7F7Fu;
        if (0 < ntile) issue(0, s0);
        cp_async_commit();
        if (1 < ntile) issue(1, pend1);
        cp_async_commit();
        if (2 < ntile) issue(2, pend2);
        cp_async_commit();
        if (0 < ntile) put_scales(0, s0);
    }

    for (int tile = 0; tile < ntile; ++tile) {
        cp_async_wait<kStages - 2>();
        __syncwarp();  // the warp's copies and scales of this tile are in place; its tile - 1 rows are free
        if (tile + 1 < ntile) put_scales(tile + 1, pend1);  // read after the next __syncwarp
        pend1 = pend2;
        if (tile + kStages - 1 < ntile) issue(tile + kStages - 1, pend2);
        cp_async_commit();

        const int valid = t1 - t0 - tile * kTile - 16 * warp;  // the warp's tokens [0, valid) are real
        if (valid <= 0) continue;
        const uint8_t *st = ring + (tile & (kStages - 1)) * STAGE;

        // ---- keys of tokens gi (MMA row gi) and gi + 8 (row gi + 8) as bf16 pairs
        uint32_t kw[2][KW];
        int Sk[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const uint8_t *src = st + koff + h * 8 * KS;
#pragma unroll
            for (int i = 0; i < KW; ++i) kw[h][i] = 0;
            if (D == 128 || kbq != 4) {  // 16 or 32 bytes, 16-byte aligned
#pragma unroll
                for (int i = 0; i < KW; i += 4)
                    if (kbq != 4 || i < KW / 2) {
                        const uint4 v = *reinterpret_cast<const uint4 *>(src + 4 * i);
                        kw[h][i] = v.x, kw[h][i + 1] = v.y, kw[h][i + 2] = v.z, kw[h][i + 3] = v.w;
                    }
            } else {  // D = 64 at 4 bits: 8 bytes
                const uint2 v = *reinterpret_cast<const uint2 *>(src);
                kw[h][0] = v.x, kw[h][1] = v.y;
            }
            Sk[h] = st[ksof + h * 8 * NBH];
        }
        uint32_t kp[2][2 * KSTEPS];
        if (__all_sync(0xffffffffu, fast_scale(Sk[0]) && fast_scale(Sk[1]))) {
            if (kbq == 4) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const uint32_t xe = e4(Sk[h], Sk[h]);
#pragma unroll
                    for (int r = 0; r < 2 * KSTEPS; ++r) kp[h][r] = deq4_pair(kw[h][r >> 2] >> (4 * (r & 3)), xe);
                }
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const Deq8 c = e8(Sk[h], Sk[h], kbq);
#pragma unroll
                    for (int r = 0; r < 2 * KSTEPS; ++r) kp[h][r] = deq8_pair(kw[h][r >> 1] >> (8 * (r & 1)), c);
                }
            }
        } else {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const float f = block_factor(Sk[h], kbq);
#pragma unroll
                for (int r = 0; r < 2 * KSTEPS; ++r)
                    kp[h][r] = pack_bf16((float)seg_code(kw[h], kbq, kpair_dim(kbq, r, 0)) * f,
                                         (float)seg_code(kw[h], kbq, kpair_dim(kbq, r, 1)) * f);
            }
        }

        // ---- scores, tokens x heads: (gi, 2q), (gi, 2q+1), (gi+8, 2q), (gi+8, 2q+1)
        float c[2][4] = {{0.0f, 0.0f, 0.0f, 0.0f}, {0.0f, 0.0f, 0.0f, 0.0f}};  // two chains of k-steps
#pragma unroll
        for (int s = 0; s < KSTEPS; ++s)
            mma_bf16(c[s & 1], kp[0][2 * s], kp[1][2 * s], kp[0][2 * s + 1], kp[1][2 * s + 1], qb[s][0], qb[s][1]);
        float sv[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int tok = gi + 8 * (e >> 1);
            sv[e] = tok < valid ? (c[0][e] + c[1][e]) * a.sl2 : -INFINITY;
        }

        // ---- online softmax of heads 2q (e = 0, 2) and 2q+1 (e = 1, 3) over the 16 tokens
        float x0 = fmaxf(sv[0], sv[2]), x1 = fmaxf(sv[1], sv[3]);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
            x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, o));
            x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, o));
        }
        // The running maximum moves only when a score passes it by more than 8
        // (so p <= 2^8): a stabiliser, rarely rescaled.
        const bool up0 = x0 > m0 + 8.0f, up1 = x1 > m1 + 8.0f;
        if (__any_sync(0xffffffffu, up0 || up1)) {
            const float n0 = up0 ? x0 : m0, n1 = up1 ? x1 : m1;
            const float al0 = ex2(m0 - n0), al1 = ex2(m1 - n1);
            l0 *= al0, l1 *= al1;
            m0 = n0, m1 = n1;
            // the weighted sums on this lane are head gi's: its factor is on lane gi / 2
            const float b0 = __shfl_sync(0xffffffffu, al0, gi >> 1), b1 = __shfl_sync(0xffffffffu, al1, gi >> 1);
            const float al = (gi & 1) ? b1 : b0;
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                acc[j][0] *= al, acc[j][1] *= al;
                acc[j][2] *= al, acc[j][3] *= al;
            }
        }
        const float p0 = ex2(sv[0] - m0), p1 = ex2(sv[1] - m1), p2 = ex2(sv[2] - m0), p3 = ex2(sv[3] - m1);
        l0 += p0 + p2, l1 += p1 + p3;
        // P as two 8x8 bf16 tiles (tokens x heads), split hi + lo, transposed into
        // the A operand (rows = heads: gi with p_hi, gi + 8 with p_lo; k = tokens)
        const uint32_t h1 = pack_bf16(p0, p1), h2 = pack_bf16(p2, p3);
        const uint32_t o1 = pack_bf16(p0 - bf16_lo(h1), p1 - bf16_hi(h1));
        const uint32_t o2 = pack_bf16(p2 - bf16_lo(h2), p3 - bf16_hi(h2));
        const uint32_t A0 = movmatrix_t(h1), A1 = movmatrix_t(o1), A2 = movmatrix_t(h2), A3 = movmatrix_t(o2);

        // ---- weighted sums: lane (gi, q) supplies tokens (2q, 2q+1) and (2q+8, 2q+9)
        //      at dimension gi * D/8 + j of n-tile j
        uint32_t wv[4][VW];
        int Sv[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int trow = 8 * (e >> 1) + (e & 1);  // row offset of token 2q + trow
            const uint8_t *src = st + voff + trow * VS;
#pragma unroll
            for (int i = 0; i < VW; ++i) wv[e][i] = 0;
            if (vbv == 4) {
                if (D == 128) {
                    const uint2 v = *reinterpret_cast<const uint2 *>(src);
                    wv[e][0] = v.x, wv[e][1] = v.y;
                } else {
                    wv[e][0] = *reinterpret_cast<const uint32_t *>(src);
                }
            } else {
                if (D == 128) {
                    const uint4 v = *reinterpret_cast<const uint4 *>(src);
                    wv[e][0] = v.x, wv[e][1] = v.y, wv[e][2] = v.z, wv[e][3] = v.w;
                } else {
                    const uint2 v = *reinterpret_cast<const uint2 *>(src);
                    wv[e][0] = v.x, wv[e][1] = v.y;
                }
            }
            Sv[e] = st[vsof + trow * NBH];
        }
        // The operands are formed per lane (the width differs between lane
        // groups when a head mixes widths) and the MMAs issued after the
        // branches join: mma.sync needs the whole warp converged.
        const bool vfast = fast_scale(Sv[0]) && fast_scale(Sv[1]) && fast_scale(Sv[2]) && fast_scale(Sv[3]);
        const bool allfast = __all_sync(0xffffffffu, vfast);
        uint32_t xe0 = 0, xe1 = 0;
        Deq8 c0 = {0, 0, 0}, c1 = {0, 0, 0};
        float f[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (!allfast) {
#pragma unroll
            for (int e = 0; e < 4; ++e) f[e] = block_factor(Sv[e], vbv);
        } else if (vbv == 4) {
            xe0 = e4(Sv[0], Sv[1]), xe1 = e4(Sv[2], Sv[3]);
        } else {
            c0 = e8(Sv[0], Sv[1], vbv), c1 = e8(Sv[2], Sv[3], vbv);
        }
#pragma unroll
        for (int g4 = 0; g4 < NT / 4; ++g4) {  // n-tiles 4 g4 .. 4 g4 + 3 (dims of the V segment)
            uint32_t bA[4], bB[4];
            if (allfast) {
                if (vbv == 4) {  // bytes 2 g4, 2 g4 + 1 of each token: dims 4 g4 .. 4 g4 + 3
                    const uint32_t sel = (g4 & 1) ? 0x7632u : 0x5410u;
                    const uint32_t x0 = prmt(wv[0][g4 >> 1], wv[1][g4 >> 1], sel);
                    const uint32_t x1 = prmt(wv[2][g4 >> 1], wv[3][g4 >> 1], sel);
#pragma unroll
                    for (int e = 0; e < 4; ++e) bA[e] = deq4_pair(x0 >> (4 * e), xe0), bB[e] = deq4_pair(x1 >> (4 * e), xe1);
                } else {  // bytes 4 g4 .. 4 g4 + 3 (one word) of each token
                    const uint32_t x0l = prmt(wv[0][g4], wv[1][g4], 0x5410u), x0h = prmt(wv[0][g4], wv[1][g4], 0x7632u);
                    const uint32_t x1l = prmt(wv[2][g4], wv[3][g4], 0x5410u), x1h = prmt(wv[2][g4], wv[3][g4], 0x7632u);
                    bA[0] = deq8_pair(x0l, c0), bA[1] = deq8_pair(x0l >> 8, c0);
                    bA[2] = deq8_pair(x0h, c0), bA[3] = deq8_pair(x0h >> 8, c0);
                    bB[0] = deq8_pair(x1l, c1), bB[1] = deq8_pair(x1l >> 8, c1);
                    bB[2] = deq8_pair(x1h, c1), bB[3] = deq8_pair(x1h >> 8, c1);
                }
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = 4 * g4 + e;
                    bA[e] = pack_bf16((float)seg_code(wv[0], vbv, j) * f[0], (float)seg_code(wv[1], vbv, j) * f[1]);
                    bB[e] = pack_bf16((float)seg_code(wv[2], vbv, j) * f[2], (float)seg_code(wv[3], vbv, j) * f[3]);
                }
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) mma_bf16(acc[4 * g4 + e], A0, A1, A2, A3, bA[e], bB[e]);
        }
    }
    cp_async_wait<0>();
    __syncthreads();  // the ring is free: the merge reuses it

    // ---- merge the warps in warp order: per warp and head, max, sum, weighted sums
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, o);
        l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    }
    float *wm = reinterpret_cast<float *>(ring);  // [kWarps][8]
    float *wl = wm + kWarps * 8;                   // [kWarps][8]
    float *wacc = wl + kWarps * 8;                 // [kWarps][8][D]
    if (gi == 0) {
        wm[warp * 8 + 2 * q] = m0, wm[warp * 8 + 2 * q + 1] = m1;
        wl[warp * 8 + 2 * q] = l0, wl[warp * 8 + 2 * q + 1] = l1;
    }
    {
        float *row = wacc + (warp * 8 + gi) * D;
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            row[(2 * q) * NT + j] = acc[j][0] + acc[j][2];
            row[(2 * q + 1) * NT + j] = acc[j][1] + acc[j][3];
        }
    }
    __syncthreads();
    // A warp (or split) without tokens has max -inf, sum 0 and zero sums: its
    // weight is 0.  One whose scores were all NaN also has max -inf, but its
    // sum is NaN, which 0 * NaN carries into the result.
    const int bh = b * a.H_kv + hk;
    float *mypart = a.part + ((int64_t)bh * a.S + split) * G * D;
    float *mystat = a.stat + ((int64_t)bh * a.S + split) * G * 2;
    for (int idx = tid; idx < G * D; idx += kThreads) {
        const int g = idx / D, d = idx - g * D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, wm[w * 8 + g]);
        float num = 0.0f, den = 0.0f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const float mw = wm[w * 8 + g];
            const float e = mw == -INFINITY ? 0.0f : exp2f(mw - M);
            num = fmaf(e, wacc[(w * 8 + g) * D + d], num);
            den = fmaf(e, wl[w * 8 + g], den);
        }
        if (a.S == 1) {
            a.out[((int64_t)b * a.H + hk * G + g) * D + d] = (den != 0.0f || den != den) ? num / den : 0.0f;
        } else {
            mypart[g * D + d] = num;
            if (d == 0) mystat[2 * g] = M, mystat[2 * g + 1] = den;
        }
    }
    if (a.S == 1) return;

    // ---- the last CTA of (sequence, KV head) to arrive combines the splits in split order
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        const uint32_t old = atomicAdd(a.count + bh, 1u);
        sh_last = old == (uint32_t)(a.S - 1);
        if (sh_last) a.count[bh] = 0;  // every split has arrived: ready for the next launch
    }
    __syncthreads();
    if (!sh_last) return;
    __threadfence();
    const float *parts = a.part + (int64_t)bh * a.S * G * D;
    const float *stats = a.stat + (int64_t)bh * a.S * G * 2;
    float *sm = reinterpret_cast<float *>(ring);  // [S][G]: max, then weight
    float *sl = sm + kMaxSplits * kMaxG;          // [S][G]: sum
    float *sM = sl + kMaxSplits * kMaxG;          // [G]: max over the splits, then the total sum
    for (int i = tid; i < a.S * G; i += kThreads) {
        const float2 v = __ldcg(reinterpret_cast<const float2 *>(stats) + i);
        sm[i] = v.x, sl[i] = v.y;
    }
    __syncthreads();
    if (tid < G) {
        float M = -INFINITY;
        for (int s = 0; s < a.S; ++s) M = fmaxf(M, sm[s * G + tid]);
        sM[tid] = M;
    }
    __syncthreads();
    for (int i = tid; i < a.S * G; i += kThreads) sm[i] = sm[i] == -INFINITY ? 0.0f : exp2f(sm[i] - sM[i % G]);
    __syncthreads();
    if (tid < G) {
        float den = 0.0f;
        for (int s = 0; s < a.S; ++s) den = fmaf(sm[s * G + tid], sl[s * G + tid], den);
        sM[tid] = den;
    }
    __syncthreads();
    // four dimensions per thread, the splits in order (their loads independent)
    for (int idx = tid; idx < G * (D / 4); idx += kThreads) {
        const int g = idx / (D / 4), d4 = idx - g * (D / 4);
        const float4 *p = reinterpret_cast<const float4 *>(parts + g * D) + d4;
        const int64_t stride = (int64_t)G * D / 4;
        float4 num = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll 16
        for (int s = 0; s < a.S; ++s) {
            const float w = sm[s * G + g];
            const float4 v = __ldcg(p + s * stride);
            num.x = fmaf(w, v.x, num.x), num.y = fmaf(w, v.y, num.y);
            num.z = fmaf(w, v.z, num.z), num.w = fmaf(w, v.w, num.w);
        }
        const float den = sM[g];
        const bool some = den != 0.0f || den != den;
        float4 r = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (some) r = make_float4(num.x / den, num.y / den, num.z / den, num.w / den);
        *(reinterpret_cast<float4 *>(a.out + ((int64_t)b * a.H + hk * G + g) * D) + d4) = r;
    }
}

// byte offset of slot s in an activation code row: 4-bit slots as 16 B of nibbles, then 6/8-bit as 32 B
int64_t act_code_offset(const Plan &p, int s) {
    return s < p.n4 ? 16 * (int64_t)s : 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4);
}

int fill_map(const uint8_t *bits, int64_t K, uint16_t *off, uint8_t *b, uint8_t *slot, int64_t *row_bytes) {
    Plan p;
    const int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    for (int s = 0; s < p.nb; ++s) {
        const int kb = p.slot_block[s];
        off[kb] = (uint16_t)act_code_offset(p, s);
        b[kb] = (uint8_t)slot_width(p, s);
        slot[kb] = (uint8_t)s;
    }
    *row_bytes = p.row_bytes;
    return MXS_OK;
}

int64_t max_splits(int64_t T_cap) { return std::min<int64_t>(kMaxSplits, (T_cap + kTile - 1) / kTile); }

// the counters first (their place does not move with the sizes), then the partials
int64_t counter_bytes(int64_t B, int64_t H) { return (B * H * 4 + 255) / 256 * 256; }

int64_t sums_bytes(int64_t B, int64_t T_cap, int64_t H, int64_t D) {
    return B * H * max_splits(T_cap) * D * (int64_t)sizeof(float);
}

int64_t workspace_bytes(int64_t B, int64_t T_cap, int64_t H, int64_t D) {
    return counter_bytes(B, H) + sums_bytes(B, T_cap, H, D) + B * H * max_splits(T_cap) * 2 * (int64_t)sizeof(float);
}

template <int D>
size_t kernel_smem() {
    const size_t ring = (size_t)kStages * kTile * (D + D + 16 + 2 * (D / 32));
    const size_t merge = (size_t)kWarps * 8 * (D + 2) * sizeof(float);
    const size_t comb = (size_t)(2 * kMaxSplits * kMaxG + kMaxG) * sizeof(float);
    return std::max(ring, std::max(merge, comb));
}

template <int D>
int launch(AttnArgs &a, int B, int64_t T_cap, cudaStream_t st) {
    const size_t smem = kernel_smem<D>();
    cudaError_t e = cudaFuncSetAttribute(attention_decode_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(attention smem)");
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attention_decode_kernel<D>, kThreads, smem);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy query");
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return cuda_fail(e, "cudaDeviceGetAttribute(SM count)");
    // one wave: as many splits per (sequence, KV head) as fill the resident CTA slots
    const int64_t slots = (int64_t)std::max(1, per_sm) * sms;
    const int64_t s0 = std::max<int64_t>(1, std::min<int64_t>(max_splits(T_cap), slots / ((int64_t)B * a.H_kv)));
    const int64_t per = ((T_cap + s0 - 1) / s0 + kTile - 1) / kTile * kTile;  // tokens per split at T_cap
    a.S = (int)((T_cap + per - 1) / per);
    const dim3 grid((unsigned)a.S, (unsigned)a.H_kv, (unsigned)B);
    attention_decode_kernel<D><<<grid, kThreads, smem, st>>>(a);
    return cuda_fail(cudaGetLastError(), "attention_decode_kernel launch");
}

int attention_impl(const void *q, int64_t B, int64_t H, int64_t H_kv, int64_t D, const void *k_codes,
                   const uint8_t *k_scales, const uint8_t *k_bits, const void *v_codes, const uint8_t *v_scales,
                   const uint8_t *v_bits, const int32_t *lengths, int64_t T_cap, float scale, float *out,
                   void *workspace, size_t ws_bytes, void *stream) {
    if (D != 64 && D != 128) return fail(MXS_ERR_UNSUPPORTED, "head dimension D=%lld (64 or 128)", (long long)D);
    if (H < 1 || H_kv < 1 || H % H_kv != 0 || H / H_kv > kMaxG)
        return fail(MXS_ERR_SHAPE, "H=%lld, H_kv=%lld: H must be a multiple of H_kv, at most %d times",
                    (long long)H, (long long)H_kv, kMaxG);
    if (H_kv * D > 32 * kMaxKvBlocks)
        return fail(MXS_ERR_SHAPE, "H_kv * D = %lld > %d", (long long)(H_kv * D), 32 * kMaxKvBlocks);
    if (B < 1 || B > 65535) return fail(MXS_ERR_SHAPE, "B=%lld (1..65535)", (long long)B);
    if (T_cap < 1 || T_cap > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "T_cap=%lld", (long long)T_cap);
    if (!q || !k_codes || !k_scales || !v_codes || !v_scales || !out || !workspace)
        return fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (!std::isfinite(scale)) return fail(MXS_ERR_INVALID_ARG, "scale is not finite");
    if (reinterpret_cast<uintptr_t>(k_codes) % 16 || reinterpret_cast<uintptr_t>(v_codes) % 16 ||
        reinterpret_cast<uintptr_t>(workspace) % 16 || reinterpret_cast<uintptr_t>(out) % 16 ||
        reinterpret_cast<uintptr_t>(q) % 2 || reinterpret_cast<uintptr_t>(lengths) % 4)
        return fail(MXS_ERR_ALIGN, "code rows, out and workspace must be 16-byte aligned, lengths 4-byte aligned");
    const int64_t need = workspace_bytes(B, T_cap, H, D);
    if ((int64_t)ws_bytes < need)
        return fail(MXS_ERR_BUFFER, "workspace %zu < %lld bytes", ws_bytes, (long long)need);
    AttnArgs a;
    const int64_t K = H_kv * D;
    int rc = fill_map(k_bits, K, a.k_off, a.k_b, a.k_slot, &a.k_row);
    if (rc) return rc;
    if ((rc = fill_map(v_bits, K, a.v_off, a.v_b, a.v_slot, &a.v_row))) return rc;
    if ((rc = check_device())) return rc;
    a.q = static_cast<const uint16_t *>(q);
    a.kc = static_cast<const uint8_t *>(k_codes);
    a.ks = k_scales;
    a.vc = static_cast<const uint8_t *>(v_codes);
    a.vs = v_scales;
    a.lengths = lengths;
    a.count = static_cast<uint32_t *>(workspace);
    a.part = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + counter_bytes(B, H));
    a.stat = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + counter_bytes(B, H) +
                                       sums_bytes(B, T_cap, H, D));
    a.out = out;
    a.T_cap = T_cap;
    a.nb = (int)(K / 32);
    a.H = (int)H;
    a.H_kv = (int)H_kv;
    a.G = (int)(H / H_kv);
    a.sl2 = (float)((double)scale * 1.4426950408889634);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    return D == 128 ? launch<128>(a, (int)B, T_cap, st) : launch<64>(a, (int)B, T_cap, st);
}

}  // namespace
}  // namespace mxs

using namespace mxs;

extern "C" {

int64_t mxs_attention_decode_workspace_bytes(int64_t T, int64_t H, int64_t D) {
    if (T < 1 || H < 1 || D < 1) return -fail(MXS_ERR_SHAPE, "T, H, D must be positive");
    return workspace_bytes(1, T, H, D);
}

int64_t mxs_attention_decode_batch_workspace_bytes(int64_t B, int64_t T_cap, int64_t H, int64_t D) {
    if (B < 1 || T_cap < 1 || H < 1 || D < 1) return -fail(MXS_ERR_SHAPE, "B, T_cap, H, D must be positive");
    return workspace_bytes(B, T_cap, H, D);
}

int mxs_attention_decode(const void *q, int64_t H, int64_t H_kv, int64_t D, const void *k_codes,
                         const uint8_t *k_scales, const uint8_t *k_bits, const void *v_codes,
                         const uint8_t *v_scales, const uint8_t *v_bits, int64_t T, float scale, float *out,
                         void *workspace, size_t ws_bytes, void *stream) {
    if (T < 1 || T > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "T=%lld", (long long)T);
    return attention_impl(q, 1, H, H_kv, D, k_codes, k_scales, k_bits, v_codes, v_scales, v_bits, nullptr, T, scale,
                          out, workspace, ws_bytes, stream);
}

int mxs_attention_decode_batch(const void *q, int64_t B, int64_t H, int64_t H_kv, int64_t D, const void *k_codes,
                               const uint8_t *k_scales, const uint8_t *k_bits, const void *v_codes,
                               const uint8_t *v_scales, const uint8_t *v_bits, const int32_t *lengths, int64_t T_cap,
                               float scale, float *out, void *workspace, size_t ws_bytes, void *stream) {
    return attention_impl(q, B, H, H_kv, D, k_codes, k_scales, k_bits, v_codes, v_scales, v_bits, lengths, T_cap,
                          scale, out, workspace, ws_bytes, stream);
}

}  // extern "C"
