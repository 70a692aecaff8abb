// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens).
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale), with the per-block widths of Sec. 4.1.
//
// Decode is bound by the weight stream, so the kernel is built around it:
//   * weights are read once, in the 16-row fragment tiles of the compact
//     layout: one 8-byte (4-bit) or 16-byte (6/8-bit) vector load per lane per
//     block gives the lane its A operand of a 16x8x32 warp MMA;
//   * the integer products run on the FP8 warp MMA (e4m3 x e4m3 -> fp32):
//     an e4m3 byte with exponent field <= 1 is exactly k * 2^-9 for its low
//     four bits k (subnormals, then the first binade), so a sign-magnitude code
//     with |m| <= 15 IS the e4m3 encoding of m * 2^-9 once its sign bit is
//     moved to bit 7.  4-bit codes take two bit operations per four elements;
//     6/8-bit codes are split |m| = 16h + l into two such digits (Sec. 6: a
//     high- and a low-precision part multiplied separately), four MMAs per
//     block combined as 256*hh + 16*(hl + lh) + ll;
//   * every block's product is therefore exact in fp32 (|dot| < 2^19, in units
//     of 2^-18) and is folded into fp32 accumulators as
//     acc += dot * 2^(Ew' + Ea' + 18), the power of two built from the scale
//     bytes, so only that add rounds;
//   * the token rows sit in shared memory, already as e4m3 B operands;
//   * K is split over the warps of a CTA (summed through shared memory) and,
//     for small N, over the CTAs of a thread-block cluster (summed through
//     distributed shared memory by the cluster's rank 0, in rank order), so no
//     global workspace and no second launch are needed.
#include <algorithm>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {
namespace {

constexpr int kWarps = 8;

struct DecodeArgs {
    const uint8_t *codes;   // [M, row_bytes]
    const uint8_t *scales;  // [M, nb]
    const uint8_t *w;       // packed weight buffer
    float *y;
    int64_t ld_y;
    int M, N, T;   // T = 16-row tiles
    int R, KS, GS; // row tiles per CTA, warps per row tile, CTAs per cluster (K split)
    int chunk;     // slots per CTA (GS split)
    int max4, max8;  // most 4-bit / 6-8-bit slots any CTA's chunk holds (shared-memory carve)
    int64_t o8, os;
};

__device__ __forceinline__ void mma_e4m3(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1,
                                         const float (&c)[4]) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%10,%11,%12,%13};"
        : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(c[0]), "f"(c[1]), "f"(c[2]),
          "f"(c[3]));
}

__device__ __forceinline__ uint2 ldg_stream8(const void *p) {
    uint2 r;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(p));
    return r;
}
__device__ __forceinline__ uint4 ldg_stream16(const void *p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// e4m3 bytes of m * 2^-9 for four sign-magnitude 4-bit codes held in the high
// nibbles (hi) or the low nibbles (lo) of the four bytes of x
__device__ __forceinline__ uint32_t e4m3_hi_nibbles(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t e4m3_lo_nibbles(uint32_t x) { return (x & 0x07070707u) | ((x << 4) & 0x80808080u); }
// the two digits of four sign-magnitude 8-bit codes: high (|m| >> 4) and low (|m| & 15)
__device__ __forceinline__ uint32_t e4m3_hi_digit(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t e4m3_lo_digit(uint32_t x) { return x & 0x8F8F8F8Fu; }

// e4m3 byte of m * 2^-9 for a two's-complement activation code (|m| <= 127
// gives the low digit / high digit split used for 6/8-bit blocks)
__device__ __forceinline__ uint32_t act_digit(int m, int which /*0: whole (|m|<=15), 1: high, 2: low*/) {
    const uint32_t s = m < 0 ? 0x80u : 0u;
    const uint32_t a = (uint32_t)(m < 0 ? -m : m);
    const uint32_t v = which == 0 ? a : (which == 1 ? (a >> 4) : (a & 15u));
    return s | v;
}

template <int NT, int U>
__global__ void __launch_bounds__(256) gemm_decode_kernel(const __grid_constant__ Plan p,
                                                          const __grid_constant__ DecodeArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint2 *act4 = reinterpret_cast<uint2 *>(smem);                                          // [max4][NT][32]
    uint4 *act8 = reinterpret_cast<uint4 *>(smem + (size_t)a.max4 * NT * 256);              // [max8][NT][32]
    float *fa = reinterpret_cast<float *>(smem + (size_t)a.max4 * NT * 256 + (size_t)a.max8 * NT * 512);  // [chunk][16]
    float *red = fa + (size_t)a.chunk * 16;                                                 // [8 warps][NT*128]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, q = lane & 3;
    const int rank = blockIdx.y;  // position in the K split (== cluster rank)
    const int c0 = rank * a.chunk;
    const int c1 = min(p.nb, c0 + a.chunk);
    const int s4 = min(max(c0, 0), p.n4), e4 = min(c1, p.n4);  // 4-bit slots [s4, e4)
    const int s8 = max(c0, p.n4);                              // 6/8-bit slots [s8, c1)

    // ---- stage the token rows of this CTA's slot range as e4m3 B operands
    for (int it = threadIdx.x; it < (c1 - c0) * NT * 32; it += blockDim.x) {
        const int c = it / (NT * 32), rem = it - c * NT * 32;
        const int nt = rem >> 5, ln = rem & 31;
        const int s = c0 + c;
        const int tok = 8 * nt + (ln >> 2), qq = ln & 3;
        if (s < p.n4) {
            uint2 v = make_uint2(0, 0);
            if (tok < a.M) {
                const uint8_t *blk = a.codes + (int64_t)tok * p.row_bytes + 16 * (int64_t)s;
                const uint32_t lo = *reinterpret_cast<const uint16_t *>(blk + 2 * qq);      // elements 4q..4q+3
                const uint32_t hi = *reinterpret_cast<const uint16_t *>(blk + 8 + 2 * qq);  // 16+4q..16+4q+3
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    int m0 = (lo >> (4 * i)) & 0xF, m1 = (hi >> (4 * i)) & 0xF;
                    m0 = m0 >= 8 ? m0 - 16 : m0;
                    m1 = m1 >= 8 ? m1 - 16 : m1;
                    v.x |= act_digit(m0, 0) << (8 * i);
                    v.y |= act_digit(m1, 0) << (8 * i);
                }
            }
            act4[((s - s4) * NT + nt) * 32 + ln] = v;
        } else {
            uint4 v = make_uint4(0, 0, 0, 0);
            if (tok < a.M) {
                const uint8_t *blk = a.codes + (int64_t)tok * p.row_bytes + 16 * (int64_t)p.n4 +
                                     32 * (int64_t)(s - p.n4);
                const uint32_t w0 = *reinterpret_cast<const uint32_t *>(blk + 4 * qq);
                const uint32_t w1 = *reinterpret_cast<const uint32_t *>(blk + 16 + 4 * qq);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int m0 = (int)(int8_t)(w0 >> (8 * i)), m1 = (int)(int8_t)(w1 >> (8 * i));
                    v.x |= act_digit(m0, 1) << (8 * i);
                    v.y |= act_digit(m1, 1) << (8 * i);
                    v.z |= act_digit(m0, 2) << (8 * i);
                    v.w |= act_digit(m1, 2) << (8 * i);
                }
            }
            act8[((s - s8) * NT + nt) * 32 + ln] = v;
        }
    }
    for (int it = threadIdx.x; it < (c1 - c0) * 16; it += blockDim.x) {
        const int c = it >> 4, tok = it & 15, s = c0 + c;
        const int b = slot_width(p, s);
        float f = 0.f;
        if (tok < a.M) {
            const int S = a.scales[(int64_t)tok * p.nb + s];
            // 2^(Ea' + 18): the operands carry m * 2^-9 on both sides
            f = S == 255 ? __int_as_float(0x7fc00000) : pow2f(S - 127 - (b - 2) + 18);
        }
        fa[it] = f;
    }
    __syncthreads();

    // ---- this warp: row tile t, slot sub-range [w0, w1)
    const int rt = warp / a.KS, kw = warp - rt * a.KS;
    const int t = blockIdx.x * a.R + rt;
    const int span = (c1 - c0 + a.KS - 1) / a.KS;
    const int w0 = c0 + kw * span, w1 = min(c1, w0 + span);

    float acc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;

    if (t < a.T) {
        const uint8_t *sc0 = a.w + a.os + (int64_t)(16 * t + g) * p.nb;
        const uint8_t *sc1 = sc0 + 8 * (int64_t)p.nb;
        const float zero[4] = {0.f, 0.f, 0.f, 0.f};

        auto fold = [&](int s, int b, int nt, const float (&d)[4]) {
            const int S0 = __ldg(sc0 + s), S1 = __ldg(sc1 + s);
            const float f0 = S0 == 255 ? __int_as_float(0x7fc00000) : pow2f(S0 - 127 - (b - 2));
            const float f1 = S1 == 255 ? __int_as_float(0x7fc00000) : pow2f(S1 - 127 - (b - 2));
            const float2 ft = *reinterpret_cast<const float2 *>(fa + (s - c0) * 16 + 8 * nt + 2 * q);
            acc[nt][0] = fmaf(d[0], f0 * ft.x, acc[nt][0]);
            acc[nt][1] = fmaf(d[1], f0 * ft.y, acc[nt][1]);
            acc[nt][2] = fmaf(d[2], f1 * ft.x, acc[nt][2]);
            acc[nt][3] = fmaf(d[3], f1 * ft.y, acc[nt][3]);
        };
        auto block4 = [&](int s, uint2 wv) {
            const uint32_t af[4] = {e4m3_hi_nibbles(wv.x), e4m3_hi_nibbles(wv.y), e4m3_lo_nibbles(wv.x),
                                    e4m3_lo_nibbles(wv.y)};
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint2 bf = act4[((s - s4) * NT + nt) * 32 + lane];
                float d[4];
                mma_e4m3(d, af, bf.x, bf.y, zero);
                fold(s, 4, nt, d);
            }
        };
        auto block8 = [&](int s, uint4 wv) {
            const uint32_t ah[4] = {e4m3_hi_digit(wv.x), e4m3_hi_digit(wv.y), e4m3_hi_digit(wv.z),
                                    e4m3_hi_digit(wv.w)};
            const uint32_t al[4] = {e4m3_lo_digit(wv.x), e4m3_lo_digit(wv.y), e4m3_lo_digit(wv.z),
                                    e4m3_lo_digit(wv.w)};
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint4 bf = act8[((s - s8) * NT + nt) * 32 + lane];  // x,y: high digit; z,w: low digit
                float hh[4], x[4], ll[4], d[4];
                mma_e4m3(hh, ah, bf.x, bf.y, zero);
                mma_e4m3(x, ah, bf.z, bf.w, zero);
                mma_e4m3(x, al, bf.x, bf.y, x);
                mma_e4m3(ll, al, bf.z, bf.w, zero);
#pragma unroll
                for (int i = 0; i < 4; ++i) d[i] = fmaf(256.f, hh[i], fmaf(16.f, x[i], ll[i]));  // exact
                fold(s, slot_width(p, s), nt, d);
            }
        };

        // 4-bit slots
        {
            const int s_beg = max(w0, s4), s_end = min(w1, e4);
            const uint8_t *base = a.w + ((int64_t)t * p.n4) * 256 + 8 * lane;
            int s = s_beg;
            for (; s + U <= s_end; s += U) {
                uint2 wv[U];
#pragma unroll
                for (int u = 0; u < U; ++u) wv[u] = ldg_stream8(base + (int64_t)(s + u) * 256);
#pragma unroll
                for (int u = 0; u < U; ++u) block4(s + u, wv[u]);
            }
            for (; s < s_end; ++s) block4(s, ldg_stream8(base + (int64_t)s * 256));
        }
        // 6/8-bit slots
        {
            const int s_beg = max(w0, s8), s_end = w1;
            const uint8_t *base = a.w + a.o8 + (int64_t)t * p.n68 * 512 + 16 * lane;  // slot n4
            int s = s_beg;
            for (; s + U / 2 <= s_end; s += U / 2) {
                uint4 wv[U / 2];
#pragma unroll
                for (int u = 0; u < U / 2; ++u) wv[u] = ldg_stream16(base + (int64_t)(s + u - p.n4) * 512);
#pragma unroll
                for (int u = 0; u < U / 2; ++u) block8(s + u, wv[u]);
            }
            for (; s < s_end; ++s) block8(s, ldg_stream16(base + (int64_t)(s - p.n4) * 512));
        }
    }

    // ---- sum the KS warps of each row tile (fixed order) into warp kw == 0's slot
    float *mine = red + warp * (NT * 128);
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) mine[(nt * 4 + i) * 32 + lane] = acc[nt][i];
    __syncthreads();
    if (a.KS > 1) {
        for (int e = threadIdx.x; e < a.R * NT * 128; e += blockDim.x) {
            const int r = e / (NT * 128), off = e - r * NT * 128;
            float sum = 0.f;
            for (int k = 0; k < a.KS; ++k) sum += red[(r * a.KS + k) * (NT * 128) + off];
            red[(r * a.KS) * (NT * 128) + off] = sum;
        }
    }

    // ---- sum over the cluster's CTAs (K split) in rank order, then store
    auto store = [&](int r, int off, float v) {
        const int nt = off / 128, rem = off - nt * 128;
        const int i = rem >> 5, ln = rem & 31;
        const int tok = 8 * nt + 2 * (ln & 3) + (i & 1);
        const int n = 16 * (blockIdx.x * a.R + r) + (ln >> 2) + 8 * (i >> 1);
        if (tok < a.M && n < a.N && blockIdx.x * a.R + r < a.T) a.y[(int64_t)tok * a.ld_y + n] = v;
    };
    if (a.GS == 1) {
        __syncthreads();
        for (int e = threadIdx.x; e < a.R * NT * 128; e += blockDim.x) {
            const int r = e / (NT * 128), off = e - r * NT * 128;
            store(r, off, red[(r * a.KS) * (NT * 128) + off]);
        }
    } else {
        cg::cluster_group cluster = cg::this_cluster();
        cluster.sync();
        if (cluster.block_rank() == 0) {
            for (int e = threadIdx.x; e < a.R * NT * 128; e += blockDim.x) {
                const int r = e / (NT * 128), off = e - r * NT * 128;
                float sum = 0.f;
                for (int k = 0; k < a.GS; ++k) {
                    const float *peer = cluster.map_shared_rank(red, k);
                    sum += peer[(r * a.KS) * (NT * 128) + off];
                }
                store(r, off, sum);
            }
        }
        cluster.sync();  // peers keep their shared memory until rank 0 has read it
    }
}

struct DecodeShape {
    int R, KS, GS, chunk, max4, max8;
    size_t smem;
};

DecodeShape shape_for(const Plan &p, int NT, int R, int GS) {
    DecodeShape sh;
    sh.R = R;
    sh.KS = kWarps / R;
    sh.GS = GS;
    sh.chunk = (p.nb + GS - 1) / GS;
    sh.max4 = sh.max8 = 0;
    for (int r = 0; r < GS; ++r) {
        const int c0 = r * sh.chunk, c1 = std::min(p.nb, c0 + sh.chunk);
        const int n4c = std::max(0, std::min(c1, p.n4) - c0);
        sh.max4 = std::max(sh.max4, n4c);
        sh.max8 = std::max(sh.max8, std::max(0, c1 - c0) - n4c);
    }
    sh.smem = (size_t)sh.max4 * NT * 256 + (size_t)sh.max8 * NT * 512 + (size_t)sh.chunk * 64 + kWarps * NT * 512;
    return sh;
}

// Split policy.  Decode streams every weight byte once; the grid needs enough
// warps in flight to cover HBM latency.  Prefer whole-K CTAs; split K across
// a cluster only when N is too small to fill the machine or the token rows of
// the slot range would not fit in shared memory.
DecodeShape pick_shape(const Plan &p, int NT, int64_t T) {
    const int sms = 152;
    for (int GS = 1; GS <= 8; GS *= 2) {
        for (int R = 8; R >= 1; R /= 2) {
            const DecodeShape sh = shape_for(p, NT, R, GS);
            if (sh.smem > 110 * 1024) break;
            const int64_t ctas = (T + R - 1) / R * GS;
            if (ctas >= 2 * sms) return sh;
        }
    }
    return shape_for(p, NT, 1, 8);
}

template <int NT>
int launch_nt(const Plan &p, const DecodeArgs &a0, cudaStream_t st) {
    DecodeArgs a = a0;
    const DecodeShape sh = pick_shape(p, NT, a.T);
    a.R = sh.R;
    a.KS = sh.KS;
    a.GS = sh.GS;
    a.chunk = sh.chunk;
    a.max4 = sh.max4;
    a.max8 = sh.max8;
    if (sh.smem > 220 * 1024) return fail(MXS_ERR_SHAPE, "decode: K too large for the shared-memory plan");
    auto kern = gemm_decode_kernel<NT, 8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((a.T + a.R - 1) / a.R), (unsigned)a.GS, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = sh.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = (unsigned)a.GS;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, p, a);
    return cuda_fail(e, "gemm_decode_kernel launch");
}

}  // namespace

int64_t decode_workspace_bytes(const Plan &, int64_t, int64_t) { return 0; }

int launch_gemm_decode(const Plan &p, const void *codes, const uint8_t *scales, const void *packed, int64_t M,
                       int64_t N, float *y, int64_t ld_y, void *, size_t, cudaStream_t st) {
    DecodeArgs a = {};
    a.codes = static_cast<const uint8_t *>(codes);
    a.scales = scales;
    a.w = static_cast<const uint8_t *>(packed);
    a.y = y;
    a.ld_y = ld_y;
    a.M = (int)M;
    a.N = (int)N;
    a.T = (int)((N + 15) / 16);
    const WeightOffsets off = weight_offsets(p, N, false);
    a.o8 = off.o8;
    a.os = off.os;
    if (N > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
    return M <= 8 ? launch_nt<1>(p, a, st) : launch_nt<2>(p, a, st);
}

}  // namespace mxs
