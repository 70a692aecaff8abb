// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens).
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale), with the per-block widths of Sec. 4.1.
//
// Decode is bound by the weight stream, so the kernel is built around it:
//   * weights are read once, in the 16-row fragment tiles of the compact
//     layout: one 8-byte (4-bit) or 16-byte (6/8-bit) vector load per lane per
//     block gives the lane its A operand of a 16x8x32 integer warp MMA;
//     a 4-bit tile is widened with two masks (each nibble becomes 16*m in the
//     high half of an int8), the factor 16 is folded into the scale;
//   * the few token rows sit in shared memory, already in B-operand order;
//   * each block's exact int32 dot is folded into fp32 accumulators as
//     acc += (float)dot * 2^Ew' * 2^Ea' (powers of two built from the scale
//     bytes, so only the final add rounds);
//   * K is split over the warps of a CTA (summed through shared memory) and,
//     for small N, over the CTAs of a thread-block cluster (summed through
//     distributed shared memory by the cluster's rank 0, in rank order), so
//     no global workspace and no second launch are needed.
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
    int M, N, T;           // T = 16-row tiles
    int R, KS, GS;         // row tiles per CTA, warps per row tile, CTAs per cluster (K split)
    int chunk;             // slots per CTA (GS split)
    int64_t o8, os;
};

__device__ __forceinline__ void mma_s8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%10,%10,%10,%10};"
        : "=r"(d[0]), "=r"(d[1]), "=r"(d[2]), "=r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "r"(0));
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

// sign-extend 4 nibbles (given as the low nibbles of two bytes each: v holds
// elements e0..e3 of a 4-bit activation block in bytes 0..1) into 4 int8
__device__ __forceinline__ uint32_t widen4(uint32_t two_bytes) {
    uint32_t out = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        int nib = (two_bytes >> (4 * i)) & 0xF;
        nib = nib >= 8 ? nib - 16 : nib;
        out |= (uint32_t)(nib & 0xFF) << (8 * i);
    }
    return out;
}

template <int NT, int U>
__global__ void __launch_bounds__(256) gemm_decode_kernel(const __grid_constant__ Plan p,
                                                          const __grid_constant__ DecodeArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int chunk = a.chunk;
    uint2 *actf = reinterpret_cast<uint2 *>(smem);                        // [chunk][NT][32]
    float *fa = reinterpret_cast<float *>(smem + (size_t)chunk * NT * 256);  // [chunk][16]
    float *red = fa + (size_t)chunk * 16;                                  // [8 warps][NT*128]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, q = lane & 3;
    const int rank = blockIdx.y;  // position in the K split (== cluster rank)
    const int c0 = rank * chunk;
    const int c1 = min(p.nb, c0 + chunk);

    // ---- stage the token rows of this CTA's slot range in B-operand order
    for (int it = threadIdx.x; it < (c1 - c0) * NT * 32; it += blockDim.x) {
        const int c = it / (NT * 32), rem = it - c * NT * 32;
        const int nt = rem >> 5, ln = rem & 31;
        const int s = c0 + c;
        const int tok = 8 * nt + (ln >> 2), qq = ln & 3;
        uint2 v = make_uint2(0, 0);
        if (tok < a.M) {
            const uint8_t *row = a.codes + (int64_t)tok * p.row_bytes;
            if (s < p.n4) {
                const uint8_t *blk = row + 16 * (int64_t)s;
                const uint32_t lo = *reinterpret_cast<const uint16_t *>(blk + 2 * qq);
                const uint32_t hi = *reinterpret_cast<const uint16_t *>(blk + 8 + 2 * qq);
                v = make_uint2(widen4(lo), widen4(hi));
            } else {
                const uint8_t *blk = row + 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4);
                v = make_uint2(*reinterpret_cast<const uint32_t *>(blk + 4 * qq),
                               *reinterpret_cast<const uint32_t *>(blk + 16 + 4 * qq));
            }
        }
        actf[(c * NT + nt) * 32 + ln] = v;
    }
    for (int it = threadIdx.x; it < (c1 - c0) * 16; it += blockDim.x) {
        const int c = it >> 4, tok = it & 15, s = c0 + c;
        const int b = slot_width(p, s);
        float f = 0.f;
        if (tok < a.M) {
            const int S = a.scales[(int64_t)tok * p.nb + s];
            // 2^(E - (b-2)), with the 1/16 of the widened 4-bit weights folded in
            f = S == 255 ? __int_as_float(0x7fc00000) : pow2f(S - 127 - (b - 2) - (b == 4 ? 4 : 0));
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

    if (rt < a.R && t < a.T) {
        const uint8_t *sc0 = a.w + a.os + (int64_t)(16 * t + g) * p.nb;
        const uint8_t *sc1 = sc0 + 8 * (int64_t)p.nb;

        auto fold = [&](int s, const uint32_t (&af)[4], int b) {
            const int S0 = __ldg(sc0 + s), S1 = __ldg(sc1 + s);
            const float f0 = S0 == 255 ? __int_as_float(0x7fc00000) : pow2f(S0 - 127 - (b - 2));
            const float f1 = S1 == 255 ? __int_as_float(0x7fc00000) : pow2f(S1 - 127 - (b - 2));
            const int c = s - c0;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const uint2 bf = actf[(c * NT + nt) * 32 + lane];
                int d[4];
                mma_s8(d, af, bf.x, bf.y);
                const float2 ft = *reinterpret_cast<const float2 *>(fa + c * 16 + 8 * nt + 2 * q);
                acc[nt][0] = fmaf((float)d[0] * f0, ft.x, acc[nt][0]);
                acc[nt][1] = fmaf((float)d[1] * f0, ft.y, acc[nt][1]);
                acc[nt][2] = fmaf((float)d[2] * f1, ft.x, acc[nt][2]);
                acc[nt][3] = fmaf((float)d[3] * f1, ft.y, acc[nt][3]);
            }
        };

        // 4-bit slots
        {
            const int s_beg = w0, s_end = min(w1, p.n4);
            const uint8_t *base = a.w + ((int64_t)t * p.n4) * 256 + 8 * lane;
            int s = s_beg;
            for (; s + U <= s_end; s += U) {
                uint2 wv[U];
#pragma unroll
                for (int u = 0; u < U; ++u) wv[u] = ldg_stream8(base + (int64_t)(s + u) * 256);
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const uint32_t af[4] = {wv[u].x & 0xF0F0F0F0u, wv[u].y & 0xF0F0F0F0u,
                                            (wv[u].x << 4) & 0xF0F0F0F0u, (wv[u].y << 4) & 0xF0F0F0F0u};
                    fold(s + u, af, 4);
                }
            }
            for (; s < s_end; ++s) {
                const uint2 wv = ldg_stream8(base + (int64_t)s * 256);
                const uint32_t af[4] = {wv.x & 0xF0F0F0F0u, wv.y & 0xF0F0F0F0u, (wv.x << 4) & 0xF0F0F0F0u,
                                        (wv.y << 4) & 0xF0F0F0F0u};
                fold(s, af, 4);
            }
        }
        // 6/8-bit slots
        {
            const int s_beg = max(w0, p.n4), s_end = w1;
            const uint8_t *base = a.w + a.o8 + (int64_t)t * p.n68 * 512 + 16 * lane;  // slot n4
            int s = s_beg;
            for (; s + U / 2 <= s_end; s += U / 2) {
                uint4 wv[U / 2];
#pragma unroll
                for (int u = 0; u < U / 2; ++u) wv[u] = ldg_stream16(base + (int64_t)(s + u - p.n4) * 512);
#pragma unroll
                for (int u = 0; u < U / 2; ++u) {
                    const uint32_t af[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
                    fold(s + u, af, slot_width(p, s + u));
                }
            }
            for (; s < s_end; ++s) {
                const uint4 wv = ldg_stream16(base + (int64_t)(s - p.n4) * 512);
                const uint32_t af[4] = {wv.x, wv.y, wv.z, wv.w};
                fold(s, af, slot_width(p, s));
            }
        }
    }

    // ---- sum the KS warps of each row tile (fixed order) into warp kw == 0's slot
    float *mine = red + warp * (NT * 128);
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) mine[(nt * 4 + i) * 32 + lane] = acc[nt][i];
    __syncthreads();
    for (int e = threadIdx.x; e < a.R * NT * 128; e += blockDim.x) {
        const int r = e / (NT * 128), off = e - r * NT * 128;
        float sum = 0.f;
        for (int k = 0; k < a.KS; ++k) sum += red[(r * a.KS + k) * (NT * 128) + off];
        red[(r * a.KS) * (NT * 128) + off] = sum;
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
    int R, KS, GS, chunk;
};

// Split policy.  Decode streams every weight byte once; the grid needs enough
// warps in flight to cover HBM latency.  Prefer whole-K CTAs; split K across
// a cluster only when N is too small to fill the machine or the token rows of
// the slot range would not fit in shared memory.
DecodeShape pick_shape(const Plan &p, int NT, int64_t T) {
    const int sms = 152;
    DecodeShape best{1, 8, 8, (p.nb + 7) / 8};
    for (int GS = 1; GS <= 8; GS *= 2) {
        const int chunk = (p.nb + GS - 1) / GS;
        const size_t smem = (size_t)chunk * (NT * 256 + 64) + kWarps * NT * 512;
        if (smem > 110 * 1024) continue;
        for (int R = 8; R >= 1; R /= 2) {
            const int64_t ctas = (T + R - 1) / R * GS;
            if (ctas >= 2 * sms || (R == 1 && GS == 8)) {
                return DecodeShape{R, kWarps / R, GS, chunk};
            }
        }
    }
    return best;
}

template <int NT>
int launch_nt(const Plan &p, const DecodeArgs &a0, cudaStream_t st) {
    DecodeArgs a = a0;
    const DecodeShape sh = pick_shape(p, NT, a.T);
    a.R = sh.R;
    a.KS = sh.KS;
    a.GS = sh.GS;
    a.chunk = sh.chunk;
    const size_t smem = (size_t)a.chunk * (NT * 256 + 64) + kWarps * NT * 512;
    auto kern = gemm_decode_kernel<NT, 8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((a.T + a.R - 1) / a.R), (unsigned)a.GS, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.dynamicSmemBytes = smem;
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
