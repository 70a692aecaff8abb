// quantize.cu -- A1: on-the-fly MXINT quantization of bf16 activations.
//
// Sec. 4.1 (one mantissa width per 32-element block, widths 4/6/8) and
// Appendix A.2 (activations of every linear layer are quantized at run time).
// One lane owns one 32-element block: it issues its four 128-bit loads
// together, finds the block maximum with packed bf16 max instructions, and
// writes its block's packed codes (16 B of nibbles or 32 B of int8), its MMA
// plane (32 B of e4m3 m/4 for a 4-bit block, 64 B of bf16 values for a
// 6/8-bit one) and its scale byte.  The work is
// enumerated in slot (grouped) order, so a warp writes 32 consecutive slots
// of one row and the lanes of one K' stage combine their scale bytes into
// one 32-bit word of the scale tile.  The grid is rows x slots.
//
// Arithmetic.  With E the block's shared exponent (S - 127), an element's
// mantissa is m = clamp(round(y), +-Q_b) where y = x * 2^(b-2-E).
//  * The clamp is applied to x, two elements per instruction: the bound
//    Q_b * 2^(E+2-b) is a bf16 value (Q_b has at most 7 significant bits),
//    so clamped elements scale to exactly +-Q_b and the others are unchanged.
//  * y is a power-of-two scaling of a bf16 value, so it is exact, and a fused
//    multiply-add with C = 1.5 * 2^23 rounds it: fma(x, 2^(b-2-E), C) rounds
//    the exact x * 2^(b-2-E) + C once with unit spacing, to nearest even, so
//    its result is C + RNE(y) (|y| <= Q_b is far inside the +-2^22 where
//    this holds) and its low bits are m in two's complement.  Ties away from
//    zero instead floor |y| + 1/2 with a round-toward-zero addition of 2^23
//    (|y| + 1/2 is exact wherever its floor is not 0).
//  * The MMA planes come from the same word: m/4 converted to e4m3, or
//    m * 2^(S-127-(b-2)) converted to bf16, both exactly.
// Blocks whose maximum is below 2^-119 (S < 8) take a slower path: 2^(b-2-E)
// is then not a normal float, so x is first scaled by 2^8 (exact) and the
// clamp is done in float.
#include <algorithm>

#include "common.cuh"

namespace mxs {
namespace {

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: C + m has m in its low bits
constexpr float kTwo23 = 8388608.0f;
constexpr int kCtaThreads = 256;

struct QuantArgs {
    const uint16_t *x;
    int64_t M, ld;
    int V;  // work slots per row (with plane padding when planes are written)
    uint8_t *codes, *scales, *planes, *sf;
    const int32_t *perm;  // column order (Alg. 3): block kb holds columns perm[32 kb ..], or nullptr
};

// low bytes of four words, in order
__device__ __forceinline__ uint32_t low_bytes(uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    return __byte_perm(__byte_perm(a, b, 0x0040), __byte_perm(c, d, 0x0040), 0x5410);
}
// max of |a|, |b| per bf16 half, NaN-propagating (the sign bits of the result are not used)
__device__ __forceinline__ uint32_t bf2_max_abs(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.NaN.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}
// two fused multiply-adds (each rounded once, to nearest even) in one instruction
__device__ __forceinline__ void fma2(float &d0, float &d1, float a0, float a1, float b0, float b1, float c0, float c1) {
    asm("{\n .reg .b64 a, b, c, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n mov.b64 c, {%6, %7};\n"
        " fma.rn.f32x2 d, a, b, c;\n mov.b64 {%0, %1}, d;\n}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ uint32_t bf2_clamp(uint32_t w, uint32_t hi, uint32_t lo) {
    uint32_t r;
    asm("min.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(w), "r"(hi));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(r), "r"(lo));
    return r;
}

template <bool kCodes, bool kPlanes, bool kRhaz, bool kPerm>
__device__ __forceinline__ void quantize_rows(const Plan &p, const QuantArgs &a) {
    // work slot vs -> real slot (or plane padding), its plane offset and its
    // scale byte (K' stage st, byte q of the stage's scale word)
    const int vs = blockIdx.x * blockDim.x + threadIdx.x;
    if ((vs & ~31) >= a.V) return;  // a warp with no slot of the row (uniform: blockDim.x is a multiple of 32)
    int s, st = 0, q = 0, poff = 0;
    if (kPlanes) {
        if (vs < 4 * p.st4) {
            s = vs < p.n4 ? vs : -1;
            st = vs >> 2;
            q = vs & 3;
            poff = 32 * vs;
        } else {
            const int j = vs - 4 * p.st4;
            s = j < p.n68 ? p.n4 + j : -1;
            st = p.st4 + (j >> 1);
            q = j & 1;
            poff = 128 * p.st4 + 64 * j;
        }
    } else {
        s = vs;
    }
    const bool in_row = vs < a.V;
    const bool live = in_row && s >= 0;
    // padding slots are written as zeros: 32 plane bytes in the 4-bit region,
    // 64 in the 6/8-bit region
    const int b = s >= 0 ? slot_width(p, s) : (vs < 4 * p.st4 ? 4 : 8);
    const float Q = (float)((1 << (b - 1)) - 1);
    const int kb = live ? p.slot_block[s] : 0;
    // the lane that writes its K' stage's scale word: the first of 4 (4-bit) or 2 (6/8-bit)
    const bool sf_writer = q == 0;
    const bool stage4 = st < p.st4;

    // a warp lies in one row (blockDim.x is a multiple of 32), so the row
    // loop is warp-uniform and every lane reaches the shuffles
    for (int64_t row = (int64_t)blockIdx.y * blockDim.y + threadIdx.y; row < a.M;
         row += (int64_t)gridDim.y * blockDim.y) {
        uint32_t w[16];
        if (kPerm && live) {  // the block's 32 columns gathered in the allocation's order
            const int4 *pc = reinterpret_cast<const int4 *>(a.perm + kBlock * kb);
            const uint16_t *xr = a.x + row * a.ld;
            const uint32_t kmax = (uint32_t)(kBlock * p.nb - 1);  // an invalid order reads wrong columns, never outside the row
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int4 c = __ldg(pc + i);
                w[2 * i] = (uint32_t)__ldg(xr + min((uint32_t)c.x, kmax)) | ((uint32_t)__ldg(xr + min((uint32_t)c.y, kmax)) << 16);
                w[2 * i + 1] =
                    (uint32_t)__ldg(xr + min((uint32_t)c.z, kmax)) | ((uint32_t)__ldg(xr + min((uint32_t)c.w, kmax)) << 16);
            }
        } else if (live) {
            const uint4 *src = reinterpret_cast<const uint4 *>(a.x + row * a.ld + kBlock * kb);
            const uint4 v0 = __ldg(src), v1 = __ldg(src + 1), v2 = __ldg(src + 2), v3 = __ldg(src + 3);
            w[0] = v0.x, w[1] = v0.y, w[2] = v0.z, w[3] = v0.w, w[4] = v1.x, w[5] = v1.y, w[6] = v1.z, w[7] = v1.w;
            w[8] = v2.x, w[9] = v2.y, w[10] = v2.z, w[11] = v2.w, w[12] = v3.x, w[13] = v3.y, w[14] = v3.z,
            w[15] = v3.w;
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = 0;
        }
        uint32_t mx = bf2_max_abs(w[0], w[1]);
#pragma unroll
        for (int i = 2; i < 16; ++i) mx = bf2_max_abs(mx, w[i]);
        mx = max(mx & 0x7FFFu, (mx >> 16) & 0x7FFFu);
        const int S = (int)(mx >> 7);  // E8M0 scale: the exponent field of the block maximum

        // k = b - 2 - E.  Blocks below 2^-119 scale x by 2^8 first (k - 8);
        // empty blocks (all zero, padding) use k = 0, which codes them as 0.
        const bool tiny = S < 8 && mx != 0;
        const int k = mx == 0 ? 0 : (tiny ? 117 + b - S : 125 + b - S);
        const float f = __int_as_float((k + 127) << 23);
        // the clamp bound Q * 2^-k (bf16-exact), for x and for 2^8 x; an Inf
        // or NaN in the block (S = 255) clamps every element to 0
        const float T = Q * __int_as_float((127 - k) << 23);
        if (!tiny) {
            const uint32_t t = S == 255 ? 0u : __float_as_uint(T) >> 16;
            const uint32_t hi = t | (t << 16), lo = hi | 0x80008000u;
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = bf2_clamp(w[i], hi, lo);
        }

        uint4 pl[4];  // 4-bit: plane halves in pl[0..1]; 6/8-bit: hi halves pl[0..1], lo halves pl[2..3]
                      // (bf16 form: elements 0-15 in pl[0..1], 16-31 in pl[2..3])
        uint4 cd[2];  // codes: 4-bit in cd[0]; 8-bit halves in cd[0..1]
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            float xf[16];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                xf[2 * i] = __uint_as_float(w[8 * h + i] << 16);
                xf[2 * i + 1] = __uint_as_float(w[8 * h + i] & 0xFFFF0000u);
            }
            if (tiny) {
#pragma unroll
                for (int j = 0; j < 16; ++j) xf[j] = fminf(fmaxf(xf[j] * 256.0f, -T), T);
            }
            float tf[16];  // C + m
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
                if (kRhaz) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        float r = __fadd_rz(fmaf(fabsf(xf[j + e]), f, 0.5f), kTwo23) - kTwo23;  // floor(|y| + 1/2)
                        r = __uint_as_float(__float_as_uint(r) | (__float_as_uint(xf[j + e]) & 0x80000000u));
                        tf[j + e] = kMagic + r;
                    }
                } else {
                    fma2(tf[j], tf[j + 1], xf[j], xf[j + 1], f, f, kMagic, kMagic);
                }
            }
            uint32_t tb[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) tb[j] = __float_as_uint(tf[j]);

            if (kCodes) {
                if (b == 4) {
                    uint32_t c[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const uint32_t ev = low_bytes(tb[8 * e], tb[8 * e + 2], tb[8 * e + 4], tb[8 * e + 6]);
                        const uint32_t od = low_bytes(tb[8 * e + 1], tb[8 * e + 3], tb[8 * e + 5], tb[8 * e + 7]);
                        c[e] = (ev & 0x0F0F0F0Fu) | ((od << 4) & 0xF0F0F0F0u);
                    }
                    if (h == 0) cd[0].x = c[0], cd[0].y = c[1];
                    else cd[0].z = c[0], cd[0].w = c[1];
                } else {
                    cd[h] = make_uint4(low_bytes(tb[0], tb[1], tb[2], tb[3]), low_bytes(tb[4], tb[5], tb[6], tb[7]),
                                       low_bytes(tb[8], tb[9], tb[10], tb[11]),
                                       low_bytes(tb[12], tb[13], tb[14], tb[15]));
                }
            }
            if (kPlanes) {
                if (b == 4) {  // one plane of m / 4
                    uint32_t c[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        float v0, v1;
                        fma2(v0, v1, tf[2 * i], tf[2 * i + 1], 0.25f, 0.25f, -0.25f * kMagic, -0.25f * kMagic);
                        c[i] = e4m3x2(v0, v1);
                    }
                    pl[h] = make_uint4(c[0] | (c[1] << 16), c[2] | (c[3] << 16), c[4] | (c[5] << 16),
                                       c[6] | (c[7] << 16));
                } else {  // the block's values m * 2^(S-127-(b-2)) in bf16 (exact)
                    const float fs = pow2f(S - 125 - b);
                    uint32_t cw[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        cw[i] = S == 255 ? 0x7FC07FC0u
                                         : bf16x2((tf[2 * i] - kMagic) * fs, (tf[2 * i + 1] - kMagic) * fs);
                    pl[2 * h] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
                    pl[2 * h + 1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
                }
            }
        }

        if (kCodes && live) {
            uint8_t *rowp = a.codes + row * p.row_bytes;
            if (b == 4) {
                *reinterpret_cast<uint4 *>(rowp + 16 * (int64_t)s) = cd[0];
            } else {
                uint4 *dst = reinterpret_cast<uint4 *>(rowp + 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4));
                dst[0] = cd[0];
                dst[1] = cd[1];
            }
            a.scales[row * p.nb + s] = (uint8_t)S;
        }
        if (kPlanes) {
            // the scale word of a K' stage row: bytes q = 0..3 (4-bit) or
            // 0..1 then two zero bytes (6/8-bit), from the stage's lanes
            const uint32_t sb = live ? (uint32_t)S : 0u;
            const uint32_t s1 = __shfl_down_sync(0xffffffffu, sb, 1);
            const uint32_t s2 = __shfl_down_sync(0xffffffffu, sb, 2);
            const uint32_t s3 = __shfl_down_sync(0xffffffffu, sb, 3);
            if (in_row) {
                uint4 *pr = reinterpret_cast<uint4 *>(a.planes + row * p.kp + poff);
                pr[0] = pl[0];
                pr[1] = pl[1];
                if (b != 4) {
                    pr[2] = pl[2];
                    pr[3] = pl[3];
                }
                if (sf_writer) {
                    const int64_t tile = row >> 7;
                    const int r = (int)(row & 127);
                    const uint32_t word = stage4 ? sb | (s1 << 8) | (s2 << 16) | (s3 << 24) : sb | (s1 << 8);
                    *reinterpret_cast<uint32_t *>(a.sf + ((tile * p.nst + st) * 32 + (r & 31)) * 16 + 4 * (r >> 5)) =
                        word;
                }
            }
        }
    }
}

// Decode shapes (M <= 16): each thread's block of x into L2 before the wait
// for the kernel before.  Every write lands in L2, so a block that kernel
// still writes is read afresh after the wait; otherwise the loads after the
// wait find it there (larger M: the quantizer is bandwidth-bound and the
// prefetch would only compete with the kernel before for L2).
template <bool kPlanes, bool kPerm>
__device__ __forceinline__ void prefetch_x(const Plan &p, const QuantArgs &a) {
    if (kPerm || a.M > 16) return;
    const int vs = blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t row = (int64_t)blockIdx.y * blockDim.y + threadIdx.y;
    if (vs >= a.V || row >= a.M) return;
    int s = vs;
    if (kPlanes) {
        const int j = vs - 4 * p.st4;
        s = vs < 4 * p.st4 ? (vs < p.n4 ? vs : -1) : (j < p.n68 ? p.n4 + j : -1);
    }
    if (s < 0) return;
    const uint16_t *src = a.x + row * a.ld + kBlock * (int64_t)p.slot_block[s];
    asm volatile("prefetch.global.L2 [%0];" ::"l"(src));
    asm volatile("prefetch.global.L2 [%0];" ::"l"(src + kBlock - 1));
}

// Programmatic dependent launch, both ways: a decode GEMM launched after
// these kernels may start at once (it waits for them before reading the
// planes), and they wait for the kernel before them (which may write x or
// still read the output buffers) before touching memory.
template <bool kCodes, bool kPlanes, bool kRhaz, bool kPerm>
__global__ void __launch_bounds__(kCtaThreads) quantize_act_kernel(const __grid_constant__ Plan p,
                                                                   const __grid_constant__ QuantArgs a) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    prefetch_x<kPlanes, kPerm>(p, a);
    asm volatile("griddepcontrol.wait;" ::: "memory");
    quantize_rows<kCodes, kPlanes, kRhaz, kPerm>(p, a);
}

// The activations of up to three layers (a grouped decode GEMM, or prefill
// layers that read one hidden state), quantized to MMA planes in one launch
// (blockIdx.z = problem): one link in the launch chain instead of one per
// problem.
struct QuantGroup {
    Plan p[3];
    QuantArgs a[3];
};
template <bool kRhaz>
__global__ void __launch_bounds__(kCtaThreads) quantize_act_group_kernel(const __grid_constant__ QuantGroup g) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    prefetch_x<true, false>(g.p[blockIdx.z], g.a[blockIdx.z]);
    asm volatile("griddepcontrol.wait;" ::: "memory");
    quantize_rows<false, true, kRhaz, false>(g.p[blockIdx.z], g.a[blockIdx.z]);
}

#ifndef MXS_QUANT_WARP_CTAS
#define MXS_QUANT_WARP_CTAS 1
#endif
// CTA shape for rows of V work slots: one CTA of whole warps for short rows
// (several rows to a CTA), else the fewest CTAs of at most 256 threads
void quant_shape(int V, int64_t M, int &nx, int &tx, int &ry, int64_t &gy) {
    nx = 1, ry = 1;
    if (MXS_QUANT_WARP_CTAS && M <= 16) {
        tx = 32;
        nx = (V + 31) / 32;
    } else if (V <= kCtaThreads) {
        tx = (V + 31) / 32 * 32;
        ry = kCtaThreads / tx;
    } else {
        nx = (V + kCtaThreads - 1) / kCtaThreads;
        tx = ((V + nx - 1) / nx + 31) / 32 * 32;
    }
    gy = std::min<int64_t>((M + ry - 1) / ry, 65535);
}

}  // namespace

int launch_quantize_group(const Plan *const *plans, const void *const *x, const int64_t *ld, int64_t M, int rounding,
                          void *const *planes, int count, cudaStream_t st) {
    if (count < 1 || count > 3) return fail(MXS_ERR_INVALID_ARG, "quantize group of %d", count);
    thread_local QuantGroup g;  // host staging of the parameter block (the launch copies it)
    static_assert(sizeof(QuantGroup) < 32000, "kernel parameter block too large");
    int Vmax = 0;
    for (int i = 0; i < 3; ++i) {
        const int k = i < count ? i : 0;
        const Plan &p = *plans[k];
        g.p[i] = p;
        QuantArgs &a = g.a[i];
        a = QuantArgs{};
        a.x = static_cast<const uint16_t *>(x[k]);
        a.M = M;
        a.ld = ld[k];
        a.planes = static_cast<uint8_t *>(planes[k]);
        a.sf = a.planes + align256(M * p.kp);
        a.V = 4 * p.st4 + 2 * ((p.n68 + 1) / 2);
        Vmax = std::max(Vmax, a.V);
    }
    if (M == 0 || Vmax == 0) return MXS_OK;
    int nx, tx, ry;
    int64_t gy;
    quant_shape(Vmax, M, nx, tx, ry, gy);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)nx, (unsigned)gy, (unsigned)count);
    cfg.blockDim = dim3((unsigned)tx, (unsigned)ry, 1);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = rounding == MXS_RHAZ ? cudaLaunchKernelEx(&cfg, quantize_act_group_kernel<true>, g)
                                               : cudaLaunchKernelEx(&cfg, quantize_act_group_kernel<false>, g);
    return cuda_fail(e, "quantize_act_group_kernel launch");
}

int launch_quantize(const Plan &p, const void *x, int64_t M, int64_t ld, int rounding, void *codes,
                    uint8_t *scales, void *planes, cudaStream_t st, const int32_t *perm) {
    QuantArgs a;
    a.perm = perm;
    a.x = static_cast<const uint16_t *>(x);
    a.M = M;
    a.ld = ld;
    a.codes = static_cast<uint8_t *>(codes);
    a.scales = scales;
    a.planes = static_cast<uint8_t *>(planes);
    a.sf = planes ? a.planes + align256(M * p.kp) : nullptr;
    a.V = planes ? 4 * p.st4 + 2 * ((p.n68 + 1) / 2) : p.nb;
    if (M == 0 || a.V == 0) return MXS_OK;
    int nx, tx, ry;
    int64_t gy;
    quant_shape(a.V, M, nx, tx, ry, gy);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)nx, (unsigned)gy, 1);
    cfg.blockDim = dim3((unsigned)tx, (unsigned)ry, 1);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // the kernel waits before any access
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    using Kernel = void (*)(Plan, QuantArgs);
    static const Kernel kernels[2][3][2] = {
        {{quantize_act_kernel<true, false, false, false>, quantize_act_kernel<true, false, true, false>},
         {quantize_act_kernel<false, true, false, false>, quantize_act_kernel<false, true, true, false>},
         {quantize_act_kernel<true, true, false, false>, quantize_act_kernel<true, true, true, false>}},
        {{quantize_act_kernel<true, false, false, true>, quantize_act_kernel<true, false, true, true>},
         {quantize_act_kernel<false, true, false, true>, quantize_act_kernel<false, true, true, true>},
         {quantize_act_kernel<true, true, false, true>, quantize_act_kernel<true, true, true, true>}}};
    const int which = !planes ? 0 : (!codes ? 1 : 2);
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernels[perm != nullptr][which][rounding == MXS_RHAZ], p, a);
    return cuda_fail(e, "quantize_act_kernel launch");
}

}  // namespace mxs
