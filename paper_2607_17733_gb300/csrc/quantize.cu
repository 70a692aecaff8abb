// quantize.cu -- A1: on-the-fly MXINT quantization of bf16 activations.
//
// Sec. 4.1 (one mantissa width per 32-element block, widths 4/6/8) and
// Appendix A.2 (activations of every linear layer are quantized at run time).
// Two lanes own one 32-element block: each lane issues its two 128-bit loads
// (16 bf16) together, the block maximum is combined with one xor-shuffle, and
// every lane writes its half of the packed codes (8 B of nibbles or 16 B of
// int8), of the e4m3 MMA planes (16 B per digit plane) and of the scale bytes.
// The grid is two-dimensional -- y walks the rows, x the work slots of a row
// -- and the work is enumerated in slot (grouped) order, so the writes of a
// warp are contiguous and the reads are 64-byte runs of one source row.
//
// Arithmetic.  With E the block's shared exponent (S - 127), an element's
// mantissa is m = clamp(round(y), +-Q_b) where y = x * 2^(b-2-E).  y is a
// power-of-two scaling of a bf16 value, so it is exact, and a fused
// multiply-add with C = 1.5 * 2^23 rounds it: fma(x, 2^(b-2-E), C) rounds the
// exact x * 2^(b-2-E) + C once with unit spacing, to nearest even, so its
// result is C + RNE(y) (|y| < 2^(b-1) is far inside the +-2^22 where this
// holds) and its low bits are m in two's complement.  Ties away from zero
// instead floor |y| + 1/2 with a round-toward-zero addition of 2^23 (|y| +
// 1/2 is exact wherever its floor is not 0).  The MMA digits come from the
// same word: lo = m mod 2^sh is read from its low bits, hi = (m - lo) / 2^sh
// by exact float arithmetic, and both are converted to e4m3 exactly.
#include <algorithm>

#include "common.cuh"

namespace mxs {
namespace {

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: C + m has m in its low bits
constexpr float kTwo23 = 8388608.0f;
constexpr float kTwo22 = 4194304.0f;
constexpr int kCtaThreads = 256;

struct QuantArgs {
    const uint16_t *x;
    int64_t M, ld;
    int V;  // work slots per row (with plane padding when planes are written)
    uint8_t *codes, *scales, *planes, *sf;
};

// low bytes of four words, in order
__device__ __forceinline__ uint32_t low_bytes(uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    return __byte_perm(__byte_perm(a, b, 0x0040), __byte_perm(c, d, 0x0040), 0x5410);
}

template <bool kRhaz>
__global__ void __launch_bounds__(kCtaThreads) quantize_act_kernel(const __grid_constant__ Plan p,
                                                                   const __grid_constant__ QuantArgs a) {
    // Programmatic dependent launch, both ways: a decode GEMM launched after
    // this kernel may start now (it waits for this grid before reading the
    // planes), and this grid waits for the kernel before it (which may write
    // x or still read the output buffers) before touching memory.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int lane_in_row = blockIdx.x * blockDim.x + threadIdx.x;
    const int l = lane_in_row & 1;
    const int vs = lane_in_row >> 1;
    const bool in_row = vs < a.V;

    // virtual slot -> real slot (or padding) and its plane / scale-tile position
    int s = -1, st = 0, q = 0, poff = 0;
    if (a.planes) {
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
    const bool live = in_row && s >= 0;
    // padding slots are written as zero digits: one plane in the 4-bit
    // region, two in the 6/8-bit region
    const int b = s >= 0 ? slot_width(p, s) : (vs < 4 * p.st4 ? 4 : 8);
    const float Q = (float)((1 << (b - 1)) - 1);
    const int kb = live ? p.slot_block[s] : 0;

    // a warp lies in one row (blockDim.x is a multiple of 32), so the row
    // loop is warp-uniform and every lane reaches the shuffle
    for (int64_t row = (int64_t)blockIdx.y * blockDim.y + threadIdx.y; row < a.M;
         row += (int64_t)gridDim.y * blockDim.y) {
        uint4 v0 = make_uint4(0, 0, 0, 0), v1 = v0;
        if (live) {
            const uint4 *src = reinterpret_cast<const uint4 *>(a.x + row * a.ld + kBlock * kb + 16 * l);
            v0 = __ldg(src);
            v1 = __ldg(src + 1);
        }
        uint32_t w[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        uint32_t mx = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) mx = __vmaxu2(mx, w[i] & 0x7FFF7FFFu);
        mx = max(mx & 0xFFFFu, mx >> 16);
        mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        const int S = (int)(mx >> 7);  // E8M0 scale: the exponent field of the block maximum

        if (S == 255) {  // an Inf or NaN in the block: every code is 0
#pragma unroll
            for (int i = 0; i < 8; ++i) w[i] = 0;
        }
        float xf[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            xf[2 * i] = __uint_as_float(w[i] << 16);
            xf[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
        int k = 125 + b - S;  // b - 2 - E
        if (S < 8) {  // 2^k would not be a normal float: move 8 powers of two into x (exact)
#pragma unroll
            for (int j = 0; j < 16; ++j) xf[j] *= 256.0f;
            k -= 8;
        }
        const float f = __int_as_float((k + 127) << 23);

        float tf[16];  // C + m
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            if (kRhaz) {
                float r = __fadd_rz(fmaf(fabsf(xf[j]), f, 0.5f), kTwo23);  // 2^23 + floor(|y| + 1/2)
                r = fminf(r, kTwo23 + Q) - kTwo23;
                r = __uint_as_float(__float_as_uint(r) | (__float_as_uint(xf[j]) & 0x80000000u));
                tf[j] = kMagic + r;
            } else {
                tf[j] = fminf(fmaxf(fmaf(xf[j], f, kMagic), kMagic - Q), kMagic + Q);
            }
        }
        uint32_t tb[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) tb[j] = __float_as_uint(tf[j]);

        if (live && a.codes) {
            uint8_t *rowp = a.codes + row * p.row_bytes;
            if (b == 4) {
                uint32_t c[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const uint32_t ev = low_bytes(tb[8 * h], tb[8 * h + 2], tb[8 * h + 4], tb[8 * h + 6]);
                    const uint32_t od = low_bytes(tb[8 * h + 1], tb[8 * h + 3], tb[8 * h + 5], tb[8 * h + 7]);
                    c[h] = (ev & 0x0F0F0F0Fu) | ((od << 4) & 0xF0F0F0F0u);
                }
                *reinterpret_cast<uint2 *>(rowp + 16 * (int64_t)s + 8 * l) = make_uint2(c[0], c[1]);
            } else {
                uint4 c;
                c.x = low_bytes(tb[0], tb[1], tb[2], tb[3]);
                c.y = low_bytes(tb[4], tb[5], tb[6], tb[7]);
                c.z = low_bytes(tb[8], tb[9], tb[10], tb[11]);
                c.w = low_bytes(tb[12], tb[13], tb[14], tb[15]);
                *reinterpret_cast<uint4 *>(rowp + 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4) + 16 * l) = c;
            }
            if (l == 0) a.scales[row * p.nb + s] = (uint8_t)S;
        }

        if (in_row && a.planes) {
            uint8_t *pr = a.planes + row * p.kp + poff + 16 * l;
            if (b == 4) {  // one plane of m / 4
                uint32_t c[8];
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    c[i] = e4m3x2(fmaf(tf[2 * i], 0.25f, -0.25f * kMagic), fmaf(tf[2 * i + 1], 0.25f, -0.25f * kMagic));
                *reinterpret_cast<uint4 *>(pr) =
                    make_uint4(c[0] | (c[1] << 16), c[2] | (c[3] << 16), c[4] | (c[5] << 16), c[6] | (c[7] << 16));
            } else {  // m = 2^sh * hi + lo: planes hi * 2^sh * fl and lo * fl
                const uint32_t mask = b == 6 ? 7u : 15u;
                const float fl = b == 6 ? 0.0625f : 0.015625f;
                float hs[16], ls[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const float L = __uint_as_float((tb[j] & mask) | 0x4B000000u);  // 2^23 + lo
                    ls[j] = fmaf(L, fl, -fl * kTwo23);
                    hs[j] = fmaf(tf[j] - L, fl, -fl * kTwo22);  // tf - L = 2^22 + (m - lo), exact
                }
                uint32_t ch[8], cl[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    ch[i] = e4m3x2(hs[2 * i], hs[2 * i + 1]);
                    cl[i] = e4m3x2(ls[2 * i], ls[2 * i + 1]);
                }
                *reinterpret_cast<uint4 *>(pr) =
                    make_uint4(ch[0] | (ch[1] << 16), ch[2] | (ch[3] << 16), ch[4] | (ch[5] << 16), ch[6] | (ch[7] << 16));
                *reinterpret_cast<uint4 *>(pr + 32) =
                    make_uint4(cl[0] | (cl[1] << 16), cl[2] | (cl[3] << 16), cl[4] | (cl[5] << 16), cl[6] | (cl[7] << 16));
            }
            // scale tile byte; 6/8-bit stages also clear their unused bytes 2 and 3
            const int64_t tile = row >> 7;
            const int r = (int)(row & 127);
            uint8_t *cell = a.sf + ((tile * p.nst + st) * 32 + (r & 31)) * 16 + 4 * (r >> 5);
            if (l == 0) cell[q] = s >= 0 ? (uint8_t)S : 0;
            if (l == 1 && st >= p.st4) cell[q + 2] = 0;
        }
    }
}

}  // namespace

int launch_quantize(const Plan &p, const void *x, int64_t M, int64_t ld, int rounding, void *codes,
                    uint8_t *scales, void *planes, cudaStream_t st) {
    QuantArgs a;
    a.x = static_cast<const uint16_t *>(x);
    a.M = M;
    a.ld = ld;
    a.codes = static_cast<uint8_t *>(codes);
    a.scales = scales;
    a.planes = static_cast<uint8_t *>(planes);
    a.sf = planes ? a.planes + align256(M * p.kp) : nullptr;
    a.V = planes ? 4 * p.st4 + 2 * ((p.n68 + 1) / 2) : p.nb;
    if (M == 0 || a.V == 0) return MXS_OK;
    // a row's 2V lanes: one CTA of whole warps for short rows (several rows
    // to a CTA), else the fewest CTAs of at most 256 threads, evenly filled
    const int T = 2 * a.V;
    int nx = 1, tx, ry = 1;
    if (T <= kCtaThreads) {
        tx = (T + 31) / 32 * 32;
        ry = kCtaThreads / tx;
    } else {
        nx = (T + kCtaThreads - 1) / kCtaThreads;
        tx = ((T + nx - 1) / nx + 31) / 32 * 32;
    }
    const int64_t gy = std::min<int64_t>((M + ry - 1) / ry, 65535);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)nx, (unsigned)gy, 1);
    cfg.blockDim = dim3((unsigned)tx, (unsigned)ry, 1);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // the kernel waits before any access
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = rounding == MXS_RHAZ ? cudaLaunchKernelEx(&cfg, quantize_act_kernel<true>, p, a)
                                               : cudaLaunchKernelEx(&cfg, quantize_act_kernel<false>, p, a);
    return cuda_fail(e, "quantize_act_kernel launch");
}

}  // namespace mxs
