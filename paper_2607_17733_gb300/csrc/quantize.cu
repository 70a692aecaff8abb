// quantize.cu -- A1: on-the-fly MXINT quantization of bf16 activations.
//
// Sec. 4.1 (one mantissa width per 32-element block, widths 4/6/8) and
// Appendix A.2 (activations of every linear layer are quantized at run time).
// Four lanes own one 32-element block: each lane does one 128-bit load of
// 8 bf16, the block maximum is combined with two xor-shuffles, and every lane
// writes its share of the packed codes (4 B of nibbles or 8 B of int8), of the
// e4m3 MMA planes (8 B per digit plane) and of the scale bytes.  The work is
// enumerated in slot (grouped) order so the writes of a warp are contiguous;
// the reads are 64-byte runs of the source row.
#include "common.cuh"

namespace mxs {
namespace {

struct QuantArgs {
    const uint16_t *x;
    int64_t M, ld;
    int64_t V;            // work slots per row (with plane padding when planes are written)
    int rhaz;
    uint8_t *codes, *scales, *planes, *sf;
};

__global__ void __launch_bounds__(256) quantize_act_kernel(const __grid_constant__ Plan p,
                                                           const __grid_constant__ QuantArgs a) {
    // Programmatic dependent launch, both ways: a decode GEMM launched after
    // this kernel may start now (it waits for this grid before reading the
    // planes), and this grid waits for the kernel before it (which may write
    // x or still read the output buffers) before touching memory.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int l = threadIdx.x & 3;
    const int64_t item = gid >> 2;
    const int64_t row = item / a.V;
    const int vs = (int)(item - row * a.V);
    const bool in_grid = row < a.M;

    // virtual slot -> real slot (or padding) and its plane / scale-tile position
    int s = -1, st = 0, q = 0;
    int64_t poff = 0;
    if (a.planes) {
        if (vs < 4 * p.st4) {
            s = vs < p.n4 ? vs : -1;
            st = vs >> 2;
            q = vs & 3;
            poff = 32 * (int64_t)vs;
        } else {
            const int j = vs - 4 * p.st4;
            s = j < p.n68 ? p.n4 + j : -1;
            st = p.st4 + (j >> 1);
            q = j & 1;
            poff = 128 * (int64_t)p.st4 + 64 * (int64_t)j;
        }
    } else {
        s = vs;
    }
    const bool valid = in_grid && s >= 0 && row < a.M;
    // padding slots are written as zero digits: one plane in the 4-bit
    // region, two in the 6/8-bit region
    const int b = s >= 0 ? slot_width(p, s) : (vs < 4 * p.st4 ? 4 : 8);

    uint4 v = make_uint4(0, 0, 0, 0);
    if (valid) {
        const int kb = p.slot_block[s];
        const uint4 *src = reinterpret_cast<const uint4 *>(a.x + row * a.ld + kBlock * kb + 8 * l);
        v = __ldg(src);
    }
    uint32_t h[8] = {v.x & 0xFFFF, v.x >> 16, v.y & 0xFFFF, v.y >> 16,
                     v.z & 0xFFFF, v.z >> 16, v.w & 0xFFFF, v.w >> 16};
    uint32_t mag = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) mag = max(mag, h[i] & 0x7FFF);
    mag = max(mag, __shfl_xor_sync(0xffffffffu, mag, 1));
    mag = max(mag, __shfl_xor_sync(0xffffffffu, mag, 2));
    const int S = (int)(mag >> 7);
    if (!in_grid) return;

    int m[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) m[i] = (S == 255 || !valid) ? 0 : quant_elem(h[i], S, b, a.rhaz);

    if (valid && a.codes) {
        uint8_t *rowp = a.codes + row * p.row_bytes;
        if (b == 4) {
            uint32_t w = 0;
#pragma unroll
            for (int i = 0; i < 8; ++i) w |= (uint32_t)(m[i] & 0xF) << (4 * i);
            *reinterpret_cast<uint32_t *>(rowp + 16 * (int64_t)s + 4 * l) = w;
        } else {
            uint32_t w0 = 0, w1 = 0;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                w0 |= (uint32_t)(m[i] & 0xFF) << (8 * i);
                w1 |= (uint32_t)(m[i + 4] & 0xFF) << (8 * i);
            }
            *reinterpret_cast<uint2 *>(rowp + 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4) + 8 * l) =
                make_uint2(w0, w1);
        }
        if (l == 0) a.scales[row * p.nb + s] = (uint8_t)S;
    }

    if (a.planes) {
        if (row < a.M) {
            uint8_t *pr = a.planes + row * p.kp + poff + 8 * l;
            if (b == 4) {
                uint16_t c[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) c[i] = e4m3x2(0.25f * m[2 * i], 0.25f * m[2 * i + 1]);
                *reinterpret_cast<uint2 *>(pr) =
                    make_uint2(c[0] | ((uint32_t)c[1] << 16), c[2] | ((uint32_t)c[3] << 16));
            } else {
                const int sh = b == 6 ? 3 : 4;
                const float fh = b == 6 ? 0.5f : 0.25f, fl = b == 6 ? 0.0625f : 0.015625f;
                uint16_t ch[4], cl[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int h0 = m[2 * i] >> sh, h1 = m[2 * i + 1] >> sh;  // floor(m / 2^sh)
                    const int l0 = m[2 * i] & ((1 << sh) - 1), l1 = m[2 * i + 1] & ((1 << sh) - 1);
                    ch[i] = e4m3x2(fh * h0, fh * h1);
                    cl[i] = e4m3x2(fl * l0, fl * l1);
                }
                *reinterpret_cast<uint2 *>(pr) =
                    make_uint2(ch[0] | ((uint32_t)ch[1] << 16), ch[2] | ((uint32_t)ch[3] << 16));
                *reinterpret_cast<uint2 *>(pr + 32) =
                    make_uint2(cl[0] | ((uint32_t)cl[1] << 16), cl[2] | ((uint32_t)cl[3] << 16));
            }
        }
        // scale tile byte; 6/8-bit stages also clear their unused bytes 2 and 3
        const int64_t tile = row >> 7;
        const int r = (int)(row & 127);
        uint8_t *cell = a.sf + ((tile * p.nst + st) * 32 + (r & 31)) * 16 + 4 * (r >> 5);
        if (l == 0) cell[q] = (s >= 0 && row < a.M) ? (uint8_t)S : 0;
        if (l == 1 && st >= p.st4) cell[q + 2] = 0;
    }
}

}  // namespace

int launch_quantize(const Plan &p, const void *x, int64_t M, int64_t ld, int rounding, void *codes,
                    uint8_t *scales, void *planes, cudaStream_t st) {
    QuantArgs a;
    a.x = static_cast<const uint16_t *>(x);
    a.M = M;
    a.ld = ld;
    a.rhaz = rounding == MXS_RHAZ;
    a.codes = static_cast<uint8_t *>(codes);
    a.scales = scales;
    a.planes = static_cast<uint8_t *>(planes);
    a.sf = planes ? a.planes + align256(M * p.kp) : nullptr;
    a.V = planes ? 4 * (int64_t)p.st4 + 2 * (int64_t)((p.n68 + 1) / 2) : p.nb;
    const int64_t threads = M * a.V * 4;
    if (threads == 0) return MXS_OK;
    const int64_t blocks = (threads + 255) / 256;
    if (blocks > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "quantize: problem too large");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks, 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // the kernel waits before any access
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_fail(cudaLaunchKernelEx(&cfg, quantize_act_kernel, p, a), "quantize_act_kernel launch");
}

}  // namespace mxs
