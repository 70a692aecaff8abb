// pack.cu -- A2: offline quantization and packing of a weight matrix.
//
// Same MXINT rule as the activations (Appendix A.2: weights and activations
// of every linear layer are quantized; Sec. 4.1: one width per 32-element
// block).  One thread owns one (row, slot) block: it loads the 32 bf16 values
// with four 128-bit loads and writes the row's sign-magnitude codes and scale
// byte into its 128-row group (read by the decode kernel), and optionally the
// planes and scale tiles read by the tensor-core prefill kernel (4-bit blocks
// as e4m3 m/4, 6/8-bit blocks as their bf16 values).  The
// buffer is cleared first, so padding rows and slots read as zero.  This runs
// once per layer and is not on the timed path.
#include "common.cuh"

namespace mxs {
namespace {

struct PackArgs {
    const uint16_t *w;
    int64_t N, ld;
    int rhaz, with_planes;
    uint8_t *out;
    WeightOffsets off;
    const int32_t *perm;  // column order (Alg. 3): block kb holds columns perm[32 kb ..], or nullptr
};

__global__ void __launch_bounds__(256) pack_weight_kernel(const __grid_constant__ Plan p,
                                                          const __grid_constant__ PackArgs a) {
    const int64_t gid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t n = gid / p.nb;
    const int s = (int)(gid - n * p.nb);
    if (n >= a.N) return;
    const int kb = p.slot_block[s];
    const int b = slot_width(p, s);

    uint32_t h[32];
    uint32_t mag = 0;
    if (a.perm) {  // the block's 32 columns gathered in the allocation's order
        const int32_t *pc = a.perm + kBlock * kb;
        const uint32_t kmax = (uint32_t)(kBlock * p.nb - 1);  // an invalid order reads wrong columns, never outside the row
#pragma unroll
        for (int i = 0; i < 32; ++i) h[i] = __ldg(a.w + n * a.ld + min((uint32_t)__ldg(pc + i), kmax));
    } else {
        const uint4 *src = reinterpret_cast<const uint4 *>(a.w + n * a.ld + kBlock * kb);
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint4 u = __ldg(src + v);
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                h[8 * v + 2 * i] = w4[i] & 0xFFFF;
                h[8 * v + 2 * i + 1] = w4[i] >> 16;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) mag = max(mag, h[i] & 0x7FFF);
    const int S = (int)(mag >> 7);
    int m[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) m[i] = S == 255 ? 0 : quant_elem(h[i], S, b, a.rhaz);

    // sign-magnitude codes: (sign << 3) | |m| for 4 bits, (sign << 7) | |m| for 6/8 bits
    auto sm4 = [](int v) { return (uint32_t)(((v < 0) << 3) | (v < 0 ? -v : v)); };
    auto sm8 = [](int v) { return (uint32_t)(((v < 0) << 7) | (v < 0 ? -v : v)); };
    const int64_t grp = n >> 7;
    const int rr = (int)(n & 127);
    uint8_t *slot = a.out + grp * a.off.GB + slot_offset(p, s);
    if (b == 4) {
        // row word i: byte j = element 8i+j (low nibble) | element 8i+4+j (high nibble)
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            w[i] = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) w[i] |= (sm4(m[8 * i + j]) | (sm4(m[8 * i + 4 + j]) << 4)) << (8 * j);
        }
        *reinterpret_cast<uint4 *>(slot + 16 * rr) = make_uint4(w[0], w[1], w[2], w[3]);
        slot[2048 + rr] = (uint8_t)S;
    } else {
        uint32_t w[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            w[i] = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) w[i] |= sm8(m[4 * i + j]) << (8 * j);
        }
        uint4 *dst = reinterpret_cast<uint4 *>(slot + 32 * rr);
        dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
        dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
        slot[4096 + rr] = (uint8_t)S;
    }

    if (a.with_planes) {
        uint8_t *prow = a.out + a.off.planes + n * p.kp;
        int st, q;
        if (b == 4) {
            uint32_t *dst = reinterpret_cast<uint32_t *>(prow + 32 * (int64_t)s);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint16_t c0 = e4m3x2(0.25f * m[4 * i], 0.25f * m[4 * i + 1]);
                const uint16_t c1 = e4m3x2(0.25f * m[4 * i + 2], 0.25f * m[4 * i + 3]);
                dst[i] = c0 | ((uint32_t)c1 << 16);
            }
            st = s >> 2;
            q = s & 3;
        } else {  // the block's values m * 2^(S-127-(b-2)) in bf16 (exact), NaN for S = 255
            const int j = s - p.n4;
            uint32_t *dst = reinterpret_cast<uint32_t *>(prow + 128 * (int64_t)p.st4 + 64 * (int64_t)j);
            const float f = pow2f(S - 125 - b);
#pragma unroll
            for (int i = 0; i < 16; ++i)
                dst[i] = S == 255 ? 0x7FC07FC0u : bf16x2((float)m[2 * i] * f, (float)m[2 * i + 1] * f);
            st = p.st4 + (j >> 1);
            q = j & 1;
        }
        const int64_t tile = n >> 7;
        const int r = (int)(n & 127);
        a.out[a.off.sf + ((tile * p.nst + st) * 32 + (r & 31)) * 16 + 4 * (r >> 5) + q] = (uint8_t)S;
    }
}

}  // namespace

int launch_pack_weight(const Plan &p, const void *w, int64_t N, int64_t ld, int rounding, bool planes,
                       void *packed, cudaStream_t st, const int32_t *perm) {
    PackArgs a;
    a.perm = perm;
    a.w = static_cast<const uint16_t *>(w);
    a.N = N;
    a.ld = ld;
    a.rhaz = rounding == MXS_RHAZ;
    a.with_planes = planes;
    a.out = static_cast<uint8_t *>(packed);
    a.off = weight_offsets(p, N, planes);
    cudaError_t e = cudaMemsetAsync(packed, 0, (size_t)a.off.total, st);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync(packed)");
    const int64_t threads = N * p.nb;
    if (threads == 0) return MXS_OK;
    const int64_t blocks = (threads + 255) / 256;
    if (blocks > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "pack_weight: problem too large");
    pack_weight_kernel<<<(unsigned)blocks, 256, 0, st>>>(p, a);
    return cuda_fail(cudaGetLastError(), "pack_weight_kernel launch");
}

}  // namespace mxs
