// attention.cu -- decode attention over an MXINT-quantized KV cache.
//
// The paper quantizes the KV cache with a 4-8 bit configuration (Appendix
// A.2) and keeps Softmax in FP16.  The cache rows are written by
// mxs_quantize_act (one token's H_kv * D values per row, quantized along the
// row with the row's width map), so appending a token is one quantizer call
// into row t; this file reads the cache.  One query token, grouped-query heads
// (query head h reads KV head h / G):
//     s_t = scale * <q_h, k_t>,  out_h = sum_t softmax(s)_t * v_t.
// Work: a CTA owns one KV head and a chunk of 128 tokens and serves the G
// query heads of that KV head.  Thread t of the chunk dequantizes token t's K
// blocks of the head (element = code * 2^(S - 127 - (b - 2)), exact in fp32)
// and forms the G scores; the chunk's maxima and exponential sums follow by
// block reductions; the chunk's V blocks are staged in shared memory and
// thread d forms the G weighted sums of dimension d.  The per-chunk (max,
// sum, weighted sum) go to a workspace and a second kernel combines the chunks
// in order (deterministic).  HBM-bound: every cache byte of the layer is read
// once per step.
#include <cmath>

#include "common.cuh"

namespace mxs {
namespace {

constexpr int kChunk = 128;   // tokens per CTA (one per thread)
constexpr int kMaxG = 8;      // query heads per KV head
constexpr int kMaxKvBlocks = 256;  // H_kv * D / 32 (H_kv * D <= 8192)

struct AttnArgs {
    const uint16_t *q;  // [H, D] bf16
    const uint8_t *kc, *ks, *vc, *vs;  // codes [T, row bytes], scales [T, nb]
    int64_t k_row, v_row;  // row bytes of the K and V code rows
    int nb;                // blocks per row (H_kv * D / 32)
    int T, H, G, D;
    float scale;
    float *part;  // [chunks][H][D + 2]: weighted sums, then max and sum
    // per block of the row: byte offset of its codes in a code row, width, slot (scale index)
    uint16_t k_off[kMaxKvBlocks], v_off[kMaxKvBlocks];
    uint8_t k_b[kMaxKvBlocks], v_b[kMaxKvBlocks];
    uint8_t k_slot[kMaxKvBlocks], v_slot[kMaxKvBlocks];
};

// element i of a block whose codes start at p: nibble (4-bit, element 2j low) or int8
__device__ __forceinline__ int code_at(const uint8_t *p, int b, int i) {
    if (b == 4) {
        const int v = (p[i >> 1] >> ((i & 1) * 4)) & 0xF;
        return v >= 8 ? v - 16 : v;
    }
    return (int)(int8_t)p[i];
}
// element i (a compile-time index) of a block held in eight words
__device__ __forceinline__ int code_of(const uint32_t (&w)[8], int b, int i) {
    if (b == 4) {
        const uint32_t v = (w[i >> 3] >> (4 * (i & 7))) & 0xF;  // byte i/2, low nibble for even i
        return (int)(v << 28) >> 28;
    }
    return (int)(w[i >> 2] << (24 - 8 * (i & 3))) >> 24;
}
// 2^(S - 127 - (b - 2)) as a float (exact power of two; NaN for S = 255)
__device__ __forceinline__ float block_factor(int S, int b) {
    if (S == 255) return __int_as_float(0x7FC00000);
    const int e = S - 127 - (b - 2);  // in [-133, 125]
    return e >= -126 ? __int_as_float((e + 127) << 23) : ldexpf(1.0f, e);
}

template <int D>
__global__ void __launch_bounds__(kChunk) attention_chunk_kernel(const __grid_constant__ AttnArgs a) {
    constexpr int NBH = D / 32;  // blocks per head
    __shared__ float qs[kMaxG][D];
    __shared__ float p[kMaxG][kChunk];
    __shared__ float red[kMaxG][kChunk / 32];
    __shared__ float stat[kMaxG][2];
    __shared__ __align__(16) uint8_t vcode[kChunk][NBH][32];
    __shared__ float vfac[kChunk][NBH];
    const int hk = blockIdx.x, chunk = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = a.G;
    const int t = chunk * kChunk + tid;
    const bool live = t < a.T;

    for (int i = tid; i < G * D; i += kChunk) {
        const int g = i / D, d = i - g * D;
        qs[g][d] = __uint_as_float((uint32_t)a.q[(int64_t)(hk * G + g) * D + d] << 16);
    }
    // this token's V blocks of the head into shared memory, with their factors
    if (live) {
        const uint8_t *vrow = a.vc + (int64_t)t * a.v_row;
#pragma unroll
        for (int j = 0; j < NBH; ++j) {
            const int kb = hk * NBH + j;
            const int b = a.v_b[kb];
            const uint4 *src = reinterpret_cast<const uint4 *>(vrow + a.v_off[kb]);
            uint4 *dst = reinterpret_cast<uint4 *>(&vcode[tid][j][0]);
            dst[0] = __ldg(src);
            if (b != 4) dst[1] = __ldg(src + 1);
            vfac[tid][j] = block_factor(a.vs[(int64_t)t * a.nb + a.v_slot[kb]], b);
        }
    }
    __syncthreads();

    // scores of this token for the G query heads
    float s[kMaxG];
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) s[g] = 0.0f;
    if (live) {
        const uint8_t *krow = a.kc + (int64_t)t * a.k_row;
#pragma unroll
        for (int j = 0; j < NBH; ++j) {
            const int kb = hk * NBH + j;
            const int b = a.k_b[kb];
            uint32_t w[8];
            const uint4 *src = reinterpret_cast<const uint4 *>(krow + a.k_off[kb]);
            const uint4 u0 = __ldg(src);
            w[0] = u0.x, w[1] = u0.y, w[2] = u0.z, w[3] = u0.w;
            if (b != 4) {
                const uint4 u1 = __ldg(src + 1);
                w[4] = u1.x, w[5] = u1.y, w[6] = u1.z, w[7] = u1.w;
            }
            const float f = block_factor(a.ks[(int64_t)t * a.nb + a.k_slot[kb]], b);
            float dot[kMaxG];
#pragma unroll
            for (int g = 0; g < kMaxG; ++g) dot[g] = 0.0f;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const float c = (float)code_of(w, b, i);
#pragma unroll
                for (int g = 0; g < kMaxG; ++g)
                    if (g < G) dot[g] = fmaf(qs[g][32 * j + i], c, dot[g]);
            }
#pragma unroll
            for (int g = 0; g < kMaxG; ++g) s[g] = fmaf(dot[g], f, s[g]);
        }
    }
    // chunk maximum and exponential sum per query head
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) {
        if (g >= G) break;
        float v = live ? s[g] * a.scale : -INFINITY;
        s[g] = v;
        float m = v;
        for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane == 0) red[g][warp] = m;
    }
    __syncthreads();
    if (tid < G) {
        float m = red[tid][0];
        for (int w = 1; w < kChunk / 32; ++w) m = fmaxf(m, red[tid][w]);
        stat[tid][0] = m;
    }
    __syncthreads();
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) {
        if (g >= G) break;
        const float m = stat[g][0];
        const float e = live ? expf(s[g] - m) : 0.0f;
        p[g][tid] = e;
        float sum = e;
        for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) red[g][warp] = sum;
    }
    __syncthreads();
    if (tid < G) {
        float sum = 0.0f;
        for (int w = 0; w < kChunk / 32; ++w) sum += red[tid][w];
        stat[tid][1] = sum;
    }
    // weighted sums: thread d (< D) over the chunk's tokens in order
    const int nt = min(kChunk, a.T - chunk * kChunk);
    for (int d = tid; d < D; d += kChunk) {
        const int j = d >> 5, i = d & 31;
        float acc[kMaxG];
#pragma unroll
        for (int g = 0; g < kMaxG; ++g) acc[g] = 0.0f;
        const int b = a.v_b[hk * NBH + j];
        for (int tt = 0; tt < nt; ++tt) {
            const float v = (float)code_at(&vcode[tt][j][0], b, i) * vfac[tt][j];
#pragma unroll
            for (int g = 0; g < kMaxG; ++g)
                if (g < G) acc[g] = fmaf(p[g][tt], v, acc[g]);
        }
#pragma unroll
        for (int g = 0; g < kMaxG; ++g)
            if (g < G) a.part[((int64_t)chunk * a.H + hk * G + g) * (D + 2) + d] = acc[g];
    }
    __syncthreads();
    if (tid < G) {
        float *st = a.part + ((int64_t)chunk * a.H + hk * G + tid) * (D + 2) + D;
        st[0] = stat[tid][0];
        st[1] = stat[tid][1];
    }
}

// out[h][d] = sum_c w_c acc_c[d] / sum_c w_c l_c with w_c = exp(m_c - max_c m_c), chunks in order
__global__ void attention_combine_kernel(const float *part, int chunks, int H, int D, float *out) {
    const int h = blockIdx.x;
    float M = -INFINITY;
    for (int c = 0; c < chunks; ++c) M = fmaxf(M, part[((int64_t)c * H + h) * (D + 2) + D]);
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
        float num = 0.0f, den = 0.0f;
        for (int c = 0; c < chunks; ++c) {
            const float *pc = part + ((int64_t)c * H + h) * (D + 2);
            const float w = expf(pc[D] - M);
            num = fmaf(w, pc[d], num);
            den = fmaf(w, pc[D + 1], den);
        }
        out[(int64_t)h * D + d] = num / den;
    }
}

int64_t attention_chunks(int64_t T) { return (T + kChunk - 1) / kChunk; }

// byte offset of slot s in an activation code row: 4-bit slots as 16 B of nibbles, then 6/8-bit as 32 B
int64_t act_code_offset(const Plan &p, int s) { return s < p.n4 ? 16 * (int64_t)s : 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4); }

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

}  // namespace
}  // namespace mxs

using namespace mxs;

extern "C" {

int64_t mxs_attention_decode_workspace_bytes(int64_t T, int64_t H, int64_t D) {
    if (T < 1 || H < 1 || D < 1) return -fail(MXS_ERR_SHAPE, "T, H, D must be positive");
    return attention_chunks(T) * H * (D + 2) * (int64_t)sizeof(float);
}

int mxs_attention_decode(const void *q, int64_t H, int64_t H_kv, int64_t D, const void *k_codes,
                         const uint8_t *k_scales, const uint8_t *k_bits, const void *v_codes,
                         const uint8_t *v_scales, const uint8_t *v_bits, int64_t T, float scale, float *out,
                         void *workspace, size_t ws_bytes, void *stream) {
    if (D != 64 && D != 128) return fail(MXS_ERR_UNSUPPORTED, "head dimension D=%lld (64 or 128)", (long long)D);
    if (H < 1 || H_kv < 1 || H % H_kv != 0 || H / H_kv > kMaxG)
        return fail(MXS_ERR_SHAPE, "H=%lld, H_kv=%lld: H must be a multiple of H_kv, at most %d times",
                    (long long)H, (long long)H_kv, kMaxG);
    if (H_kv * D > 32 * kMaxKvBlocks) return fail(MXS_ERR_SHAPE, "H_kv * D = %lld > %d", (long long)(H_kv * D), 32 * kMaxKvBlocks);
    if (T < 1 || T > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "T=%lld", (long long)T);
    if (!q || !k_codes || !k_scales || !v_codes || !v_scales || !out || !workspace)
        return fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (!std::isfinite(scale)) return fail(MXS_ERR_INVALID_ARG, "scale is not finite");
    if (reinterpret_cast<uintptr_t>(k_codes) % 16 || reinterpret_cast<uintptr_t>(v_codes) % 16 ||
        reinterpret_cast<uintptr_t>(workspace) % 16 || reinterpret_cast<uintptr_t>(out) % 4 ||
        reinterpret_cast<uintptr_t>(q) % 2)
        return fail(MXS_ERR_ALIGN, "code rows and workspace must be 16-byte aligned");
    const int64_t need = mxs_attention_decode_workspace_bytes(T, H, D);
    if ((int64_t)ws_bytes < need) return fail(MXS_ERR_BUFFER, "workspace %zu < %lld bytes", ws_bytes, (long long)need);
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
    a.nb = (int)(K / 32);
    a.T = (int)T;
    a.H = (int)H;
    a.G = (int)(H / H_kv);
    a.D = (int)D;
    a.scale = scale;
    a.part = static_cast<float *>(workspace);
    const int64_t chunks = attention_chunks(T);
    if (chunks > 65535) return fail(MXS_ERR_SHAPE, "T=%lld too long", (long long)T);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const dim3 grid((unsigned)H_kv, (unsigned)chunks, 1);
    if (D == 128)
        attention_chunk_kernel<128><<<grid, kChunk, 0, st>>>(a);
    else
        attention_chunk_kernel<64><<<grid, kChunk, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "attention_chunk_kernel launch");
    attention_combine_kernel<<<(unsigned)H, 128, 0, st>>>(static_cast<const float *>(workspace), (int)chunks,
                                                          (int)H, (int)D, out);
    return cuda_fail(cudaGetLastError(), "attention_combine_kernel launch");
}

}  // extern "C"
