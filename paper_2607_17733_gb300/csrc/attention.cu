// attention.cu -- decode attention over an MXINT-quantized KV cache.
//
// The paper quantizes the KV cache with a 4-8 bit configuration (Appendix
// A.2) and keeps Softmax in FP16.  The cache rows are written by
// mxs_quantize_act (one token's H_kv * D values per row, quantized along the
// row with the row's width map), so appending a token is one quantizer call
// into row t; this file reads the cache.  One query token, grouped-query heads
// (query head h reads KV head h / G):
//     s_t = scale * <q_h, k_t>,  out_h = sum_t softmax(s)_t * v_t.
// Work: a CTA owns one KV head and a chunk of 64 tokens and serves the G
// query heads of that KV head.  Two threads per token dequantize its K blocks
// of the head (element = code * 2^(S - 127 - (b - 2)), exact in fp32) and form
// the G scores; one warp per head forms the chunk's maximum and exponential
// sum; the chunk's V blocks are staged in shared memory, each lane owns D/32
// dimensions and the four warps split the tokens, their sums added in warp
// order.  The per-chunk (max,
// sum, weighted sum) go to a workspace and a second kernel combines the chunks
// in order (deterministic).  HBM-bound: every cache byte of the layer is read
// once per step.
#include <cmath>

#include "common.cuh"

namespace mxs {
namespace {

constexpr int kChunk = 64;    // tokens per CTA
constexpr int kThreads = 128; // two score threads per token; four warps share the weighted sums
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

template <int D, int G>
__global__ void __launch_bounds__(kThreads) attention_chunk_kernel(const __grid_constant__ AttnArgs a) {
    constexpr int NBH = D / 32;   // blocks per head
    constexpr int DL = D / 32;    // dimensions per lane in the weighted sums
    constexpr int HALF = NBH / 2; // blocks per score thread (two threads per token)
    __shared__ __align__(16) float qs[G][D];
    __shared__ __align__(16) uint8_t vcode[kChunk][NBH][32];
    __shared__ float vfac[kChunk][NBH];
    __shared__ float sc[2][G][kChunk];  // score halves, then (row 0) the weights p
    __shared__ float stat[G][2];
    __shared__ float accw[kThreads / 32][G][D];
    const int hk = blockIdx.x, chunk = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int t0 = chunk * kChunk;
    const int nt = min(kChunk, a.T - t0);

    // this thread's K blocks (scores: two threads per token, half of the head's
    // blocks each), loaded first so that their latency overlaps the staging below
    const int stt = tid % kChunk, shalf = tid / kChunk;
    uint4 kw[HALF][2];
    float kf[HALF];
#pragma unroll
    for (int jj = 0; jj < HALF; ++jj) {
        kw[jj][0] = kw[jj][1] = make_uint4(0, 0, 0, 0);
        kf[jj] = 0.0f;
        if (stt < nt) {
            const int kb = hk * NBH + shalf * HALF + jj;
            const uint8_t *krow = a.kc + (int64_t)(t0 + stt) * a.k_row;
            const uint4 *src = reinterpret_cast<const uint4 *>(krow + a.k_off[kb]);
            kw[jj][0] = __ldg(src);
            if (a.k_b[kb] != 4) kw[jj][1] = __ldg(src + 1);
            kf[jj] = block_factor(a.ks[(int64_t)(t0 + stt) * a.nb + a.k_slot[kb]], a.k_b[kb]);
        }
    }
    for (int i = tid; i < G * D; i += kThreads) {
        const int g = i / D, d = i - g * D;
        qs[g][d] = __uint_as_float((uint32_t)a.q[(int64_t)(hk * G + g) * D + d] << 16);
    }
    // the chunk's V blocks of this head into shared memory, with their factors
    for (int i = tid; i < nt * NBH; i += kThreads) {
        const int tt = i / NBH, j = i - tt * NBH;
        const int kb = hk * NBH + j;
        const int b = a.v_b[kb];
        const int64_t t = t0 + tt;
        const uint4 *src = reinterpret_cast<const uint4 *>(a.vc + t * a.v_row + a.v_off[kb]);
        uint4 *dst = reinterpret_cast<uint4 *>(&vcode[tt][j][0]);
        dst[0] = __ldg(src);
        if (b != 4) dst[1] = __ldg(src + 1);
        vfac[tt][j] = block_factor(a.vs[t * a.nb + a.v_slot[kb]], b);
    }
    __syncthreads();

    // scores: two threads per token, each over half of the head's blocks
    {
        const int tt = stt, half = shalf;
        float s[G];
#pragma unroll
        for (int g = 0; g < G; ++g) s[g] = 0.0f;
        if (tt < nt) {
#pragma unroll
            for (int jj = 0; jj < HALF; ++jj) {
                const int j = half * HALF + jj;
                const int b = a.k_b[hk * NBH + j];
                const uint32_t w[8] = {kw[jj][0].x, kw[jj][0].y, kw[jj][0].z, kw[jj][0].w,
                                       kw[jj][1].x, kw[jj][1].y, kw[jj][1].z, kw[jj][1].w};
                const float f = kf[jj];
                float dot[G];
#pragma unroll
                for (int g = 0; g < G; ++g) dot[g] = 0.0f;
#pragma unroll
                for (int i4 = 0; i4 < 8; ++i4) {
                    float c[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) c[e] = (float)code_of(w, b, 4 * i4 + e);
#pragma unroll
                    for (int g = 0; g < G; ++g) {
                        const float4 qv = *reinterpret_cast<const float4 *>(&qs[g][32 * j + 4 * i4]);
                        dot[g] = fmaf(qv.x, c[0], fmaf(qv.y, c[1], fmaf(qv.z, c[2], fmaf(qv.w, c[3], dot[g]))));
                    }
                }
#pragma unroll
                for (int g = 0; g < G; ++g) s[g] = fmaf(dot[g], f, s[g]);
            }
        }
#pragma unroll
        for (int g = 0; g < G; ++g) sc[half][g][tt] = s[g];
    }
    __syncthreads();
    // softmax statistics of the chunk: warp w takes heads w, w + 4, ...
    for (int g = warp; g < G; g += kThreads / 32) {
        float v[kChunk / 32];
        float m = -INFINITY;
#pragma unroll
        for (int r = 0; r < kChunk / 32; ++r) {
            const int tt = lane + 32 * r;
            v[r] = tt < nt ? (sc[0][g][tt] + sc[1][g][tt]) * a.scale : -INFINITY;
            m = fmaxf(m, v[r]);
        }
        for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        float sum = 0.0f;
#pragma unroll
        for (int r = 0; r < kChunk / 32; ++r) {
            const int tt = lane + 32 * r;
            const float e = tt < nt ? expf(v[r] - m) : 0.0f;
            sc[0][g][tt] = e;
            sum += e;
        }
        for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) stat[g][0] = m, stat[g][1] = sum;
    }
    __syncthreads();
    // weighted sums: lane l owns dimensions DL*l.., warp w the tokens w, w + 4, ...
    {
        const int d0 = DL * lane, j = d0 >> 5, i0 = d0 & 31;
        const int b = a.v_b[hk * NBH + j];
        float acc[G][DL];
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < DL; ++e) acc[g][e] = 0.0f;
        for (int tt = warp; tt < nt; tt += kThreads / 32) {
            const uint8_t *cb = &vcode[tt][j][0];
            const float f = vfac[tt][j];
            float v[DL];
#pragma unroll
            for (int e = 0; e < DL; ++e) v[e] = (float)code_at(cb, b, i0 + e) * f;
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const float pg = sc[0][g][tt];
#pragma unroll
                for (int e = 0; e < DL; ++e) acc[g][e] = fmaf(pg, v[e], acc[g][e]);
            }
        }
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < DL; ++e) accw[warp][g][d0 + e] = acc[g][e];
    }
    __syncthreads();
    for (int i = tid; i < G * D; i += kThreads) {
        const int g = i / D, d = i - g * D;
        float t = 0.0f;
#pragma unroll
        for (int w = 0; w < kThreads / 32; ++w) t += accw[w][g][d];  // warp order
        a.part[((int64_t)chunk * a.H + hk * G + g) * (D + 2) + d] = t;
    }
    if (tid < G) {
        float *st = a.part + ((int64_t)chunk * a.H + hk * G + tid) * (D + 2) + D;
        st[0] = stat[tid][0];
        st[1] = stat[tid][1];
    }
}

// out[h][d] = sum_c w_c acc_c[d] / sum_c w_c l_c with w_c = exp(m_c - max_c m_c), chunks in order.
// The chunk statistics go to shared memory first, so the sums over chunks read
// independent addresses (no chain of dependent loads).
constexpr int kCombineChunks = 1024;  // chunks a combine CTA stages at once
template <int D>
__global__ void __launch_bounds__(D) attention_combine_kernel(const float *part, int chunks, int H, float *out) {
    __shared__ float wgt[kCombineChunks];
    __shared__ float red[D];
    const int h = blockIdx.x, d = threadIdx.x;
    float M = -INFINITY;
    for (int c = d; c < chunks; c += D) M = fmaxf(M, part[((int64_t)c * H + h) * (D + 2) + D]);
    red[d] = M;
    __syncthreads();
    for (int o = D / 2; o; o >>= 1) {
        if (d < o) red[d] = fmaxf(red[d], red[d + o]);
        __syncthreads();
    }
    M = red[0];
    float num = 0.0f, den = 0.0f;
    for (int c0 = 0; c0 < chunks; c0 += kCombineChunks) {
        const int n = min(kCombineChunks, chunks - c0);
        __syncthreads();
        for (int c = d; c < n; c += D) wgt[c] = expf(part[((int64_t)(c0 + c) * H + h) * (D + 2) + D] - M);
        __syncthreads();
        const float *pc = part + ((int64_t)c0 * H + h) * (D + 2);
        const int64_t stride = (int64_t)H * (D + 2);
#pragma unroll 16
        for (int c = 0; c < n; ++c) {  // in order; the loads of 16 chunks are independent
            const float w = wgt[c];
            num = fmaf(w, pc[c * stride + d], num);
            den = fmaf(w, pc[c * stride + D + 1], den);
        }
    }
    out[(int64_t)h * D + d] = num / den;
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
    using Kernel = void (*)(AttnArgs);
    static const Kernel kernels[2][4] = {
        {attention_chunk_kernel<64, 1>, attention_chunk_kernel<64, 2>, attention_chunk_kernel<64, 4>,
         attention_chunk_kernel<64, 8>},
        {attention_chunk_kernel<128, 1>, attention_chunk_kernel<128, 2>, attention_chunk_kernel<128, 4>,
         attention_chunk_kernel<128, 8>}};
    const int gi = a.G == 1 ? 0 : (a.G == 2 ? 1 : (a.G == 4 ? 2 : (a.G == 8 ? 3 : -1)));
    if (gi < 0) return fail(MXS_ERR_UNSUPPORTED, "H / H_kv = %d (1, 2, 4 or 8)", a.G);
    kernels[D == 128][gi]<<<grid, kThreads, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "attention_chunk_kernel launch");
    if (D == 128)
        attention_combine_kernel<128><<<(unsigned)H, 128, 0, st>>>(static_cast<const float *>(workspace), (int)chunks,
                                                                   (int)H, out);
    else
        attention_combine_kernel<64><<<(unsigned)H, 64, 0, st>>>(static_cast<const float *>(workspace), (int)chunks,
                                                                 (int)H, out);
    return cuda_fail(cudaGetLastError(), "attention_combine_kernel launch");
}

}  // extern "C"
