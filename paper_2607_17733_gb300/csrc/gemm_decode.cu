// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens), and
// its fusion with A1 (activation quantization in the GEMM prologue).
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale) with the per-block widths of Sec. 4.1.
//
// Decode streams every weight byte once, so the kernel is built around that
// stream:
//   * persistent CTAs, one per SM; warp 0 is a producer that copies, per
//     16-row weight tile and 16-slot K chunk, the contiguous packed codes and
//     scale bytes into a ring of shared-memory stages with cp.async.bulk
//     (completion on mbarriers, every wait bounded);
//   * the other 8 warps split each stage's slots; a weight block arrives in
//     warp-MMA fragment order, so one 8-byte (4-bit) or 16-byte (6/8-bit)
//     shared-memory load per lane is its A operand;
//   * the integer products run on the FP8 warp MMA (e4m3 x e4m3 -> fp32): an
//     e4m3 byte with exponent field <= 1 is exactly k * 2^-9 for its low four
//     bits k, so a sign-magnitude code |m| <= 15 becomes an FP8 operand with
//     two bit operations; 6/8-bit codes are split |m| = 16h + l into two such
//     digits (Sec. 6: high- and low-precision parts multiplied separately), four
//     MMAs combined exactly as 256 hh + 16 (hl + lh) + ll;
//   * each block product is exact in fp32 and is folded as
//     acc += dot * 2^(Ew' + Ea' + 18) (powers of two from the scale bytes);
//   * the token operands (<= 16 rows) are built once per CTA in shared memory,
//     either from the packed activation codes or, in the fused entry point,
//     by quantizing the bf16 activations in the prologue (same integer
//     rounding as the standalone quantizer);
//   * when the token operands of the whole K range do not fit in one SM's
//     shared memory, or N is too small to occupy the GPU, K is split over the
//     CTAs of a thread-block cluster: the other ranks hand their partial tile
//     to rank 0 through distributed shared memory (mbarrier-signalled, double
//     buffered) and rank 0 adds them in rank order.
#include <algorithm>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {

__device__ int g_decode_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

constexpr int kConsumers = 8;
constexpr int kThreads = 32 * (kConsumers + 1);
constexpr int kCH = 64;  // slots per stage: one bulk copy of 17-34 KB (copies cost per count, not per byte)
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock

struct DecodeArgs {
    const uint8_t *codes;   // [M, row_bytes] packed activation codes (or NULL when x is given)
    const uint8_t *scales;  // [M, nb]
    const uint16_t *x;      // bf16 [M, ld_x] activations for the fused entry point (or NULL)
    int64_t ld_x;
    int rhaz;
    const uint8_t *w;  // packed weight buffer
    float *y;
    int64_t ld_y;
    int M, N, T;
    int GS, chunk;        // CTAs per cluster along K, slots per CTA
    int stages, stage_bytes;
    int b_bytes;  // shared-memory bytes of the token operands (largest rank)
    int64_t TB;  // bytes of one 16-row weight tile
};

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_remote(uint64_t *bar, uint32_t rank) {
    asm volatile(
        "{\n .reg .b32 ra;\n mapa.shared::cluster.u32 ra, %0, %1;\n"
        " mbarrier.arrive.release.cluster.shared::cluster.b64 _, [ra];\n}" ::"r"(su32(bar)),
        "r"(rank)
        : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// waits on barriers that threads of other CTAs of the cluster arrive on
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
template <bool kCluster = false>
__device__ __forceinline__ bool poll(uint64_t *bar, uint32_t parity) {
    return kCluster ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity);
}
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (poll<kCluster>(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (poll<kCluster>(bar, parity)) return true;
        if ((i & 63) == 0) {  // the bound is checked every 64 polls: reading a clock is not free
            if (*abort) return false;
            if (clock64() - t0 > kWaitCycles) {
                *abort = 1;
                atomicExch(&g_decode_status, MXS_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
// Whole-warp wait: one lane polls (256 threads spinning on one barrier word
// would compete with the shared-memory traffic they are waiting for), then
// every lane takes its own, immediately successful, acquiring test.
template <bool kCluster = false>
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    const int lane = threadIdx.x & 31;
    bool ok = true;
    if (lane == 0) ok = mbar_wait<kCluster>(bar, parity, abort);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok) poll<kCluster>(bar, parity);
    return ok;
}

__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     su32(dst)),
                 "l"(src), "r"(bytes), "r"(su32(bar))
                 : "memory");
}
__device__ __forceinline__ void st_remote_f32(const float *local_addr, uint32_t rank, float v) {
    asm volatile(
        "{\n .reg .b32 ra;\n mapa.shared::cluster.u32 ra, %0, %1;\n st.shared::cluster.f32 [ra], %2;\n}" ::"r"(
            su32(local_addr)),
        "r"(rank), "f"(v)
        : "memory");
}
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(32 * kConsumers) : "memory"); }
// consumer-warp barrier that also ORs a flag over all consumer threads, so a
// stop decision is taken by every consumer warp at the same point
__device__ __forceinline__ bool consumer_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.or.pred p, 1, %2, q;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(r)
        : "r"((uint32_t)v), "n"(32 * kConsumers)
        : "memory");
    return r != 0;
}

__device__ __forceinline__ void mma_e4m3(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1,
                                         const float (&c)[4]) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%10,%11,%12,%13};"
        : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(c[0]), "f"(c[1]), "f"(c[2]),
          "f"(c[3]));
}

// e4m3 bytes of m * 2^-9 for four sign-magnitude 4-bit codes in the high /
// low nibbles of the bytes of x
__device__ __forceinline__ uint32_t e4m3_hi_nib(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t e4m3_lo_nib(uint32_t x) { return (x & 0x07070707u) | ((x << 4) & 0x80808080u); }
// high (|m| >> 4) and low (|m| & 15) digit of four sign-magnitude 8-bit codes
__device__ __forceinline__ uint32_t e4m3_hi_dig(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t e4m3_lo_dig(uint32_t x) { return x & 0x8F8F8F8Fu; }

__device__ __forceinline__ uint32_t signmag4(int m) { return (uint32_t)(((m < 0) << 3) | (m < 0 ? -m : m)); }
__device__ __forceinline__ uint32_t signmag8(int m) { return (uint32_t)(((m < 0) << 7) | (m < 0 ? -m : m)); }

// Token operands in shared memory (B of the warp MMA, 16 tokens = 2 n-tiles):
//   4-bit slot c, n-tile nt, lane l = 4g+q: one u32, byte j: high nibble =
//     element 4q+j, low nibble = element 16+4q+j of token 8nt+g (sign-magnitude);
//   6/8-bit slot: one uint2, x = elements 4q..4q+3, y = 16+4q..16+4q+3 (sign-magnitude bytes);
//   fa[c][token] = 2^(Ea' + 18) (the two operands carry m * 2^-9 each), 0 for padding tokens.
template <int NT>
__device__ void write_token_block(uint32_t *B4, uint2 *B8, float *fa, int c, int c4, int c8, bool four, int tok,
                                  const int (&m)[32], int S, int b, bool real) {
    const int nt = tok >> 3, g = tok & 7;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int l = 4 * g + q;
        if (four) {
            uint32_t w = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) w |= ((signmag4(m[4 * q + j]) << 4) | signmag4(m[16 + 4 * q + j])) << (8 * j);
            B4[(c4 * NT + nt) * 32 + l] = w;
        } else {
            uint32_t lo = 0, hi = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                lo |= signmag8(m[4 * q + j]) << (8 * j);
                hi |= signmag8(m[16 + 4 * q + j]) << (8 * j);
            }
            B8[(c8 * NT + nt) * 32 + l] = make_uint2(lo, hi);
        }
    }
    fa[c * 16 + tok] = !real ? 0.f : (S == 255 ? __int_as_float(0x7fc00000) : pow2f(S - 127 - (b - 2) + 18));
}

template <int NT>
__global__ void __launch_bounds__(kThreads, 1) gemm_decode_kernel(const __grid_constant__ Plan p,
                                                                  const __grid_constant__ DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *ring = smem;                                                    // stages x stage_bytes
    uint32_t *B4 = reinterpret_cast<uint32_t *>(ring + (size_t)a.stages * a.stage_bytes);
    float *fa = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(B4) + a.b_bytes);  // [chunk][16]
    float *red = fa + (size_t)a.chunk * 16;                       // [2][kConsumers][NT*128]
    float *xbuf = red + 2 * kConsumers * NT * 128;                // [GS-1][2][NT*128] (rank 0)
    uint64_t *bars = reinterpret_cast<uint64_t *>(xbuf + (size_t)(a.GS - 1) * 2 * NT * 128);
    uint64_t *full = bars, *empty = bars + a.stages, *xfull = bars + 2 * a.stages, *xempty = xfull + 2;
    int *abort_flag = reinterpret_cast<int *>(xempty + 2);
    volatile int *abort = abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = a.GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = (int)rank * a.chunk, c1 = min(p.nb, c0 + a.chunk);
    const int nchunks = (c1 - c0 + kCH - 1) / kCH;
    const int n4lo = min(c0, p.n4), n4hi = min(c1, p.n4);  // 4-bit slots of this CTA: [n4lo, n4hi)
    const int s8lo = max(c0, p.n4);                        // 6/8-bit slots: [s8lo, c1)
    uint2 *B8 = reinterpret_cast<uint2 *>(B4 + (size_t)max(0, n4hi - n4lo) * NT * 32);
    constexpr int kOut = NT * 128;

    if (threadIdx.x == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumers);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&xfull[i], (uint32_t)(a.GS - 1) * kOut);
            mbar_init(&xempty[i], kOut);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (a.GS > 1) cg::this_cluster().sync();  // partners' barriers exist before any remote access

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0) {
            uint32_t qn = 0;
            bool stop = false;
            for (int t = blockIdx.x; t < a.T && !stop; t += gridDim.x) {
                for (int j = 0; j < nchunks; ++j, ++qn) {
                    const int s = (int)(qn % a.stages);
                    if (!mbar_wait(&empty[s], ((qn / a.stages) & 1) ^ 1, abort)) { stop = true; break; }
                    const int lo = c0 + j * kCH, hi = min(c1, lo + kCH);
                    const int64_t off = slot_offset(p, lo);
                    const uint32_t bytes = (uint32_t)(slot_offset(p, hi) - off);  // slots [lo, hi) of tile t: contiguous
                    mbar_expect_tx(&full[s], bytes);
                    bulk_load(ring + (size_t)s * a.stage_bytes, a.w + (int64_t)t * a.TB + off, bytes, &full[s]);
                }
            }
            // drain: every copy issued must land before the CTA leaves
            const uint32_t first = qn > (uint32_t)a.stages ? qn - a.stages : 0;
            for (uint32_t k = first; k < qn; ++k) {
                const long long t0 = clock64();
                while (!mbar_try_wait(&full[k % a.stages], (k / a.stages) & 1) && clock64() - t0 < kWaitCycles) {
                }
            }
        }
    } else {
        // ---------------------------------------------------------- consumers
        const int cw = warp - 1, ctid = threadIdx.x - 32;
        const int g = lane >> 2, q = lane & 3;

        // token operands of this CTA's slots [c0, c1), for 8*NT token rows
        for (int it = ctid; it < (c1 - c0) * 8 * NT; it += 32 * kConsumers) {
            const int c = it / (8 * NT), tok = it - c * (8 * NT);
            const int s = c0 + c;
            const bool four = s < p.n4;
            const int b = slot_width(p, s);
            int m[32];
            int S = 0;
            const bool real = tok < a.M;
            if (!real) {
#pragma unroll
                for (int i = 0; i < 32; ++i) m[i] = 0;
            } else if (a.x) {  // fused: quantize the bf16 block here
                const uint4 *src = reinterpret_cast<const uint4 *>(a.x + (int64_t)tok * a.ld_x + kBlock * p.slot_block[s]);
                uint32_t h[32];
                uint32_t mag = 0;
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
#pragma unroll
                for (int i = 0; i < 32; ++i) mag = max(mag, h[i] & 0x7FFF);
                S = (int)(mag >> 7);
#pragma unroll
                for (int i = 0; i < 32; ++i) m[i] = S == 255 ? 0 : quant_elem(h[i], S, b, a.rhaz);
            } else {  // from the packed activation codes
                const uint8_t *row = a.codes + (int64_t)tok * p.row_bytes;
                S = a.scales[(int64_t)tok * p.nb + s];
                if (four) {
                    const uint4 v = *reinterpret_cast<const uint4 *>(row + 16 * (int64_t)s);
                    const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int nib = (w4[i >> 3] >> (4 * (i & 7))) & 0xF;
                        m[i] = nib >= 8 ? nib - 16 : nib;
                    }
                } else {
                    const uint4 *v = reinterpret_cast<const uint4 *>(row + 16 * (int64_t)p.n4 + 32 * (int64_t)(s - p.n4));
                    const uint4 v0 = v[0], v1 = v[1];
                    const uint32_t w8[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
                    for (int i = 0; i < 32; ++i) m[i] = (int)(int8_t)(w8[i >> 2] >> (8 * (i & 3)));
                }
            }
            write_token_block<NT>(B4, B8, fa, c, s - n4lo, s - s8lo, four, tok, m, S, b, real);
        }
        consumer_sync();

        const float zero[4] = {0.f, 0.f, 0.f, 0.f};
        uint32_t qn = 0;
        int iter = 0;
        bool stop = false;
        for (int t = blockIdx.x; t < a.T; t += gridDim.x, ++iter) {
            float acc[NT][4];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;

            for (int j = 0; j < nchunks && !stop; ++j, ++qn) {
                const int s = (int)(qn % a.stages);
                if (!warp_wait(&full[s], (qn / a.stages) & 1, abort)) { stop = true; break; }
                const int lo = c0 + j * kCH, hi = min(c1, lo + kCH);
                const uint8_t *st = ring + (size_t)s * a.stage_bytes - slot_offset(p, lo);  // + slot_offset(sl)
                const int per = (hi - lo + kConsumers - 1) / kConsumers;
                const int my0 = lo + cw * per, my1 = min(hi, my0 + per);
                for (int sl = my0; sl < my1; ++sl) {
                    const int b = slot_width(p, sl);
                    const uint8_t *blk = st + slot_offset(p, sl);
                    const uint8_t *scb = blk + (b == 4 ? 256 : 512);
                    const int S0 = scb[g], S1 = scb[g + 8];
                    const float f0 = S0 == 255 ? __int_as_float(0x7fc00000) : pow2f(S0 - 127 - (b - 2));
                    const float f1 = S1 == 255 ? __int_as_float(0x7fc00000) : pow2f(S1 - 127 - (b - 2));
                    const float *fs = fa + (sl - c0) * 16 + 2 * q;
                    if (sl < p.n4) {
                        const uint2 wv = *reinterpret_cast<const uint2 *>(blk + 8 * lane);
                        const uint32_t af[4] = {e4m3_hi_nib(wv.x), e4m3_hi_nib(wv.y), e4m3_lo_nib(wv.x),
                                                e4m3_lo_nib(wv.y)};
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt) {
                            const uint32_t bx = B4[((sl - n4lo) * NT + nt) * 32 + lane];
                            float d[4];
                            mma_e4m3(d, af, e4m3_hi_nib(bx), e4m3_lo_nib(bx), zero);
                            const float2 ft = *reinterpret_cast<const float2 *>(fs + 8 * nt);
                            acc[nt][0] = fmaf(d[0], f0 * ft.x, acc[nt][0]);
                            acc[nt][1] = fmaf(d[1], f0 * ft.y, acc[nt][1]);
                            acc[nt][2] = fmaf(d[2], f1 * ft.x, acc[nt][2]);
                            acc[nt][3] = fmaf(d[3], f1 * ft.y, acc[nt][3]);
                        }
                    } else {
                        const uint4 wv = *reinterpret_cast<const uint4 *>(blk + 16 * lane);
                        const uint32_t ah[4] = {e4m3_hi_dig(wv.x), e4m3_hi_dig(wv.y), e4m3_hi_dig(wv.z),
                                                e4m3_hi_dig(wv.w)};
                        const uint32_t al[4] = {e4m3_lo_dig(wv.x), e4m3_lo_dig(wv.y), e4m3_lo_dig(wv.z),
                                                e4m3_lo_dig(wv.w)};
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt) {
                            const uint2 bx = B8[((sl - s8lo) * NT + nt) * 32 + lane];
                            const uint32_t bh0 = e4m3_hi_dig(bx.x), bh1 = e4m3_hi_dig(bx.y);
                            const uint32_t bl0 = e4m3_lo_dig(bx.x), bl1 = e4m3_lo_dig(bx.y);
                            float hh[4], xx[4], ll[4];
                            mma_e4m3(hh, ah, bh0, bh1, zero);
                            mma_e4m3(xx, ah, bl0, bl1, zero);
                            mma_e4m3(xx, al, bh0, bh1, xx);
                            mma_e4m3(ll, al, bl0, bl1, zero);
                            const float2 ft = *reinterpret_cast<const float2 *>(fs + 8 * nt);
                            float d[4];
#pragma unroll
                            for (int i = 0; i < 4; ++i) d[i] = fmaf(256.f, hh[i], fmaf(16.f, xx[i], ll[i]));  // exact
                            acc[nt][0] = fmaf(d[0], f0 * ft.x, acc[nt][0]);
                            acc[nt][1] = fmaf(d[1], f0 * ft.y, acc[nt][1]);
                            acc[nt][2] = fmaf(d[2], f1 * ft.x, acc[nt][2]);
                            acc[nt][3] = fmaf(d[3], f1 * ft.y, acc[nt][3]);
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);
            }

            // ---- this tile: sum the 8 warps (fixed order), then the cluster's ranks.
            // Every consumer warp reaches this barrier; a stop anywhere stops all.
            const int buf = iter & 1;
            float *rb = red + buf * kConsumers * kOut;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) rb[cw * kOut + (nt * 4 + i) * 32 + lane] = acc[nt][i];
            if (consumer_sync_or(stop || *abort)) break;
            if (ctid < kOut) {
                const int o = ctid;
                float v = 0.f;
#pragma unroll
                for (int k = 0; k < kConsumers; ++k) v += rb[k * kOut + o];
                if (a.GS > 1 && rank > 0) {
                    if (!mbar_wait<true>(&xempty[buf], ((iter >> 1) & 1) ^ 1, abort)) { stop = true; }
                    else {
                        st_remote_f32(xbuf + ((rank - 1) * 2 + buf) * kOut + o, 0, v);
                        mbar_arrive_remote(&xfull[buf], 0);
                    }
                } else {
                    if (a.GS > 1) {
                        if (!mbar_wait<true>(&xfull[buf], (iter >> 1) & 1, abort)) { stop = true; }
                        else {
                            for (int r = 1; r < a.GS; ++r) v += xbuf[((r - 1) * 2 + buf) * kOut + o];
                            for (int r = 1; r < a.GS; ++r) mbar_arrive_remote(&xempty[buf], (uint32_t)r);
                        }
                    }
                    const int nt = o / 128, rem = o - nt * 128;
                    const int i = rem >> 5, ln = rem & 31;
                    const int tok = 8 * nt + 2 * (ln & 3) + (i & 1);
                    const int n = 16 * t + (ln >> 2) + 8 * (i >> 1);
                    if (!stop && tok < a.M && n < a.N) a.y[(int64_t)tok * a.ld_y + n] = v;
                }
            }
        }
    }
    __syncthreads();
    if (a.GS > 1) cg::this_cluster().sync();  // no CTA leaves while a partner may still touch its memory
}

struct DecodeShape {
    int GS, chunk, stages, stage_bytes, b_bytes, grid;
    size_t smem;
};

DecodeShape shape_for(const Plan &p, int NT, int GS, int64_t T, int sms) {
    DecodeShape sh;
    sh.GS = GS;
    sh.chunk = (p.nb + GS - 1) / GS;
    int max_b = 0, max_stage = 0;
    for (int r = 0; r < GS; ++r) {
        const int c0 = r * sh.chunk, c1 = std::min(p.nb, c0 + sh.chunk);
        const int n4c = std::max(0, std::min(c1, p.n4) - std::min(c0, p.n4));
        const int n8c = std::max(0, c1 - c0) - n4c;
        max_b = std::max(max_b, n4c * NT * 128 + n8c * NT * 256);
        for (int lo = c0; lo < c1; lo += kCH) {
            const int hi = std::min(c1, lo + kCH);
            max_stage = std::max(max_stage, (int)(slot_offset(p, hi) - slot_offset(p, lo)));
        }
    }
    sh.stage_bytes = (max_stage + 127) / 128 * 128;
    sh.b_bytes = (max_b + 127) / 128 * 128;
    const size_t fixed = (size_t)sh.b_bytes + (size_t)sh.chunk * 64 + 2 * kConsumers * NT * 512 +
                         (size_t)(GS - 1) * 2 * NT * 512;
    const size_t budget = 220 * 1024;
    sh.stages = 0;
    if (fixed + 2 * (size_t)sh.stage_bytes + 512 <= budget)
        sh.stages = (int)std::min<size_t>(12, (budget - fixed - 512) / sh.stage_bytes);
    sh.smem = fixed + (size_t)sh.stages * sh.stage_bytes + (2 * sh.stages + 4) * 8 + 16;
    sh.grid = (int)std::min<int64_t>(T, std::max(1, sms / GS));
    return sh;
}

// GS = 1 unless the token operands do not fit next to a useful ring, or N is
// too small to give every SM a row tile.
DecodeShape pick_shape(const Plan &p, int NT, int64_t T, int sms) {
    const int gs_max = std::max(1, std::min(8, p.nb));
    DecodeShape best = shape_for(p, NT, 1, T, sms), most = best;
    bool found = false;
    for (int GS = 1; GS <= gs_max; GS *= 2) {
        const DecodeShape sh = shape_for(p, NT, GS, T, sms);
        if (sh.stages > most.stages) most = sh;
        if (sh.stages < 3) continue;
        best = sh;
        found = true;
        if (T * GS >= sms || 2 * GS > gs_max) break;
    }
    return found ? best : most;
}

int sm_count() {
    static int cached = 0;
    if (!cached) {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) ==
                                                      cudaSuccess && n > 0)
            cached = n;
        else
            return 152;
    }
    return cached;
}

template <int NT>
int launch_nt(const Plan &p, const DecodeArgs &a0, cudaStream_t st) {
    DecodeArgs a = a0;
    const DecodeShape sh = pick_shape(p, NT, a.T, sm_count());
    if (sh.stages < 2) return fail(MXS_ERR_SHAPE, "decode: K=%d too large for the shared-memory plan", 32 * p.nb);
    a.GS = sh.GS;
    a.chunk = sh.chunk;
    a.stages = sh.stages;
    a.stage_bytes = sh.stage_bytes;
    a.b_bytes = sh.b_bytes;
    auto kern = gemm_decode_kernel<NT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
    if (sh.GS > 1) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(cluster)");
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)sh.grid, (unsigned)sh.GS, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = sh.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = (unsigned)sh.GS;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, p, a);
    return cuda_fail(e, "gemm_decode_kernel launch");
}

int launch(const Plan &p, DecodeArgs a, int64_t M, int64_t N, cudaStream_t st) {
    a.M = (int)M;
    a.N = (int)N;
    a.T = (int)((N + 15) / 16);
    const WeightOffsets off = weight_offsets(p, N, false);
    a.TB = off.TB;
    if (N > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
    return M <= 8 ? launch_nt<1>(p, a, st) : launch_nt<2>(p, a, st);
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
    return launch(p, a, M, N, st);
}

int launch_linear_decode(const Plan &p, const void *x, int64_t ld_x, int rounding, const void *packed, int64_t M,
                         int64_t N, float *y, int64_t ld_y, cudaStream_t st) {
    DecodeArgs a = {};
    a.x = static_cast<const uint16_t *>(x);
    a.ld_x = ld_x;
    a.rhaz = rounding == MXS_RHAZ;
    a.w = static_cast<const uint8_t *>(packed);
    a.y = y;
    a.ld_y = ld_y;
    return launch(p, a, M, N, st);
}

int decode_status(int *status, int reset) {
    int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_decode_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyFromSymbol(decode status)");
    *status = v;
    if (reset && v != 0) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_decode_status, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyToSymbol(decode status)");
    }
    return MXS_OK;
}

}  // namespace mxs
