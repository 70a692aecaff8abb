// gemv_decode.cu -- A1 + A4 for decode shapes of one to four tokens: the
// activations are quantized inside the GEMM's prologue and the integer block
// dot products run on the CUDA cores.
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * D, D the exact
// integer dot of the two blocks' mantissas: the MXINT product of Sec. 2 with
// the per-block widths of Sec. 4.1, the activations quantized on the fly
// (Appendix A.2).
//
// Why a second decode kernel.  On GB300 a block-scaled tensor-core MMA costs
// a fixed number of cycles per instruction whatever its N up to 128
// (mxs_probe_mma), so the tensor-core decode GEMM spends the same time on one
// token as on sixteen.  With one token the dot products are cheap enough for
// the CUDA cores: per weight word, a few integer operations turn four
// sign-magnitude codes into two's-complement bytes and one dp4a per token
// adds four products exactly.  The work per token grows with M while the
// tensor-core path's does not: over twelve LLaMA-2-70B layers this kernel
// takes 1.91 ms at M = 1 against 2.41 ms, but 3.6 ms at M = 4 against 2.43 ms,
// so the library sends it M <= kGemvMaxM (1) tokens.
//
// Work.  A CTA owns 128-row weight groups (and, in a thread-block cluster, a
// K range of them).  Prologue: it quantizes the activations of its K range
// (x is bf16; the rule, bit for bit, of mxs_quantize_act) into shared memory
// as int8 codes and scale bytes, in slot order.  Main loop: thread t of four
// sets of 128 is weight row t % 128 of the group, and set t / 128 takes every
// fourth slot of the range; per slot it loads its row's codes (16 or 32
// bytes, coalesced across the set) and scale byte, forms the integer dots with
// dp4a and adds 2^(Ea'+Ew') * D into an fp32 accumulator per token (the
// product is exact: |D| < 2^20 times a power of two).  The sets' sums are
// added in set order; cluster ranks write theirs into rank 0's shared memory
// (distributed shared-memory stores, then a cluster barrier) and rank 0 adds
// them in rank order: deterministic.  Lanes of warp 0 stream the group's
// weight bytes into L2 ahead of the loads (bulk L2 prefetches, issued in
// turn), so the loads are L2 hits.
#include <algorithm>
#include <cstring>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {
namespace {

constexpr int kGThreads = 512;
constexpr int kGSets = 4;                  // thread sets; a set is 128 threads, one per weight row
constexpr int kGMaxProblems = 3;
#ifndef MXS_GEMV_AHEAD_KB
#define MXS_GEMV_AHEAD_KB 192
#endif
#ifndef MXS_GEMV_UNROLL
#define MXS_GEMV_UNROLL 8
#endif
constexpr int kPrefetchAhead = MXS_GEMV_AHEAD_KB * 1024;  // bytes of the weight stream kept in flight to L2
constexpr int kUnroll4 = MXS_GEMV_UNROLL;  // 4-bit slots a thread loads before it computes
#ifndef MXS_GEMV_PF_KB
#define MXS_GEMV_PF_KB 64
#endif
#ifndef MXS_GEMV_PF_LANES
#define MXS_GEMV_PF_LANES 1
#endif
constexpr int kPrefetchChunk = MXS_GEMV_PF_KB * 1024;  // bytes per bulk L2 prefetch
constexpr int kPfLanes = MXS_GEMV_PF_LANES;            // lanes of warp 0 that issue them, in turn

struct GemvProblem {
    const uint16_t *x;  // bf16 [M, K], row stride ld_x
    const uint8_t *w;   // packed weights (compact part)
    float *y;
    int64_t ld_x, ld_y, GB;
    int N, G, GS, nb, n4, n6;
    int bound[9];       // cluster rank r owns slots [bound[r], bound[r+1])
    int cta0, ncta;
};
struct GemvParams {
    GemvProblem prob[kGMaxProblems];
    uint16_t slot_block[kGMaxProblems][kMaxNb];  // slot -> block of each problem's plan
    int nprob, M, rhaz;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ uint4 ld_stream(const void *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ uint32_t map_rank(const void *p, uint32_t rank) {
    uint32_t ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(su32(p)), "r"(rank));
    return ra;
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release;\n barrier.cluster.wait.acquire;" ::: "memory");
}
__host__ __device__ __forceinline__ int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ int64_t slot_off_g(int n4, int s) {
    return s < n4 ? 2176 * (int64_t)s : 2176 * (int64_t)n4 + 4224 * (int64_t)(s - n4);
}

// Four sign-magnitude codes (sign at bit `sb` of each byte, magnitude below
// it, never a negative zero) as two's-complement bytes: (m ^ -s) + s per
// byte, which never carries since m >= 1 wherever s = 1.
__device__ __forceinline__ int twos4(uint32_t x, uint32_t mag_mask, int sb) {
    const uint32_t m = x & mag_mask;
    const uint32_t s = (x >> sb) & 0x01010101u;
    return (int)((m ^ (s * 0xFFu)) + s);
}

// acc + D * 2^e (D exact in fp32); NaN when either scale byte is 255
__device__ __forceinline__ float fold(float acc, int D, int Sa, int Sw, int b) {
    if (Sa == 255 || Sw == 255) return __int_as_float(0x7FC00000);
    if (D == 0) return acc;
    const int e = Sa + Sw - 254 - 2 * (b - 2);
    if (e >= -126 && e <= 127) return fmaf((float)D, __int_as_float((e + 127) << 23), acc);
    return acc + ldexpf((float)D, e);  // scales outside the normal range (|x| near 2^-126 or 2^127)
}

template <int MT>
__global__ void __launch_bounds__(kGThreads, 1) gemv_decode_kernel(const __grid_constant__ GemvParams gp) {
    int pi = 0;
    while (pi + 1 < gp.nprob && (int)blockIdx.x >= gp.prob[pi + 1].cta0) ++pi;
    const GemvProblem &P = gp.prob[pi];
    const uint16_t *sblk = gp.slot_block[pi];
    const int bx = (int)blockIdx.x - P.cta0, gx = P.ncta;
    const uint32_t rank = P.GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = P.bound[rank], c1 = P.bound[rank + 1], ns = c1 - c0;
    const int M = gp.M, tid = threadIdx.x, set = tid >> 7, r = tid & 127;
    const int e4 = max(c0, min(c1, P.n4));  // 4-bit slots [c0, e4), 6/8-bit slots [e4, c1)

    // shared memory: the cluster exchange first, so that its offset is the same
    // in every rank (the ranks' K ranges, and so their token buffers, differ)
    extern __shared__ __align__(16) uint8_t smem[];
    float *xbuf = reinterpret_cast<float *>(smem);                      // [2][GS][MT][128] (read in rank 0)
    float *part = xbuf + 2 * P.GS * MT * 128;                           // [sets][MT][128]
    int8_t *tcode = reinterpret_cast<int8_t *>(part + kGSets * MT * 128);  // [ns][MT][32] token codes
    uint8_t *tsc = reinterpret_cast<uint8_t *>(tcode) + (size_t)ns * MT * 32;  // [ns][MT] token scale bytes

    if (tid == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int ngroups = bx < P.G ? (P.G - 1 - bx) / gx + 1 : 0;
    // the weights are static: start their stream into L2 before the wait.
    // Thread 0 keeps the prefetch kPrefetchAhead bytes ahead of set 0 and, once
    // a group's range is covered, sends out the head of the next group.
    const int64_t r0 = slot_off_g(P.n4, c0), rbytes = slot_off_g(P.n4, c1) - r0;
    const int64_t head = imin64(rbytes, kPrefetchAhead);
    int64_t pf = 0;     // bytes of the current group's range prefetched
    bool next_out = false;  // the next group's head has been prefetched
    // the prefetch state is kept alike in lanes 0 .. kPfLanes-1; chunk i of a
    // range is issued by lane i % kPfLanes
    auto prefetch_range = [&](const uint8_t *base, int64_t from, int64_t to) {
        for (int64_t q = from + (int64_t)tid * kPrefetchChunk; q < to; q += (int64_t)kPfLanes * kPrefetchChunk)
            prefetch_l2(base + q, (uint32_t)imin64(kPrefetchChunk, to - q));
    };
    if (tid < kPfLanes && ngroups > 0) {
        prefetch_range(P.w + (int64_t)bx * P.GB + r0, 0, head);
        pf = head;
    }
    // x may come from the kernel before this one (programmatic dependent launch)
    asm volatile("griddepcontrol.wait;" ::: "memory");

    // ---- prologue: the activations of slots [c0, c1) as int8 codes (mxs_quantize_act's rule)
    for (int i = tid; i < ns * MT; i += kGThreads) {
        const int j = i / MT, t = i - j * MT, s = c0 + j;
        uint4 *dst = reinterpret_cast<uint4 *>(tcode + ((size_t)j * MT + t) * 32);
        if (t >= M) {
            dst[0] = dst[1] = make_uint4(0, 0, 0, 0);
            tsc[j * MT + t] = 0;
            continue;
        }
        const int b = s < P.n4 ? 4 : (s < P.n4 + P.n6 ? 6 : 8);
        const uint4 *src = reinterpret_cast<const uint4 *>(P.x + (int64_t)t * P.ld_x + 32 * (int64_t)sblk[s]);
        uint32_t h[32];
        uint32_t mag = 0;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint4 u = __ldg(src + v);
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                h[8 * v + 2 * k] = w4[k] & 0xFFFF;
                h[8 * v + 2 * k + 1] = w4[k] >> 16;
            }
        }
#pragma unroll
        for (int k = 0; k < 32; ++k) mag = max(mag, h[k] & 0x7FFF);
        const int S = (int)(mag >> 7);
        uint32_t cw[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            cw[k] = 0;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int m = S == 255 ? 0 : quant_elem(h[4 * k + q], S, b, gp.rhaz);
                cw[k] |= (uint32_t)(m & 0xFF) << (8 * q);
            }
        }
        dst[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
        dst[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
        tsc[j * MT + t] = (uint8_t)S;
    }
    __syncthreads();
    if (P.GS > 1) cluster_sync_all();  // every rank runs before the first store into rank 0

    for (int gi = 0; gi < ngroups; ++gi) {
        const int g = bx + gi * gx;
        const uint8_t *wg = P.w + (int64_t)g * P.GB;
        const uint8_t *rng = wg + r0;
        float acc[MT];
#pragma unroll
        for (int t = 0; t < MT; ++t) acc[t] = 0.0f;
        if (tid < kPfLanes && gi > 0) {  // the head of this group went out with the previous one
            pf = next_out ? head : 0;
            next_out = false;
        }
        auto advance = [&](int64_t done) {
            if (tid >= kPfLanes) return;
            const int64_t to = imin64(rbytes, done + kPrefetchAhead);
            if (pf < to) {
                prefetch_range(rng, pf, to);
                pf = to;
            }
            if (pf >= rbytes && !next_out && gi + 1 < ngroups) {
                prefetch_range(wg + (int64_t)gx * P.GB + r0, 0, head);
                next_out = true;
            }
        };
        // ---- 4-bit slots: 16 code bytes of row r (byte 4i+j: element 8i+j low, 8i+4+j high)
        for (int s0 = c0 + set; s0 < e4; s0 += kUnroll4 * kGSets) {
            uint4 v[kUnroll4];
            int Sw[kUnroll4];
#pragma unroll
            for (int u = 0; u < kUnroll4; ++u) {
                const int s = s0 + u * kGSets;
                if (s < e4) {
                    const uint8_t *sl = wg + slot_off_g(P.n4, s);
                    v[u] = ld_stream(sl + 16 * r);
                    Sw[u] = __ldg(sl + 2048 + r);
                }
            }
            advance(slot_off_g(P.n4, s0) - r0);
#pragma unroll
            for (int u = 0; u < kUnroll4; ++u) {
                const int s = s0 + u * kGSets;
                if (s >= e4) break;
                const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
                int lo[4], hi[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    lo[i] = twos4(wd[i], 0x07070707u, 3);
                    hi[i] = twos4(wd[i] >> 4, 0x07070707u, 3);
                }
                const int j = s - c0;
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    const uint4 *tc = reinterpret_cast<const uint4 *>(tcode + ((size_t)j * MT + t) * 32);
                    const uint4 ta = tc[0], tb = tc[1];
                    const int tw[8] = {(int)ta.x, (int)ta.y, (int)ta.z, (int)ta.w,
                                       (int)tb.x, (int)tb.y, (int)tb.z, (int)tb.w};
                    int D = 0;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        D = __dp4a(lo[i], tw[2 * i], D);
                        D = __dp4a(hi[i], tw[2 * i + 1], D);
                    }
                    acc[t] = fold(acc[t], D, tsc[j * MT + t], Sw[u], 4);
                }
            }
        }
        // ---- 6/8-bit slots: 32 code bytes of row r (byte e = element e)
        for (int s0 = e4 + set; s0 < c1; s0 += 2 * kGSets) {
            uint4 v[2][2];
            int Sw[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int s = s0 + u * kGSets;
                if (s < c1) {
                    const uint8_t *sl = wg + slot_off_g(P.n4, s);
                    v[u][0] = ld_stream(sl + 32 * r);
                    v[u][1] = ld_stream(sl + 32 * r + 16);
                    Sw[u] = __ldg(sl + 4096 + r);
                }
            }
            advance(slot_off_g(P.n4, s0) - r0);
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int s = s0 + u * kGSets;
                if (s >= c1) break;
                const int b = s < P.n4 + P.n6 ? 6 : 8;
                const uint32_t wd[8] = {v[u][0].x, v[u][0].y, v[u][0].z, v[u][0].w,
                                        v[u][1].x, v[u][1].y, v[u][1].z, v[u][1].w};
                int c[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) c[i] = twos4(wd[i], 0x7F7F7F7Fu, 7);
                const int j = s - c0;
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    const uint4 *tc = reinterpret_cast<const uint4 *>(tcode + ((size_t)j * MT + t) * 32);
                    const uint4 ta = tc[0], tb = tc[1];
                    const int tw[8] = {(int)ta.x, (int)ta.y, (int)ta.z, (int)ta.w,
                                       (int)tb.x, (int)tb.y, (int)tb.z, (int)tb.w};
                    int D = 0;
#pragma unroll
                    for (int i = 0; i < 8; ++i) D = __dp4a(c[i], tw[i], D);
                    acc[t] = fold(acc[t], D, tsc[j * MT + t], Sw[u], b);
                }
            }
        }
        advance(rbytes);  // (the prefetch lanes) the rest of this range and the next group's head

        // ---- the sets' sums in set order, then the ranks' in rank order
#pragma unroll
        for (int t = 0; t < MT; ++t) part[(set * MT + t) * 128 + r] = acc[t];
        __syncthreads();
        float val[MT];
        if (set == 0) {
#pragma unroll
            for (int t = 0; t < MT; ++t) {
                float v = part[t * 128 + r];
#pragma unroll
                for (int k = 1; k < kGSets; ++k) v += part[(k * MT + t) * 128 + r];
                val[t] = v;
            }
        }
        const int n = 128 * g + r;
        if (P.GS == 1) {
            if (set == 0 && n < P.N)
#pragma unroll
                for (int t = 0; t < MT; ++t)
                    if (t < M) P.y[(int64_t)t * P.ld_y + n] = val[t];
        } else {
            float *xb = xbuf + (gi & 1) * P.GS * MT * 128;
            if (set == 0)
#pragma unroll
                for (int t = 0; t < MT; ++t) st_cluster_f32(map_rank(xb + (rank * MT + t) * 128 + r, 0), val[t]);
            cluster_sync_all();  // every rank's partial sums are in rank 0
            if (rank == 0 && set == 0 && n < P.N)
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    if (t >= M) continue;
                    float v = xb[t * 128 + r];
                    for (int k = 1; k < P.GS; ++k) v += xb[(k * MT + t) * 128 + r];
                    P.y[(int64_t)t * P.ld_y + n] = v;
                }
        }
        __syncthreads();  // `part` is reused by the next group
    }
}

// ------------------------------------------------------------------ host side
int gemv_stage_lo(const Plan &p, int sg) {
    return sg <= p.st4 ? std::min(4 * sg, p.n4) : std::min(p.n4 + 2 * (sg - p.st4), p.nb);
}

// slot boundaries of `parts` K ranges of about the same packed bytes (stage-aligned)
void gemv_split(const Plan &p, int parts, int *bound) {
    const int g1 = p.nst;
    const int64_t total = slot_off_g(p.n4, gemv_stage_lo(p, g1));
    int gb[9];
    gb[0] = 0;
    for (int r = 1; r < parts; ++r) {
        int s = gb[r - 1] + 1;
        while (s < g1 - (parts - r) && slot_off_g(p.n4, gemv_stage_lo(p, s)) * parts < total * r) ++s;
        gb[r] = s;
    }
    gb[parts] = g1;
    for (int r = 0; r <= parts; ++r) bound[r] = gemv_stage_lo(p, gb[r]);
}

size_t gemv_smem(int ns, int MT, int GS) {
    return (size_t)2 * GS * MT * 128 * 4 + (size_t)kGSets * MT * 128 * 4 + ((size_t)ns * MT * 33 + 15) / 16 * 16;
}

int sms_now() {
    static int cached = 0;
    if (!cached) {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0)
            cached = n;
        else
            return 152;
    }
    return cached;
}

}  // namespace

int launch_gemv_decode(const Plan *const *plans, const void *const *x, const int64_t *ld_x, const void *const *packed,
                       const int64_t *N, float *const *y, const int64_t *ld_y, int count, int64_t M, int rounding,
                       bool pdl, cudaStream_t st) {
    if (count < 1 || count > kGMaxProblems) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d)", count, kGMaxProblems);
    if (M < 1 || M > kGemvMaxM) return fail(MXS_ERR_SHAPE, "the CUDA-core decode path takes 1 <= M <= %d", kGemvMaxM);
    const int MT = M == 1 ? 1 : (M == 2 ? 2 : 4);
    const int sms = sms_now();
    int64_t G[kGMaxProblems], bytes[kGMaxProblems];
    for (int i = 0; i < count; ++i) {
        if (N[i] > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
        G[i] = weight_offsets(*plans[i], N[i], false).G;
        bytes[i] = weight_offsets(*plans[i], N[i], false).GB;
    }
    // One cluster size for the launch.  A CTA's time is about its groups x the
    // bytes of its K range of one group (the stream), plus a fixed cost per
    // group and, in a cluster, per cluster barrier; CTAs are handed one at a
    // time to the problem whose slowest CTA costs most.
    auto cost = [&](int i, int GS, int n) {
        const double rounds = (double)((G[i] + n - 1) / n);
        return rounds * ((double)bytes[i] / GS / 40.0 + (GS > 1 ? 3000.0 : 1500.0));  // ~40 bytes per cycle per SM
    };
    double best = 1e300;
    int bestGS = 1, bestn[kGMaxProblems] = {};
    for (int GS = 1; GS <= 8; GS *= 2) {
        bool ok = sms / GS >= count;
        for (int i = 0; i < count && ok; ++i) {
            ok = GS <= plans[i]->nst;
            if (!ok) break;
            int bound[9], most = 0;
            gemv_split(*plans[i], GS, bound);
            for (int r = 0; r < GS; ++r) most = std::max(most, bound[r + 1] - bound[r]);
            ok = gemv_smem(most, MT, GS) <= (size_t)200 * 1024;
        }
        if (!ok) continue;
        int n[kGMaxProblems], used = count;
        for (int i = 0; i < count; ++i) n[i] = 1;
        while (used < sms / GS) {
            int worst = -1;
            double wc = -1.0;
            for (int i = 0; i < count; ++i)
                if (n[i] < G[i] && cost(i, GS, n[i]) > wc) wc = cost(i, GS, n[i]), worst = i;
            if (worst < 0) break;
            ++n[worst];
            ++used;
        }
        double c = 0.0;
        for (int i = 0; i < count; ++i) c = std::max(c, cost(i, GS, n[i]));
        if (c < best * 0.98) {
            best = c;
            bestGS = GS;
            for (int i = 0; i < count; ++i) bestn[i] = n[i];
        }
    }
    if (best >= 1e299) return fail(MXS_ERR_SHAPE, "decode: K too large for the CUDA-core path");
    // the parameter block carries the slot tables (a few KB): built on the host
    static thread_local GemvParams gp;
    std::memset(&gp, 0, sizeof(gp));
    gp.nprob = count;
    gp.M = (int)M;
    gp.rhaz = rounding == MXS_RHAZ;
    int cta = 0, max_ns = 0;
    for (int i = 0; i < count; ++i) {
        const Plan &p = *plans[i];
        GemvProblem &P = gp.prob[i];
        P.x = static_cast<const uint16_t *>(x[i]);
        P.w = static_cast<const uint8_t *>(packed[i]);
        P.y = y[i];
        P.ld_x = ld_x[i];
        P.ld_y = ld_y[i];
        P.GB = bytes[i];
        P.N = (int)N[i];
        P.G = (int)G[i];
        P.GS = bestGS;
        P.nb = p.nb, P.n4 = p.n4, P.n6 = p.n6;
        gemv_split(p, bestGS, P.bound);
        for (int r = bestGS + 1; r < 9; ++r) P.bound[r] = P.bound[bestGS];
        for (int r = 0; r < bestGS; ++r) max_ns = std::max(max_ns, P.bound[r + 1] - P.bound[r]);
        P.cta0 = cta;
        P.ncta = bestn[i];
        cta += bestn[i];
        std::memcpy(gp.slot_block[i], p.slot_block, sizeof(uint16_t) * (size_t)p.nb);
    }
    const size_t smem = gemv_smem(max_ns, MT, bestGS);
    using Kernel = void (*)(GemvParams);
    const Kernel k = MT == 1 ? gemv_decode_kernel<1> : (MT == 2 ? gemv_decode_kernel<2> : gemv_decode_kernel<4>);
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(gemv smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cta, (unsigned)bestGS, 1);
    cfg.blockDim = dim3(kGThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    int na = 0;
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = (unsigned)bestGS;
    attr[na].val.clusterDim.z = 1;
    ++na;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    e = cudaLaunchKernelEx(&cfg, k, gp);
    return cuda_fail(e, "gemv_decode_kernel launch");
}

}  // namespace mxs
