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
// the CUDA cores: per weight word of four codes, two integer operations and
// two dp4a per token add four products exactly.  The work per token grows
// with M while the tensor-core path's does not (an earlier form of this
// kernel, over twelve LLaMA-2-70B layers: 1.91 ms at M = 1 against 2.41 ms,
// but 3.6 ms at M = 4 against 2.43 ms), so the library sends it
// M <= kGemvMaxM (1) tokens.
//
// Work.  A CTA owns 128-row weight groups (and, in a thread-block cluster, a
// K range of them).  Prologue: it quantizes the activations of its K range
// (x is bf16; the rule, bit for bit, of mxs_quantize_act) into shared memory
// as int8 codes and scale bytes, in slot order.  One lane of a producer warp
// streams the group's K range into a ring of shared-memory stages with
// cp.async.bulk (sixteen 4-bit slots or eight 6/8-bit slots, about 34 KB per
// stage, four stages in flight), starting before the wait for the kernel
// before (the weights are static).  Main loop: consumer thread t of four sets
// of 128 is weight row t % 128, and set t / 128 takes the slots
// lo + t / 128 + 4j of a stage; per slot it reads its row's codes (16 or 32
// bytes) and scale byte from the stage, forms the integer dots with dp4a
// straight from the sign-magnitude codes (two integer operations and two dp4a
// per four codes) and adds 2^(Ea'+Ew') * D into an fp32 accumulator per token
// (the product is exact: |D| < 2^20 times a power of two).  Copies in flight
// keep HBM busy; the consumers' integer work is what bounds the kernel.  The
// sets' sums are added in set order; cluster ranks write theirs into rank 0's
// shared memory (distributed shared-memory stores, then a cluster barrier)
// and rank 0 adds them in rank order: deterministic.  Every wait on a stage is
// bounded: on expiry the kernel records MXS_ERR_TIMEOUT (mxs_device_status),
// skips the rest of its arithmetic while still taking its barriers, and waits
// for its copies.
#include <algorithm>
#include <cstring>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {

__device__ int g_gemv_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

constexpr int kGSets = 4;                    // consumer sets; a set is 128 threads, one per weight row
constexpr int kConsumers = 4 * kGSets;       // consumer warps
constexpr int kCThreads = 32 * kConsumers;   // 512
constexpr int kGThreads = kCThreads + 32;    // + the producer warp
constexpr int kGMaxProblems = 3;
#ifndef MXS_GEMV_RING
#define MXS_GEMV_RING 4
#endif
constexpr int kRing = MXS_GEMV_RING;         // shared-memory stages in flight
constexpr int kSlots4 = 16, kSlots68 = 8;    // slots per stage: four (two) per consumer set
constexpr int kStageBytes = 2176 * kSlots4;  // 34816 >= 8 x 4224
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock

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

__host__ __device__ __forceinline__ int64_t slot_off_g(int n4, int s) {
    return s < n4 ? 2176 * (int64_t)s : 2176 * (int64_t)n4 + 4224 * (int64_t)(s - n4);
}
// stage k of a rank's slot range [c0, c1), 4-bit slots [c0, e4): slots [lo, hi)
__host__ __device__ __forceinline__ void stage_range(int c0, int e4, int c1, int k, int &lo, int &hi) {
    const int n4s = (e4 - c0 + kSlots4 - 1) / kSlots4;
    if (k < n4s) {
        lo = c0 + kSlots4 * k;
        hi = min(lo + kSlots4, e4);
    } else {
        lo = e4 + kSlots68 * (k - n4s);
        hi = min(lo + kSlots68, c1);
    }
}
__host__ __device__ __forceinline__ int stage_count(int c0, int e4, int c1) {
    return (e4 - c0 + kSlots4 - 1) / kSlots4 + (c1 - e4 + kSlots68 - 1) / kSlots68;
}
// shared memory: the cluster exchange first (its offset is the same in every
// rank), the sets' partial sums, the barriers and abort flag, the stage ring
// (128-byte aligned), the token codes and scale bytes
__host__ __device__ __forceinline__ size_t off_part(int GS, int MT) { return (size_t)2 * GS * MT * 128 * 4; }
__host__ __device__ __forceinline__ size_t off_bars(int GS, int MT) {
    return off_part(GS, MT) + (size_t)kGSets * MT * 128 * 4;
}
__host__ __device__ __forceinline__ size_t off_ring(int GS, int MT) {
    return (off_bars(GS, MT) + 2 * kRing * 8 + 16 + 127) / 128 * 128;
}
__host__ __device__ __forceinline__ size_t off_tok(int GS, int MT) {
    return off_ring(GS, MT) + (size_t)kRing * kStageBytes;
}

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
__device__ __forceinline__ bool mbar_poll(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait; on expiry the CTA's abort flag and the sticky status are set
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (mbar_poll(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (mbar_poll(bar, parity)) return true;
        if ((i & 63) == 0) {
            if (*abort) return false;
            if (clock64() - t0 > kWaitCycles) {
                *abort = 1;
                atomicExch(&g_gemv_status, MXS_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
// whole-warp wait: lane 0 polls, then every lane takes its own acquiring test
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok) mbar_poll(bar, parity);
    return ok;
}
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_poll(bar, parity) && clock64() - t0 < kWaitCycles) {
    }
}
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     su32(dst)),
                 "l"(src), "r"(bytes), "r"(su32(bar))
                 : "memory");
}
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ uint32_t map_rank(const void *p, uint32_t rank) {
    uint32_t ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(su32(p)), "r"(rank));
    return ra;
}
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire;" ::: "memory"); }

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
// 0xFF in every byte of x whose bit 7 is set (prmt's sign-replicate mode)
__device__ __forceinline__ uint32_t sign_bytes(uint32_t x) { return prmt(x, 0u, 0xBA98u); }

// acc + D * 2^(Sa+Sw-254-2(b-2)) (D exact in fp32); NaN when either scale
// byte is 255; scales outside the normal fp32 range take ldexpf
__device__ __forceinline__ float fold(float acc, int D, int Sa, int Sw, int b) {
    const int e = Sa + Sw - 127 - 2 * (b - 2);  // the biased fp32 exponent of the block's unit
    if ((uint32_t)(e - 1) < 254u && Sa != 255 && Sw != 255) return fmaf((float)D, __int_as_float(e << 23), acc);
    if (Sa == 255 || Sw == 255) return __int_as_float(0x7FC00000);
    return acc + ldexpf((float)D, e - 127);
}

// The integer dot of a weight row's block with a token's block, from the
// sign-magnitude codes as stored.  With smask = 0xFF in the bytes of the
// negative codes, y = |m| ^ smask is |m| for a positive code and -|m| - 1
// (two's complement) for a negative one, so
//   sum v_i a_i = dp4a(y, a) - dp4a(smask, a)
// (a negative zero gives y = smask = -1 and adds nothing).  Two integer
// operations and two dp4a per four codes, each dp4a chain exact (|sum| < 2^20).

// one 4-bit slot of row r from a stage: 16 code bytes (byte 4i+j: element
// 8i+j low nibble, 8i+4+j high nibble) and the scale byte; tc / ts the slot's
// token codes and scale bytes
template <int MT>
__device__ __forceinline__ void slot4(const uint8_t *sl, int r, const int8_t *tc, const uint8_t *ts,
                                      float (&acc)[MT]) {
    const uint4 v = *reinterpret_cast<const uint4 *>(sl + 16 * r);
    const int Sw = sl[2048 + r];
    const uint32_t wd[4] = {v.x, v.y, v.z, v.w};
    uint32_t ylo[4], slo[4], yhi[4], shi[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        slo[i] = sign_bytes(wd[i] << 4);  // the low nibble's sign (bit 3) moved to bit 7
        shi[i] = sign_bytes(wd[i]);
        ylo[i] = (wd[i] & 0x07070707u) ^ slo[i];
        yhi[i] = ((wd[i] >> 4) & 0x07070707u) ^ shi[i];
    }
#pragma unroll
    for (int t = 0; t < MT; ++t) {
        const uint4 *tq = reinterpret_cast<const uint4 *>(tc + 32 * t);
        const uint4 ta = tq[0], tb = tq[1];
        const int tw[8] = {(int)ta.x, (int)ta.y, (int)ta.z, (int)ta.w, (int)tb.x, (int)tb.y, (int)tb.z, (int)tb.w};
        int D0 = 0, D1 = 0, E0 = 0, E1 = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            D0 = __dp4a((int)ylo[i], tw[2 * i], D0);
            E0 = __dp4a((int)slo[i], tw[2 * i], E0);
            D1 = __dp4a((int)yhi[i], tw[2 * i + 1], D1);
            E1 = __dp4a((int)shi[i], tw[2 * i + 1], E1);
        }
        acc[t] = fold(acc[t], (D0 + D1) - (E0 + E1), ts[t], Sw, 4);
    }
}

// one 6/8-bit slot of row r: 32 code bytes (byte e: element e, sign at bit 7)
// and the scale byte
template <int MT>
__device__ __forceinline__ void slot68(const uint8_t *sl, int r, int b, const int8_t *tc, const uint8_t *ts,
                                       float (&acc)[MT]) {
    const uint4 v0 = *reinterpret_cast<const uint4 *>(sl + 32 * r);
    const uint4 v1 = *reinterpret_cast<const uint4 *>(sl + 32 * r + 16);
    const int Sw = sl[4096 + r];
    const uint32_t wd[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
    uint32_t y[8], sm[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        sm[i] = sign_bytes(wd[i]);
        y[i] = (wd[i] & 0x7F7F7F7Fu) ^ sm[i];
    }
#pragma unroll
    for (int t = 0; t < MT; ++t) {
        const uint4 *tq = reinterpret_cast<const uint4 *>(tc + 32 * t);
        const uint4 ta = tq[0], tb = tq[1];
        const int tw[8] = {(int)ta.x, (int)ta.y, (int)ta.z, (int)ta.w, (int)tb.x, (int)tb.y, (int)tb.z, (int)tb.w};
        int D0 = 0, D1 = 0, E0 = 0, E1 = 0;
#pragma unroll
        for (int i = 0; i < 8; i += 2) {
            D0 = __dp4a((int)y[i], tw[i], D0);
            E0 = __dp4a((int)sm[i], tw[i], E0);
            D1 = __dp4a((int)y[i + 1], tw[i + 1], D1);
            E1 = __dp4a((int)sm[i + 1], tw[i + 1], E1);
        }
        acc[t] = fold(acc[t], (D0 + D1) - (E0 + E1), ts[t], Sw, b);
    }
}

template <int MT>
__global__ void __launch_bounds__(kGThreads, 1) gemv_decode_kernel(const __grid_constant__ GemvParams gp) {
    int pi = 0;
    while (pi + 1 < gp.nprob && (int)blockIdx.x >= gp.prob[pi + 1].cta0) ++pi;
    const GemvProblem &P = gp.prob[pi];
    const uint16_t *sblk = gp.slot_block[pi];
    const int bx = (int)blockIdx.x - P.cta0, gx = P.ncta, GS = P.GS;
    const uint32_t rank = GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = P.bound[rank], c1 = P.bound[rank + 1], ns = c1 - c0;
    const int e4 = max(c0, min(c1, P.n4));  // 4-bit slots [c0, e4), 6/8-bit slots [e4, c1)
    const int nst = stage_count(c0, e4, c1);
    const int M = gp.M, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ngroups = bx < P.G ? (P.G - 1 - bx) / gx + 1 : 0;

    extern __shared__ __align__(128) uint8_t smem[];
    float *xbuf = reinterpret_cast<float *>(smem);                          // [2][GS][MT][128] (read in rank 0)
    float *part = reinterpret_cast<float *>(smem + off_part(GS, MT));       // [sets][MT][128]
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + off_bars(GS, MT));  // [kRing]
    uint64_t *empty = full + kRing;                                          // [kRing]
    volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + kRing);
    uint8_t *ring = smem + off_ring(GS, MT);                                // [kRing][kStageBytes]
    int8_t *tcode = reinterpret_cast<int8_t *>(smem + off_tok(GS, MT));    // [ns][MT][32] token codes
    uint8_t *tsc = reinterpret_cast<uint8_t *>(tcode) + (size_t)ns * MT * 32;  // [ns][MT] token scale bytes

    if (tid == 0) {
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kConsumers);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == kConsumers) {
        // ---- producer: the weight bytes of [c0, c1) of each group, stage by
        // stage (the weights are static: no wait for the kernel before).  Its
        // cluster barriers run one phase late, so that the copies run ahead:
        // phase 0 is the consumers' start, phase gi + 1 the end of group gi.
        int ctr = 0;
        bool ok = true;
        if (GS > 1) cluster_arrive();  // phase 0
        for (int gi = 0; gi < ngroups; ++gi) {
            if (lane == 0 && ok) {
                const uint8_t *base = P.w + (int64_t)(bx + gi * gx) * P.GB;
                for (int k = 0; k < nst; ++k, ++ctr) {
                    int lo, hi;
                    stage_range(c0, e4, c1, k, lo, hi);
                    const int i = ctr % kRing;
                    const uint32_t n = (uint32_t)(ctr / kRing);
                    if (*abort_flag || (n > 0 && !mbar_wait(&empty[i], (n - 1) & 1, abort_flag))) {
                        ok = false;
                        break;
                    }
                    const int64_t off = slot_off_g(P.n4, lo);
                    const uint32_t bytes = (uint32_t)(slot_off_g(P.n4, hi) - off);
                    mbar_expect_tx(&full[i], bytes);
                    bulk_load(ring + (size_t)i * kStageBytes, base + off, bytes, &full[i]);
                }
            }
            __syncwarp();
            if (GS > 1) {  // wait for phase gi, arrive for gi + 1
                cluster_wait();
                cluster_arrive();
            }
        }
        if (GS > 1) cluster_wait();  // the last phase
        if (lane == 0 && *abort_flag)  // drain: the last copy issued into each ring slot
            for (int i = 0; i < kRing && i < ctr; ++i) {
                const int last = i + (ctr - 1 - i) / kRing * kRing;
                drain_wait(&full[i], (uint32_t)(last / kRing) & 1);
            }
        return;
    }

    // ---- consumers.  Prologue: the activations of slots [c0, c1) as int8
    // codes (mxs_quantize_act's rule); x may come from the kernel before
    // (programmatic dependent launch)
    const int set = tid >> 7, r = tid & 127;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int i = tid; i < ns * MT; i += kCThreads) {
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
    named_sync(1, kCThreads);
    if (GS > 1) {  // phase 0: every rank runs before the first store into rank 0
        cluster_arrive();
        cluster_wait();
    }

    bool aborted = false;
    int ctr = 0;
    for (int gi = 0; gi < ngroups; ++gi) {
        const int g = bx + gi * gx;
        float acc[MT];
#pragma unroll
        for (int t = 0; t < MT; ++t) acc[t] = 0.0f;
        for (int k = 0; k < nst; ++k, ++ctr) {
            int lo, hi;
            stage_range(c0, e4, c1, k, lo, hi);
            const int i = ctr % kRing;
            if (!aborted && !warp_wait(&full[i], (uint32_t)(ctr / kRing) & 1, abort_flag)) aborted = true;
            if (!aborted) {
                const uint8_t *sb = ring + (size_t)i * kStageBytes;
                if (lo < P.n4) {
#pragma unroll
                    for (int j = 0; j < kSlots4 / kGSets; ++j) {
                        const int s = lo + set + kGSets * j;
                        if (s < hi) slot4<MT>(sb + 2176 * (s - lo), r, tcode + (size_t)(s - c0) * MT * 32,
                                              tsc + (s - c0) * MT, acc);
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < kSlots68 / kGSets; ++j) {
                        const int s = lo + set + kGSets * j;
                        if (s < hi) slot68<MT>(sb + 4224 * (s - lo), r, s < P.n4 + P.n6 ? 6 : 8,
                                               tcode + (size_t)(s - c0) * MT * 32, tsc + (s - c0) * MT, acc);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[i]);
        }

        // ---- the sets' sums in set order, then the ranks' in rank order
#pragma unroll
        for (int t = 0; t < MT; ++t) part[(set * MT + t) * 128 + r] = acc[t];
        named_sync(1, kCThreads);
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
        if (GS == 1) {
            if (set == 0 && n < P.N && !aborted)
#pragma unroll
                for (int t = 0; t < MT; ++t)
                    if (t < M) P.y[(int64_t)t * P.ld_y + n] = val[t];
        } else {
            float *xb = xbuf + (gi & 1) * GS * MT * 128;
            if (set == 0)
#pragma unroll
                for (int t = 0; t < MT; ++t) st_cluster_f32(map_rank(xb + (rank * MT + t) * 128 + r, 0), val[t]);
            cluster_arrive();  // phase gi + 1: every rank's partial sums are in rank 0
            cluster_wait();
            if (rank == 0 && set == 0 && n < P.N && !aborted)
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    if (t >= M) continue;
                    float v = xb[t * 128 + r];
                    for (int k = 1; k < GS; ++k) v += xb[(k * MT + t) * 128 + r];
                    P.y[(int64_t)t * P.ld_y + n] = v;
                }
        }
        named_sync(1, kCThreads);  // `part` is reused by the next group
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

size_t gemv_smem(int ns, int MT, int GS) { return off_tok(GS, MT) + ((size_t)ns * MT * 33 + 15) / 16 * 16; }

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

int gemv_status(int *status, int reset) {
    int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_gemv_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyFromSymbol(gemv status)");
    *status = v;
    if (reset && v != 0) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_gemv_status, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyToSymbol(gemv status)");
    }
    return MXS_OK;
}

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
