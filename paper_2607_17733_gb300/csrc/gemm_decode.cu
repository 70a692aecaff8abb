// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens) on
// the 5th-generation tensor cores, and its fusion with A1 (the activations
// quantized in the kernel's prologue).
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale) with the per-block widths of Sec. 4.1.
//
// Decode reads every weight byte once, so the kernel keeps the weights in
// their compact form (4-bit nibbles, 6/8-bit bytes) all the way into shared
// memory and does all arithmetic on the tensor core:
//   * the block-scaled FP8 MMA (tcgen05.mma kind::mxf8f6f4, scale_vec::1X)
//     with the weights as the 128-row A operand and the <= 16 tokens as the
//     N = 16 B operand; per-block scales are applied by the hardware and the
//     sum over K stays in an fp32 tensor-memory accumulator;
//   * a code of magnitude <= 15 is fed as the e4m3 byte (sign << 7) | |m|,
//     whose value is |m| * 2^-9 (subnormals and the first binade); 6/8-bit
//     codes split as |m| = 16h + l into two such digits (Sec. 6: high- and
//     low-precision parts multiplied separately).  The fixed-point weight of
//     each digit goes into the E8M0 scale byte (+7 for a 4-bit code, +9/+5
//     for the high/low digit of a 6-bit code, +7/+3 for an 8-bit one), on both
//     operands, so every MMA term is exact;
//   * warp 0 streams each 128-row weight group's K range into a ring of
//     shared-memory stages with cp.async.bulk (about 17 KB per copy; the copy
//     count, not the byte count, limits bulk-copy throughput);
//   * warps 6-9 convert a stage into e4m3 digit planes in the 128-byte
//     swizzled K-major layout the MMA reads (one row per thread, a handful of
//     integer operations per 8 codes) and write the weight scale tile;
//   * warp 1 owns tensor memory and issues tcgen05.cp (scales) and the MMAs;
//   * warps 2-5 build the token operand for the CTA's whole K range before
//     the main loop, then drain the accumulator (tcgen05.ld) and store y;
//   * K is split over the CTAs of a thread-block cluster when N alone cannot
//     occupy the GPU or the token operand would not fit; the other ranks hand
//     their partial accumulators to rank 0 through distributed shared memory
//     (mbarrier-signalled) and rank 0 adds them in rank order.  A K range too
//     large for one cluster's shared memory runs as several passes, each
//     adding into y.
// Every mbarrier wait is bounded; on expiry the kernel records
// MXS_ERR_TIMEOUT, stops, drains what it issued and frees tensor memory.
// Scale bytes above 245 (|x| >= 2^118) saturate at 254 after the digit shift.
#include <algorithm>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {

__device__ int g_decode_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

constexpr int kThreads = 320;  // 10 warps
constexpr int kConv = 3;        // converted weight-plane stages
constexpr int kPlaneBytes = 128 * 128;  // 128 rows x 128 bytes of K' (SW128)
constexpr int kTokBytes = 16 * 128;     // 16 token rows x 128 bytes of K'
constexpr int kTmemCols = 64;           // 2 x 16 accumulator columns + kConv x 8 scale columns
constexpr int kSfCol = 32;
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock

struct DecodeArgs {
    const uint8_t *codes;   // [M, row_bytes] packed activation codes (NULL when x is given)
    const uint8_t *scales;  // [M, nb]
    const uint16_t *x;      // bf16 [M, ld_x] activations for the fused entry point (or NULL)
    int64_t ld_x;
    int rhaz;
    const uint8_t *w;  // packed weight buffer
    float *y;
    int64_t ld_y;
    int M, N, G;           // tokens, output features, 128-row groups
    int GS;                // CTAs per cluster along K
    int bound[9];          // rank r streams slots [bound[r], bound[r+1]) (balanced by bytes)
    int ring, ring_bytes;  // copy stages, bytes per copy stage
    int max_mst;           // most MMA stages any rank holds (token operand carve)
    int accumulate;        // add into y (a later K pass) instead of storing
    int64_t GB;            // bytes of one 128-row weight group
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
template <bool kCluster>
__device__ __forceinline__ bool poll(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    if (kCluster)
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
            " selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(su32(bar)), "r"(parity)
            : "memory");
    else
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(su32(bar)), "r"(parity)
            : "memory");
    return ok != 0;
}
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (poll<kCluster>(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (poll<kCluster>(bar, parity)) return true;
        if ((i & 63) == 0) {  // the bound is checked every 64 polls
            if (*abort) return false;
            if (clock64() - t0 > kWaitCycles) {
                *abort = 1;
                atomicExch(&g_decode_status, MXS_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
// whole-warp wait: one lane polls, then every lane takes its own acquiring test
template <bool kCluster = false>
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    bool ok = true;
    if ((threadIdx.x & 31) == 0) ok = mbar_wait<kCluster>(bar, parity, abort);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok) poll<kCluster>(bar, parity);
    return ok;
}
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!poll<false>(bar, parity) && clock64() - t0 < kWaitCycles) {
    }
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
// generic-proxy shared-memory writes -> visible to the tensor core / tcgen05.cp
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// UMMA shared-memory descriptors (as in the prefill kernel): 128B-swizzled
// K-major operand tiles (8-row atoms of 1024 B) and 32 x 16 B scale tiles.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t desc_sf(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)(128 >> 4) << 32) | ((uint64_t)1 << 46);
}
// kind::mxf8f6f4, e4m3 x e4m3, K-major, N = 16, UE8M0 scales, M = 128
constexpr uint32_t kIdesc = ((uint32_t)(16 >> 3) << 17) | (1u << 23) | ((uint32_t)(128 >> 4) << 24);
__device__ __forceinline__ uint32_t idesc(int sfa_id, int sfb_id) {
    return kIdesc | ((uint32_t)sfb_id << 4) | ((uint32_t)sfa_id << 29);
}
__device__ __forceinline__ void mma_mx(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t sfa, uint32_t sfb,
                                       uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"(accum), "r"(sfa), "r"(sfb)
        : "memory");
}
__device__ __forceinline__ void tmem_cp_sf(uint32_t taddr, uint64_t desc) {
    asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
                 : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// byte offset of 16-byte chunk c (0..7) of row r in a 128B-swizzled K-major tile
__device__ __forceinline__ uint32_t sw128(int r, int c) { return (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4); }

// e4m3 bytes of |m| * 2^-9 with sign, for four sign-magnitude 4-bit codes held
// one per byte (low nibble): (s << 3) | |m|  ->  (s << 7) | |m|
__device__ __forceinline__ uint32_t nib_to_e4m3(uint32_t v) { return v + 15u * (v & 0x08080808u); }
// high (|m| >> 4) and low (|m| & 15) digit of four sign-magnitude 8-bit codes
__device__ __forceinline__ uint32_t hi_digit(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t lo_digit(uint32_t x) { return x & 0x8F8F8F8Fu; }
// scale byte carrying the digit's fixed-point weight; 255 (NaN) stays
__device__ __forceinline__ uint32_t shifted(int S, int sh) { return S == 255 ? 255u : (uint32_t)min(S + sh, 254); }

struct Stages {  // MMA stages of a CTA's K range [c0, c1): 4-bit ones (4 slots), then 6/8-bit ones (2 slots)
    int a4, e4, a8, e8, st4, n;
    __device__ void init(const Plan &p, int c0, int c1) {
        a4 = min(c0, p.n4);
        e4 = min(c1, p.n4);
        a8 = max(c0, p.n4);
        e8 = max(c1, p.n4);
        st4 = (max(0, e4 - a4) + 3) / 4;
        n = st4 + (max(0, e8 - a8) + 1) / 2;
    }
    __device__ void range(int st, int &lo, int &hi) const {
        if (st < st4) {
            lo = a4 + 4 * st;
            hi = min(e4, lo + 4);
        } else {
            lo = a8 + 2 * (st - st4);
            hi = min(e8, lo + 2);
        }
    }
};

__global__ void __launch_bounds__(kThreads, 1) gemm_decode_kernel(const __grid_constant__ Plan p,
                                                                  const __grid_constant__ DecodeArgs a) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sbase = su32(smem_raw);
    uint8_t *smem = smem_raw + (((sbase + 1023) & ~1023u) - sbase);  // 1024-aligned for the swizzled tiles
    uint8_t *planes = smem;                                   // kConv x 16 KB
    uint8_t *tok = planes + kConv * kPlaneBytes;              // max_mst x 2 KB
    uint8_t *sfa = tok + (size_t)a.max_mst * kTokBytes;       // kConv x 512
    uint8_t *sfb = sfa + kConv * 512;                         // max_mst x 512
    uint8_t *ring = sfb + (size_t)a.max_mst * 512;            // ring x ring_bytes
    float *xbuf = reinterpret_cast<float *>(ring + (size_t)a.ring * a.ring_bytes);  // [GS-1][128][16]
    uint64_t *bars = reinterpret_cast<uint64_t *>(xbuf + (size_t)(a.GS - 1) * 128 * 16);
    uint64_t *full_c = bars, *empty_c = full_c + a.ring;
    uint64_t *conv_full = empty_c + a.ring, *conv_empty = conv_full + kConv;
    uint64_t *acc_full = conv_empty + kConv, *acc_empty = acc_full + 2;
    uint64_t *tok_ready = acc_empty + 2, *xfull = tok_ready + 1, *xempty = xfull + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(xempty + 1);
    int *abort_flag = reinterpret_cast<int *>(tmem_slot + 1);
    volatile int *abort = abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = a.GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = a.bound[rank], c1 = a.bound[rank + 1];
    Stages S;
    S.init(p, c0, c1);
    const int nchunks = (S.n + 1) / 2;  // a copy stage holds two MMA stages

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.ring; ++i) {
            mbar_init(&full_c[i], 1);
            mbar_init(&empty_c[i], 4);  // the four converter warps
        }
        for (int i = 0; i < kConv; ++i) {
            mbar_init(&conv_full[i], 4);
            mbar_init(&conv_empty[i], 1);  // tcgen05.commit
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);  // the four epilogue warps
        }
        mbar_init(tok_ready, 4);
        mbar_init(xfull, (uint32_t)(a.GS - 1) * 128);
        mbar_init(xempty, 128);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    if (a.GS > 1) cg::this_cluster().sync();  // partners' barriers exist before any remote access
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t qc = 0;
            bool stop = false;
            for (int g = blockIdx.x; g < a.G && !stop; g += gridDim.x) {
                for (int k = 0; k < nchunks; ++k, ++qc) {
                    const int s = (int)(qc % a.ring);
                    if (!mbar_wait(&empty_c[s], ((qc / a.ring) & 1) ^ 1, abort)) { stop = true; break; }
                    int lo, hi, lo2, hi2;
                    S.range(2 * k, lo, hi);
                    if (2 * k + 1 < S.n) S.range(2 * k + 1, lo2, hi2); else hi2 = hi;
                    const int64_t off = slot_offset(p, lo);
                    const uint32_t bytes = (uint32_t)(slot_offset(p, hi2) - off);
                    mbar_expect_tx(&full_c[s], bytes);
                    bulk_load(ring + (size_t)s * a.ring_bytes, a.w + (int64_t)g * a.GB + off, bytes, &full_c[s]);
                }
            }
            const uint32_t first = qc > (uint32_t)a.ring ? qc - a.ring : 0;
            for (uint32_t k = first; k < qc; ++k) drain_wait(&full_c[k % a.ring], (k / a.ring) & 1);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = mbar_wait(tok_ready, 0, abort);
            uint32_t qs = 0;
            int gi = 0, last = -1;
            for (int g = blockIdx.x; g < a.G && ok; g += gridDim.x, ++gi) {
                const int b = gi & 1;
                if (!mbar_wait(&acc_empty[b], ((gi >> 1) & 1) ^ 1, abort)) break;
                fence_after();
                const uint32_t acc = tmem + 16 * b;
                for (int st = 0; st < S.n; ++st, ++qs) {
                    const int pc = (int)(qs % kConv);
                    if (!mbar_wait(&conv_full[pc], (qs / kConv) & 1, abort)) { ok = false; break; }
                    fence_after();
                    const uint32_t sfa_t = tmem + kSfCol + 8 * pc, sfb_t = sfa_t + 4;
                    tmem_cp_sf(sfa_t, desc_sf(su32(sfa + pc * 512)));
                    tmem_cp_sf(sfb_t, desc_sf(su32(sfb + st * 512)));
                    const uint32_t a_addr = su32(planes + pc * kPlaneBytes), b_addr = su32(tok + st * kTokBytes);
                    if (st < S.st4) {
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            mma_mx(acc, desc_sw128(a_addr + 32 * q), desc_sw128(b_addr + 32 * q), idesc(q, q), sfa_t,
                                   sfb_t, (st > 0 || q > 0) ? 1u : 0u);
                    } else {
#pragma unroll
                        for (int j = 0; j < 2; ++j)
#pragma unroll
                            for (int pp = 0; pp < 4; ++pp) {
                                const int pa = pp >> 1, pb = pp & 1;
                                mma_mx(acc, desc_sw128(a_addr + 64 * j + 32 * pa), desc_sw128(b_addr + 64 * j + 32 * pb),
                                       idesc(2 * j + pa, 2 * j + pb), sfa_t, sfb_t, (st > 0 || j > 0 || pp > 0) ? 1u : 0u);
                            }
                    }
                    mma_commit(&conv_empty[pc]);  // frees the plane stage once these MMAs have read it
                    last = (int)qs;
                }
                if (!ok) break;
                mma_commit(&acc_full[b]);
            }
            if (last >= 0) drain_wait(&conv_empty[last % kConv], ((uint32_t)last / kConv) & 1);
        }
    } else if (warp >= 6) {
        // ------------------------------------------------------------ converters: one weight row per thread
        const int r = threadIdx.x - 192;  // 0..127
        uint32_t qc = 0, qs = 0;
        bool stop = false;
        for (int g = blockIdx.x; g < a.G && !stop; g += gridDim.x) {
            for (int k = 0; k < nchunks && !stop; ++k, ++qc) {
                const int s = (int)(qc % a.ring);
                if (!warp_wait(&full_c[s], (qc / a.ring) & 1, abort)) { stop = true; break; }
                int clo, chi;
                S.range(2 * k, clo, chi);
                const uint8_t *chunk = ring + (size_t)s * a.ring_bytes - slot_offset(p, clo);  // + slot_offset(slot)
                for (int st = 2 * k; st < min(2 * k + 2, S.n); ++st, ++qs) {
                    const int pc = (int)(qs % kConv);
                    if (!warp_wait(&conv_empty[pc], ((qs / kConv) & 1) ^ 1, abort)) { stop = true; break; }
                    int lo, hi;
                    S.range(st, lo, hi);
                    uint8_t *pl = planes + pc * kPlaneBytes;
                    uint32_t sfw = 0;
                    if (st < S.st4) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 o0 = make_uint4(0, 0, 0, 0), o1 = o0;
                            if (lo + q < hi) {
                                const uint8_t *slot = chunk + slot_offset(p, lo + q);
                                const uint4 v = *reinterpret_cast<const uint4 *>(slot + 16 * r);
                                // word i: bytes hold elements 8i..8i+3 (low nibbles), 8i+4..8i+7 (high nibbles)
                                o0 = make_uint4(nib_to_e4m3(v.x & 0x0F0F0F0Fu), nib_to_e4m3((v.x >> 4) & 0x0F0F0F0Fu),
                                                nib_to_e4m3(v.y & 0x0F0F0F0Fu), nib_to_e4m3((v.y >> 4) & 0x0F0F0F0Fu));
                                o1 = make_uint4(nib_to_e4m3(v.z & 0x0F0F0F0Fu), nib_to_e4m3((v.z >> 4) & 0x0F0F0F0Fu),
                                                nib_to_e4m3(v.w & 0x0F0F0F0Fu), nib_to_e4m3((v.w >> 4) & 0x0F0F0F0Fu));
                                sfw |= shifted(slot[2048 + r], 7) << (8 * q);
                            }
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 2 * q)) = o0;
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 2 * q + 1)) = o1;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 2; ++j) {
                            uint4 h0 = make_uint4(0, 0, 0, 0), h1 = h0, l0 = h0, l1 = h0;
                            if (lo + j < hi) {
                                const uint8_t *slot = chunk + slot_offset(p, lo + j);
                                const uint4 v0 = *reinterpret_cast<const uint4 *>(slot + 32 * r);
                                const uint4 v1 = *reinterpret_cast<const uint4 *>(slot + 32 * r + 16);
                                h0 = make_uint4(hi_digit(v0.x), hi_digit(v0.y), hi_digit(v0.z), hi_digit(v0.w));
                                h1 = make_uint4(hi_digit(v1.x), hi_digit(v1.y), hi_digit(v1.z), hi_digit(v1.w));
                                l0 = make_uint4(lo_digit(v0.x), lo_digit(v0.y), lo_digit(v0.z), lo_digit(v0.w));
                                l1 = make_uint4(lo_digit(v1.x), lo_digit(v1.y), lo_digit(v1.z), lo_digit(v1.w));
                                const int Sw = slot[4096 + r];
                                const bool six = slot_width(p, lo + j) == 6;
                                sfw |= (shifted(Sw, six ? 9 : 7) | (shifted(Sw, six ? 5 : 3) << 8)) << (16 * j);
                            }
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * j)) = h0;
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * j + 1)) = h1;
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * j + 2)) = l0;
                            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * j + 3)) = l1;
                        }
                    }
                    // scale tile: row r at lane r%32, column r/32; byte = sf id
                    *reinterpret_cast<uint32_t *>(sfa + pc * 512 + (r & 31) * 16 + (r >> 5) * 4) = sfw;
                    fence_async_smem();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&conv_full[pc]);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty_c[s]);
            }
        }
    } else {
        // ------------------------------------------------------------ warps 2-5: token operand, then epilogue
        const int et = threadIdx.x - 64;  // 0..127
        // zero the token planes and scale tiles of every stage, then fill them
        for (int i = et; i < S.n * (kTokBytes + 512) / 16; i += 128) {
            const int off = i * 16;
            uint8_t *dst = off < S.n * kTokBytes ? tok + off : sfb + (off - S.n * kTokBytes);
            *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        for (int it = et; it < (c1 - c0) * 16; it += 128) {
            const int s = c0 + it / 16, t = it % 16;
            if (t >= a.M) continue;
            const int b = slot_width(p, s);
            int m[32];
            int Sa;
            if (a.x) {  // fused: quantize the bf16 block here (same integer rounding as mxs_quantize_act)
                const uint4 *src = reinterpret_cast<const uint4 *>(a.x + (int64_t)t * a.ld_x + kBlock * p.slot_block[s]);
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
                Sa = (int)(mag >> 7);
#pragma unroll
                for (int i = 0; i < 32; ++i) m[i] = Sa == 255 ? 0 : quant_elem(h[i], Sa, b, a.rhaz);
            } else {  // from the packed activation codes
                const uint8_t *row = a.codes + (int64_t)t * p.row_bytes;
                Sa = a.scales[(int64_t)t * p.nb + s];
                if (b == 4) {
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
            // digits (sign-magnitude e4m3 bytes) at this slot's K' position of its MMA stage
            int st, pos;
            if (s < p.n4) {
                st = (s - S.a4) / 4;
                pos = 32 * ((s - S.a4) % 4);
            } else {
                st = S.st4 + (s - S.a8) / 2;
                pos = 64 * ((s - S.a8) % 2);
            }
            uint32_t d0[8], d1[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                uint32_t hw = 0, lw = 0;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int v = m[4 * i + j];
                    const uint32_t sg = v < 0 ? 0x80u : 0u, mg = (uint32_t)(v < 0 ? -v : v);
                    if (b == 4) {
                        hw |= (sg | mg) << (8 * j);
                    } else {
                        hw |= (sg | (mg >> 4)) << (8 * j);
                        lw |= (sg | (mg & 15u)) << (8 * j);
                    }
                }
                d0[i] = hw;
                d1[i] = lw;
            }
            uint8_t *trow = tok + st * kTokBytes;
            const int c = pos / 16;  // first 16-byte chunk
            *reinterpret_cast<uint4 *>(trow + sw128(t, c)) = make_uint4(d0[0], d0[1], d0[2], d0[3]);
            *reinterpret_cast<uint4 *>(trow + sw128(t, c + 1)) = make_uint4(d0[4], d0[5], d0[6], d0[7]);
            uint8_t *sft = sfb + st * 512 + (t & 31) * 16 + (t >> 5) * 4;
            if (b == 4) {
                sft[(s - S.a4) % 4] = (uint8_t)shifted(Sa, 7);
            } else {
                *reinterpret_cast<uint4 *>(trow + sw128(t, c + 2)) = make_uint4(d1[0], d1[1], d1[2], d1[3]);
                *reinterpret_cast<uint4 *>(trow + sw128(t, c + 3)) = make_uint4(d1[4], d1[5], d1[6], d1[7]);
                const int j = (s - S.a8) % 2;
                sft[2 * j] = (uint8_t)shifted(Sa, b == 6 ? 9 : 7);
                sft[2 * j + 1] = (uint8_t)shifted(Sa, b == 6 ? 5 : 3);
            }
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(tok_ready);

        // epilogue: accumulator row (= weight row) 32*quad + lane, columns = tokens
        const int quad = warp & 3;
        const int r = 32 * quad + lane;
        int gi = 0;
        for (int g = blockIdx.x; g < a.G; g += gridDim.x, ++gi) {
            const int b = gi & 1;
            if (!warp_wait(&acc_full[b], (gi >> 1) & 1, abort)) break;
            fence_after();
            uint32_t v[16];
            tmem_ld16(tmem + ((uint32_t)(32 * quad) << 16) + 16 * b, v);
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
            const int n = 128 * g + r;
            if (a.GS > 1 && rank > 0) {
                if (!mbar_wait<true>(xempty, (gi & 1) ^ 1, abort)) break;
#pragma unroll
                for (int t = 0; t < 16; ++t) st_remote_f32(xbuf + ((rank - 1) * 128 + r) * 16 + t, 0, __uint_as_float(v[t]));
                mbar_arrive_remote(xfull, 0);
            } else {
                float out[16];
#pragma unroll
                for (int t = 0; t < 16; ++t) out[t] = __uint_as_float(v[t]);
                if (a.GS > 1) {
                    if (!mbar_wait<true>(xfull, gi & 1, abort)) break;
                    for (int k = 1; k < a.GS; ++k)
#pragma unroll
                        for (int t = 0; t < 16; ++t) out[t] += xbuf[((k - 1) * 128 + r) * 16 + t];
                    for (int k = 1; k < a.GS; ++k) mbar_arrive_remote(xempty, (uint32_t)k);
                }
                if (n < a.N) {
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        if (t < a.M) {
                            float *dst = a.y + (int64_t)t * a.ld_y + n;
                            *dst = a.accumulate ? *dst + out[t] : out[t];  // a later K pass, same thread
                        }
                }
            }
        }
    }

    fence_before();
    __syncthreads();
    if (a.GS > 1) cg::this_cluster().sync();  // no CTA leaves while a partner may still touch its memory
    if (warp == 1) {
        __syncwarp();
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

struct DecodeShape {
    int GS, ring, ring_bytes, max_mst, grid;
    int bound[9];
    size_t smem;
};

// Boundaries splitting slots [w0, w1) into `parts` ranges of about the same
// packed bytes (a 6/8-bit slot weighs about twice a 4-bit one); every range
// gets at least one slot.
bool split_bytes(const Plan &p, int w0, int w1, int parts, int *bound) {
    if (parts > w1 - w0) return false;
    const int64_t base = slot_offset(p, w0), total = slot_offset(p, w1) - base;
    bound[0] = w0;
    for (int r = 1; r < parts; ++r) {
        int s = bound[r - 1] + 1;
        while (s < w1 - (parts - r) && (slot_offset(p, s) - base) * parts < total * r) ++s;
        bound[r] = s;
    }
    bound[parts] = w1;
    return true;
}

DecodeShape shape_for(const Plan &p, int GS, int64_t G, int sms, int w0, int w1) {
    DecodeShape sh;
    sh.GS = GS;
    sh.ring = 0;
    sh.max_mst = 0;
    sh.smem = 0;
    sh.grid = 1;
    if (!split_bytes(p, w0, w1, GS, sh.bound)) return sh;
    int max_copy = 0;
    for (int r = 0; r < GS; ++r) {
        const int c0 = sh.bound[r], c1 = sh.bound[r + 1];
        const int a4 = std::min(c0, p.n4), e4 = std::min(c1, p.n4), a8 = std::max(c0, p.n4), e8 = std::max(c1, p.n4);
        const int st4 = (std::max(0, e4 - a4) + 3) / 4;
        const int n = st4 + (std::max(0, e8 - a8) + 1) / 2;
        sh.max_mst = std::max(sh.max_mst, n);
        auto rng = [&](int st, int &lo, int &hi) {
            if (st < st4) {
                lo = a4 + 4 * st;
                hi = std::min(e4, lo + 4);
            } else {
                lo = a8 + 2 * (st - st4);
                hi = std::min(e8, lo + 2);
            }
        };
        for (int k = 0; 2 * k < n; ++k) {
            int lo, hi, lo2, hi2;
            rng(2 * k, lo, hi);
            if (2 * k + 1 < n) rng(2 * k + 1, lo2, hi2); else hi2 = hi;
            max_copy = std::max(max_copy, (int)(slot_offset(p, hi2) - slot_offset(p, lo)));
        }
    }
    sh.ring_bytes = (max_copy + 127) / 128 * 128;
    const size_t fixed = 1024 + (size_t)kConv * (kPlaneBytes + 512) + (size_t)sh.max_mst * (kTokBytes + 512) +
                         (size_t)(GS - 1) * 128 * 16 * 4 + 512;
    const size_t budget = 225 * 1024;
    sh.ring = fixed + 2 * (size_t)sh.ring_bytes <= budget
                  ? (int)std::min<size_t>(8, (budget - fixed) / std::max(1, sh.ring_bytes))
                  : 0;
    sh.smem = fixed + (size_t)sh.ring * sh.ring_bytes;
    sh.grid = (int)std::min<int64_t>(G, std::max(1, sms / GS));
    return sh;
}

// Choose the K split: the fewest rounds of 128-row groups per CTA, weighted by
// the K share each CTA streams, among plans that fit shared memory with at
// least two copy stages; ties go to the smaller split.
DecodeShape pick_shape(const Plan &p, int64_t G, int sms, int w0, int w1) {
    DecodeShape best{};
    double best_cost = 1e30;
    for (int GS = 1; GS <= 8 && GS <= w1 - w0; GS *= 2) {
        const DecodeShape sh = shape_for(p, GS, G, sms, w0, w1);
        if (sh.ring < 2) continue;
        const double rounds = (double)((G + sh.grid - 1) / sh.grid);
        const double cost = rounds / GS * (1.0 + 0.02 * GS);  // small charge for the cross-CTA reduction
        if (cost < best_cost - 1e-9) {
            best_cost = cost;
            best = sh;
        }
    }
    return best;
}

int sm_count() {
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

int launch(const Plan &p, DecodeArgs a, int64_t M, int64_t N, cudaStream_t st) {
    if (N > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
    a.M = (int)M;
    a.N = (int)N;
    const WeightOffsets off = weight_offsets(p, N, false);
    a.G = (int)off.G;
    a.GB = off.GB;
    // One launch normally; a K range whose token operand does not fit one
    // cluster's shared memory runs as several passes, each adding into y.
    for (int passes = 1; passes <= 16 && passes <= p.nb; ++passes) {
        int win[17];
        split_bytes(p, 0, p.nb, passes, win);
        DecodeShape plan[16];
        bool ok = true;
        for (int k = 0; k < passes && ok; ++k) {
            plan[k] = pick_shape(p, a.G, sm_count(), win[k], win[k + 1]);
            ok = plan[k].ring >= 2;
        }
        if (!ok) continue;
        for (int k = 0; k < passes; ++k) {
            const DecodeShape &sh = plan[k];
            a.GS = sh.GS;
            for (int i = 0; i < 9; ++i) a.bound[i] = i <= sh.GS ? sh.bound[i] : win[k + 1];
            a.ring = sh.ring;
            a.ring_bytes = sh.ring_bytes;
            a.max_mst = sh.max_mst;
            a.accumulate = k > 0;
            cudaError_t e =
                cudaFuncSetAttribute(gemm_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
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
            e = cudaLaunchKernelEx(&cfg, gemm_decode_kernel, p, a);
            if (e != cudaSuccess) return cuda_fail(e, "gemm_decode_kernel launch");
        }
        return MXS_OK;
    }
    return fail(MXS_ERR_SHAPE, "decode: no shared-memory plan for K=%d", 32 * p.nb);
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
