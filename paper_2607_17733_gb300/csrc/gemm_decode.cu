// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens) on
// the 5th-generation tensor cores.
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale) with the per-block widths of Sec. 4.1.
//
// Decode reads every weight byte once, so the kernel keeps the weights in
// their compact form (4-bit nibbles, 6/8-bit bytes) until they are in
// registers, and does all arithmetic on the tensor core:
//   * the block-scaled FP8 MMA (tcgen05.mma kind::mxf8f6f4, scale_vec::1X)
//     with 128 weight rows as the A operand and the <= 16 tokens as the N = 16
//     B operand; per-block scales are applied by the hardware and the sum over
//     K stays in fp32 tensor-memory accumulators;
//   * a weight code of magnitude <= 15 is fed as the e4m3 byte
//     (sign << 7) | |m|, whose value is |m| * 2^-9 (subnormals and the first
//     binade); 6/8-bit codes split as |m| = 16h + l into two such digits
//     (Sec. 6: high- and low-precision parts multiplied separately).  The
//     fixed-point weight of each digit goes into the E8M0 scale byte (+7 for
//     a 4-bit code, +9/+5 for the high/low digit of a 6-bit code, +7/+3 for
//     an 8-bit one), so every MMA term is exact;
//   * the token operand is the activations' MMA-plane form (the layout the
//     prefill GEMM reads: e4m3 values m/4, or a high and a low digit, under
//     the block's own scale byte).  It is either loaded by TMA from planes
//     written by mxs_quantize_act -- the launch may then overlap the kernel
//     before it (programmatic dependent launch) -- or built in the prologue
//     from packed codes.
// Work: a CTA owns 128-row weight groups and (in a cluster) a K range of them,
// cut into MMA stages of 128 K'-bytes (four 4-bit slots or two 6/8-bit
// slots).  Up to ten worker warps own whole stages, round robin: a worker
// loads its stage's codes straight from HBM into registers (coalesced 16-byte
// loads, the next stage in flight while it converts the current one), writes
// the e4m3 digits into its own 128-byte-swizzled plane buffer and the weight
// scale tile, and issues the stage's MMAs into its own accumulator.  Workers
// never wait for one another; the epilogue warps add the workers' partial
// accumulators in worker order (a fixed order: results are deterministic).
// Other warps: warp 0 owns tensor memory and loads the token operand; warps
// 1-4 run the epilogue (and build the token operand from codes).
// K is split over the CTAs of a thread-block cluster when N alone cannot
// occupy the GPU.  The ranks then reduce-scatter through distributed shared
// memory: rank k receives rows [k*R, (k+1)*R) (R = 128/cluster size) of every
// other rank's partial tile by bulk copy, adds the partials in rank order and
// stores those rows.  A K range whose token operand does not fit shared
// memory runs as several passes, each adding into y.
// Every mbarrier wait is bounded; on expiry the kernel records
// MXS_ERR_TIMEOUT, stops, drains what it issued and frees tensor memory.
// Weight scale bytes above 245 (|w| >= 2^118) saturate at 254 after the digit
// shift.
#include <algorithm>
#include <cstring>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {

__device__ int g_decode_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

constexpr int kMaxWorkers = 10;                                 // worker warps per CTA, chosen per launch
constexpr int kWorkerWarp0 = 5;                                 // warps 5..
constexpr int kMaxThreads = (kWorkerWarp0 + kMaxWorkers) * 32;  // 480
constexpr int kPlaneBytes = 128 * 128;  // 128 rows x 128 bytes of K' (SW128)
constexpr int kTokBytes = 16 * 128;     // 16 token rows x 128 bytes of K'
constexpr int kAccCols = 16;            // one accumulator: 16 token columns
constexpr int kSfaCol = 2 * kMaxWorkers * kAccCols;  // 320: 4 columns of weight scales per worker
constexpr int kSfbCol = kSfaCol + 4 * kMaxWorkers;   // 360: 4 columns per MMA stage of token scales
constexpr int kTmemCols = 512;
constexpr int kMaxStages = (kTmemCols - kSfbCol) / 4;  // 38
constexpr int kXBytes = 128 * 16 * 4;  // one fp32 partial tile
constexpr int kMinSmem = 116 * 1024;   // one CTA per SM (each allocates all of tensor memory)
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock

struct DecodeArgs {
    const uint8_t *codes;   // [M, row_bytes] packed activation codes (codes mode)
    const uint8_t *scales;  // [M, nb]
    const uint8_t *tok_sf;  // activation scale tiles of the planes buffer (planes mode), else NULL
    const uint8_t *w;       // packed weight buffer
    float *y;
    int64_t ld_y;
    int M, N, G;      // tokens, output features, 128-row groups
    int GS;           // CTAs per cluster along K
    int bound[9];     // rank r owns slots [bound[r], bound[r+1]) (stage-aligned)
    int max_mst;      // most MMA stages any rank holds (token operand carve)
    int workers;      // worker warps (blockDim = (5 + workers) warps)
    int accumulate;   // add into y (a later K pass) instead of storing
    int64_t GB;       // bytes of one 128-row weight group
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
__device__ __forceinline__ uint32_t map_rank(const void *p, uint32_t rank) {
    uint32_t ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(su32(p)), "r"(rank));
    return ra;
}
__device__ __forceinline__ void mbar_arrive_remote(uint64_t *bar, uint32_t rank) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(map_rank(bar, rank))
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
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
            su32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(su32(bar)), "r"(x), "r"(y)
        : "memory");
}
// own shared memory -> another rank's shared memory (cluster address), the
// bytes completing on that rank's barrier (cluster address); the copy is
// known to be done (source read included) only through that barrier
__device__ __forceinline__ void bulk_to_rank(uint32_t dst_cluster, const void *src, uint32_t bytes,
                                             uint32_t bar_cluster) {
    asm volatile(
        "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            dst_cluster),
        "r"(su32(src)), "r"(bytes), "r"(bar_cluster)
        : "memory");
}
// streaming loads of weight codes: read once, not kept in L1
__device__ __forceinline__ uint4 ld_stream16(const uint8_t *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ uint32_t ld_stream1(const uint8_t *p) {
    uint16_t v;
    asm volatile("ld.global.nc.L1::no_allocate.u8 %0, [%1];" : "=h"(v) : "l"(p));
    return v;
}
// generic-proxy shared-memory writes -> visible to the tensor core / bulk copies
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire;" ::: "memory"); }

// UMMA shared-memory descriptors (as in the prefill kernel): 128B-swizzled
// K-major operand tiles (8-row atoms of 1024 B) and 32 x 16 B scale tiles.
// A byte offset d (all of shared memory is below 256 KB) moves the
// descriptor by d >> 4.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t desc_sf(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)(128 >> 4) << 32) | ((uint64_t)1 << 46);
}
// kind::mxf8f6f4, e4m3 x e4m3, K-major, N = 16, UE8M0 scales, M = 128
constexpr uint32_t kIdesc = ((uint32_t)(16 >> 3) << 17) | (1u << 23) | ((uint32_t)(128 >> 4) << 24);
__device__ __forceinline__ constexpr uint32_t idesc(int sfa_id, int sfb_id) {
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

// e4m3 digit bytes (sign << 7) | |m| of the four low / four high
// sign-magnitude nibbles (s << 3) | |m| held in a word
__device__ __forceinline__ uint32_t lo_nib(uint32_t w) { return (w & 0x07070707u) | ((w << 4) & 0x80808080u); }
__device__ __forceinline__ uint32_t hi_nib(uint32_t w) { return ((w >> 4) & 0x07070707u) | (w & 0x80808080u); }
// high (|m| >> 4) and low (|m| & 15) digit of four sign-magnitude 8-bit codes
__device__ __forceinline__ uint32_t hi_digit(uint32_t x) { return ((x >> 4) & 0x07070707u) | (x & 0x80808080u); }
__device__ __forceinline__ uint32_t lo_digit(uint32_t x) { return x & 0x8F8F8F8Fu; }
// scale byte carrying the digit's fixed-point weight; 255 (NaN) stays
__device__ __forceinline__ uint32_t shifted(uint32_t S, uint32_t sh) { return S == 255 ? 255u : min(S + sh, 254u); }

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

// One half of a worker's stage in registers: lane l holds rows l + 32i
// (i < 4).  A 4-bit half is slots 2h, 2h+1 (v[4k+i] = slot 2h+k, row i); a
// 6/8-bit half is slot h (v[2i], v[2i+1] = the two 16-byte words of row i).
// Either way the half fills 16-byte chunks 4h..4h+3 of each row and
// scale-tile bytes 2h, 2h+1.
struct Half {
    uint4 v[8];
    uint32_t s[8];  // scale bytes (4-bit: [4k+i] = slot 2h+k, row i; 6/8-bit: [i] = row i)
};

// Load half `h` of stage `st` of the weight group at `wg` (lane l: rows l + 32i).
__device__ __forceinline__ void load_half(const Plan &p, const Stages &S, const uint8_t *wg, int st, int h, int l,
                                          Half &x) {
    int lo, hi;
    S.range(st, lo, hi);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        x.v[i] = make_uint4(0, 0, 0, 0);
        x.s[i] = 0;
    }
    if (st < S.st4) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int q = 2 * h + k;
            if (lo + q < hi) {  // a partial last stage has fewer slots
                const uint8_t *slot = wg + slot_offset(p, lo + q);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    x.v[4 * k + i] = ld_stream16(slot + 16 * (l + 32 * i));
                    x.s[4 * k + i] = ld_stream1(slot + 2048 + l + 32 * i);
                }
            }
        }
    } else if (lo + h < hi) {
        const uint8_t *slot = wg + slot_offset(p, lo + h);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x.v[2 * i] = ld_stream16(slot + 32 * (l + 32 * i));
            x.v[2 * i + 1] = ld_stream16(slot + 32 * (l + 32 * i) + 16);
            x.s[i] = ld_stream1(slot + 4096 + l + 32 * i);
        }
    }
}

// Convert a loaded half into digit-plane chunks 4h..4h+3 of rows l + 32i and
// return the row's scale-tile bytes 2h, 2h+1 (bits 16i..16i+15 for row i).
__device__ __forceinline__ uint64_t store_half(const Plan &p, const Stages &S, int st, int h, int l, const Half &x,
                                               uint8_t *pl) {
    int lo, hi;
    S.range(st, lo, hi);
    uint64_t sf = 0;
    if (st < S.st4) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int q = 2 * h + k;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = l + 32 * i;
                const uint4 v = x.v[4 * k + i];
                // word j: bytes hold elements 8j..8j+3 (low nibbles), 8j+4..8j+7 (high nibbles)
                *reinterpret_cast<uint4 *>(pl + sw128(r, 2 * q)) =
                    make_uint4(lo_nib(v.x), hi_nib(v.x), lo_nib(v.y), hi_nib(v.y));
                *reinterpret_cast<uint4 *>(pl + sw128(r, 2 * q + 1)) =
                    make_uint4(lo_nib(v.z), hi_nib(v.z), lo_nib(v.w), hi_nib(v.w));
                // absent slots hold zero codes under scale byte 0 (a zero term)
                sf |= (uint64_t)(lo + q < hi ? shifted(x.s[4 * k + i], 7) : 0u) << (16 * i + 8 * k);
            }
        }
    } else {
        const bool six = lo + h < hi && slot_width(p, lo + h) == 6;
        const uint32_t sh_hi = six ? 9 : 7, sh_lo = six ? 5 : 3;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int r = l + 32 * i;
            const uint4 v0 = x.v[2 * i], v1 = x.v[2 * i + 1];
            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * h)) =
                make_uint4(hi_digit(v0.x), hi_digit(v0.y), hi_digit(v0.z), hi_digit(v0.w));
            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * h + 1)) =
                make_uint4(hi_digit(v1.x), hi_digit(v1.y), hi_digit(v1.z), hi_digit(v1.w));
            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * h + 2)) =
                make_uint4(lo_digit(v0.x), lo_digit(v0.y), lo_digit(v0.z), lo_digit(v0.w));
            *reinterpret_cast<uint4 *>(pl + sw128(r, 4 * h + 3)) =
                make_uint4(lo_digit(v1.x), lo_digit(v1.y), lo_digit(v1.z), lo_digit(v1.w));
            const uint32_t b2 = lo + h < hi ? (shifted(x.s[i], sh_hi) | (shifted(x.s[i], sh_lo) << 8)) : 0u;
            sf |= (uint64_t)b2 << (16 * i);
        }
    }
    return sf;
}

__global__ void __launch_bounds__(kMaxThreads, 1) gemm_decode_kernel(const __grid_constant__ Plan p,
                                                                     const __grid_constant__ DecodeArgs a,
                                                                     const __grid_constant__ CUtensorMap tok_map) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sbase = su32(smem_raw);
    uint8_t *smem = smem_raw + (((sbase + 1023) & ~1023u) - sbase);  // 1024-aligned for the swizzled tiles
    const int W = a.workers;
    uint8_t *planes = smem;                              // W x 16 KB
    uint8_t *tok = planes + W * kPlaneBytes;             // max_mst x 2 KB
    uint8_t *sfa = tok + (size_t)a.max_mst * kTokBytes;  // W x 512
    uint8_t *sfb = sfa + W * 512;                        // max_mst x 512
    // cluster reduce-scatter: rank k adds up rows [k*R, (k+1)*R) of the GS partial
    // tiles (R = 128/GS) and stores them; xout is this rank's whole partial tile,
    // xbuf the slices the other ranks send here (slot of sender j: j, or j-1 past k)
    const int R = 128 / a.GS;
    float *xout = reinterpret_cast<float *>(sfb + (size_t)a.max_mst * 512);  // [128][16] (GS > 1)
    float *xbuf = xout + (a.GS > 1 ? 128 * 16 : 0);                          // [GS-1][R][16]
    uint64_t *bars = reinterpret_cast<uint64_t *>(xbuf + (size_t)(a.GS - 1) * R * 16);
    uint64_t *plane_free = bars;  // [W] tcgen05.commit
    uint64_t *acc_full = plane_free + W, *acc_empty = acc_full + 2;
    uint64_t *tok_full = acc_empty + 2, *tok_ready = tok_full + 1;
    uint64_t *xfull = tok_ready + 1, *xempty = xfull + 1, *xstage = xempty + 1, *xread = xstage + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(xread + 1);
    int *abort_flag = reinterpret_cast<int *>(tmem_slot + 1);
    volatile int *abort = abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = a.GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = a.bound[rank], c1 = a.bound[rank + 1];
    const bool from_planes = a.tok_sf != nullptr;
    Stages S;
    S.init(p, c0, c1);
    const int nw = min(W, S.n);  // workers with a stage in every group
    const uint32_t xslice = (uint32_t)(R * 16 * 4);

    // Workers put their first stage's loads in flight before anything else:
    // the weights are static (see mxs_linear_decode), so they need no wait.
    Half A, B;
    if (warp >= kWorkerWarp0 && warp - kWorkerWarp0 < nw && (int)blockIdx.x < a.G) {
        const uint8_t *wg = a.w + (int64_t)blockIdx.x * a.GB;
        load_half(p, S, wg, warp - kWorkerWarp0, 0, lane, A);
        load_half(p, S, wg, warp - kWorkerWarp0, 1, lane, B);
    }

    // the next kernel on the stream may launch now (it waits for this grid
    // before it touches what this grid writes)
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (threadIdx.x == 0) {
        for (int i = 0; i < W; ++i) mbar_init(&plane_free[i], 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], nw);  // each active worker commits once per group
            mbar_init(&acc_empty[i], 4);  // the four epilogue warps
        }
        mbar_init(tok_full, from_planes ? 1 : 4);
        mbar_init(tok_ready, 1);              // tcgen05.commit once the token scales are in tensor memory
        mbar_init(xfull, 1);                  // armed per tile with the bytes of GS-1 slices
        mbar_init(xempty, max(1, a.GS - 1));  // every receiver took this rank's previous slices (copies done)
        mbar_init(xstage, 4);                 // the four epilogue warps have staged the partial tile
        mbar_init(xread, 4);                  // the four epilogue warps are done with xout and xbuf
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (a.GS > 1) mbar_expect_tx(xfull, (uint32_t)(a.GS - 1) * xslice);  // the first tile's slices
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    // Partners' barriers must exist before any remote access: every thread
    // arrives now; the epilogue warps (the only ones with remote traffic) wait
    // before their first remote operation, the others just before the teardown.
    if (a.GS > 1) cluster_arrive();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ token operand -> smem, scales -> TMEM
        if (lane == 0) {
            if (from_planes) {
                // the planes may come from the kernel just before this one (programmatic
                // dependent launch): wait for it before the first read
                asm volatile("griddepcontrol.wait;" ::: "memory");
                const int sg0 = c0 < p.n4 ? c0 / 4 : p.st4 + (c0 - p.n4) / 2;
                mbar_expect_tx(tok_full, (uint32_t)S.n * (kTokBytes + 512));
                for (int st = 0; st < S.n; ++st)
                    tma_load_2d(tok + st * kTokBytes, &tok_map, tok_full, 128 * (sg0 + st), 0);
                bulk_load(sfb, a.tok_sf + (int64_t)sg0 * 512, (uint32_t)S.n * 512, tok_full);
            }
            if (mbar_wait(tok_full, 0, abort)) {
                fence_after();
                const uint64_t dsfb = desc_sf(su32(sfb));
                for (int st = 0; st < S.n; ++st) tmem_cp_sf(tmem + kSfbCol + 4 * st, dsfb + 32 * st);
                mma_commit(tok_ready);
                drain_wait(tok_ready, 0);
            }
        }
    } else if (warp >= kWorkerWarp0) {
        // ------------------------------------------------------------ workers
        const int w = warp - kWorkerWarp0;
        if (w < nw) {
            uint8_t *pl = planes + w * kPlaneBytes;
            uint8_t *sfa_cell = sfa + w * 512 + 16 * lane;  // rows lane + 32i: bytes 4i..4i+3
            const uint64_t dA = desc_sw128(su32(pl)), dB = desc_sw128(su32(tok));
            const uint64_t dsfa = desc_sf(su32(sfa + w * 512));
            const uint32_t sfa_t = tmem + kSfaCol + 4 * w;
            bool ok = warp_wait(tok_ready, 0, abort);
            if (ok) fence_after();
            uint32_t qw = 0;  // stages this worker has issued (plane_free phases)
            int g = blockIdx.x, st = w, gi = 0;
            bool first_in_group = true;
            while (ok && g < a.G) {
                const int b = gi & 1;
                if (first_in_group) ok = warp_wait(&acc_empty[b], ((gi >> 1) & 1) ^ 1, abort);
                // the plane buffer is free once this worker's previous MMAs have read it
                if (ok && qw > 0) ok = warp_wait(&plane_free[w], (qw - 1) & 1, abort);
                if (!ok) break;
                // next stage of this worker: st + W, else its first stage of the next group
                int g2 = g, st2 = st + W;
                if (st2 >= S.n) {
                    g2 = g + gridDim.x;
                    st2 = w;
                }
                const uint8_t *wg2 = a.w + (int64_t)(g2 < a.G ? g2 : g) * a.GB;
                const uint64_t sf0 = store_half(p, S, st, 0, lane, A, pl);
                if (g2 < a.G) load_half(p, S, wg2, st2, 0, lane, A);
                const uint64_t sf1 = store_half(p, S, st, 1, lane, B, pl);
                if (g2 < a.G) load_half(p, S, wg2, st2, 1, lane, B);
                // scale tile: the lane's 16 bytes are rows lane + 32i, 4 bytes each
                // (sf ids 0, 1 from half 0 and 2, 3 from half 1)
                uint32_t cell[4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    cell[i] = (uint32_t)((sf0 >> (16 * i)) & 0xFFFF) | ((uint32_t)((sf1 >> (16 * i)) & 0xFFFF) << 16);
                *reinterpret_cast<uint4 *>(sfa_cell) = make_uint4(cell[0], cell[1], cell[2], cell[3]);
                fence_async_smem();
                __syncwarp();
                if (lane == 0) {
                    fence_after();
                    tmem_cp_sf(sfa_t, dsfa);
                    const uint32_t acc = tmem + kAccCols * (kMaxWorkers * b + w);
                    const uint32_t sfb_t = tmem + kSfbCol + 4 * st;
                    const uint64_t db = dB + (uint64_t)(st * (kTokBytes >> 4));
                    const uint32_t accum = first_in_group ? 0u : 1u;
                    if (st < S.st4) {
                        // slot q: weight digits at K' bytes 32q.., token values at 32q..
                        mma_mx(acc, dA, db, idesc(0, 0), sfa_t, sfb_t, accum);
                        mma_mx(acc, dA + 2, db + 2, idesc(1, 1), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 4, db + 4, idesc(2, 2), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 6, db + 6, idesc(3, 3), sfa_t, sfb_t, 1u);
                    } else {
                        // slot j: weight digit pa (high, low) at 64j + 32pa under scale 2j + pa;
                        // token digit pb at 64j + 32pb under the slot's scale byte j
                        mma_mx(acc, dA, db, idesc(0, 0), sfa_t, sfb_t, accum);
                        mma_mx(acc, dA, db + 2, idesc(0, 0), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 2, db, idesc(1, 0), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 2, db + 2, idesc(1, 0), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 4, db + 4, idesc(2, 1), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 4, db + 6, idesc(2, 1), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 6, db + 4, idesc(3, 1), sfa_t, sfb_t, 1u);
                        mma_mx(acc, dA + 6, db + 6, idesc(3, 1), sfa_t, sfb_t, 1u);
                    }
                    mma_commit(&plane_free[w]);  // planes + scale tile free once these MMAs have read them
                    if (g2 != g) mma_commit(&acc_full[b]);  // this worker's share of the group is issued
                }
                __syncwarp();
                ++qw;
                first_in_group = g2 != g;
                if (g2 != g) ++gi;
                g = g2;
                st = st2;
            }
            if (lane == 0 && qw > 0) drain_wait(&plane_free[w], (qw - 1) & 1);
        }
    } else {
        // ------------------------------------------------------------ warps 1-4: token operand (codes), epilogue
        const int et = threadIdx.x - 32;  // 0..127
        if (!from_planes) {
            // the codes may come from the kernel just before this one
            asm volatile("griddepcontrol.wait;" ::: "memory");
            // zero the token planes and scale tiles of every stage, then fill them from the codes
            for (int i = et; i < S.n * (kTokBytes + 512) / 16; i += 128) {
                const int off = i * 16;
                uint8_t *dst = off < S.n * kTokBytes ? tok + off : sfb + (off - S.n * kTokBytes);
                *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
            }
            named_sync(1, 128);
            for (int it = et; it < (c1 - c0) * a.M; it += 128) {
                const int s = c0 + it / a.M, t = it % a.M;
                const int b = slot_width(p, s);
                const uint8_t *row = a.codes + (int64_t)t * p.row_bytes;
                const uint32_t Sa = a.scales[(int64_t)t * p.nb + s];
                int m[32];
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
                // the plane form of the prefill layout: m/4 (4-bit), or a high digit
                // floor(m / 2^sh) and a low digit m mod 2^sh, scaled so that they sum
                // to m * 2^-(b-2) (6/8-bit)
                uint32_t d0[8], d1[8];
                const int sh = b == 6 ? 3 : 4;
                const float fh = b == 6 ? 0.5f : 0.25f, fl = b == 6 ? 0.0625f : 0.015625f;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (b == 4) {
                        d0[i] = e4m3x2(0.25f * m[4 * i], 0.25f * m[4 * i + 1]) |
                                ((uint32_t)e4m3x2(0.25f * m[4 * i + 2], 0.25f * m[4 * i + 3]) << 16);
                        d1[i] = 0;
                    } else {
                        int hd[4], ld[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            hd[k] = m[4 * i + k] >> sh;
                            ld[k] = m[4 * i + k] & ((1 << sh) - 1);
                        }
                        d0[i] = e4m3x2(fh * hd[0], fh * hd[1]) | ((uint32_t)e4m3x2(fh * hd[2], fh * hd[3]) << 16);
                        d1[i] = e4m3x2(fl * ld[0], fl * ld[1]) | ((uint32_t)e4m3x2(fl * ld[2], fl * ld[3]) << 16);
                    }
                }
                int st, pos, sfid;
                if (s < p.n4) {
                    st = (s - S.a4) / 4;
                    sfid = (s - S.a4) % 4;
                    pos = 32 * sfid;
                } else {
                    st = S.st4 + (s - S.a8) / 2;
                    sfid = (s - S.a8) % 2;
                    pos = 64 * sfid;
                }
                uint8_t *trow = tok + st * kTokBytes;
                const int c = pos / 16;  // first 16-byte chunk
                *reinterpret_cast<uint4 *>(trow + sw128(t, c)) = make_uint4(d0[0], d0[1], d0[2], d0[3]);
                *reinterpret_cast<uint4 *>(trow + sw128(t, c + 1)) = make_uint4(d0[4], d0[5], d0[6], d0[7]);
                if (b != 4) {
                    *reinterpret_cast<uint4 *>(trow + sw128(t, c + 2)) = make_uint4(d1[0], d1[1], d1[2], d1[3]);
                    *reinterpret_cast<uint4 *>(trow + sw128(t, c + 3)) = make_uint4(d1[4], d1[5], d1[6], d1[7]);
                }
                sfb[st * 512 + (t & 31) * 16 + (t >> 5) * 4 + sfid] = (uint8_t)Sa;
            }
            fence_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(tok_full);
        }

        // epilogue: accumulator row (= weight row) 32*quad + lane, columns = tokens;
        // the workers' partial sums are added in worker order
        if (a.GS > 1) cluster_wait();
        const int quad = warp & 3;
        const int r = 32 * quad + lane;
        int gi = 0;
        for (int g = blockIdx.x; g < a.G; g += gridDim.x, ++gi) {
            const int b = gi & 1;
            if (!warp_wait(&acc_full[b], (gi >> 1) & 1, abort)) break;
            fence_after();
            float out[16];
            for (int w = 0; w < nw; ++w) {
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(32 * quad) << 16) + kAccCols * (kMaxWorkers * b + w), v);
#pragma unroll
                for (int t = 0; t < 16; ++t) out[t] = w == 0 ? __uint_as_float(v[t]) : out[t] + __uint_as_float(v[t]);
            }
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
            const bool more = g + (int)gridDim.x < a.G;  // another group follows
            if (a.GS == 1) {
                const int n = 128 * g + r;
                if (n < a.N) {
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        if (t < a.M) {
                            float *dst = a.y + (int64_t)t * a.ld_y + n;
                            *dst = a.accumulate ? *dst + out[t] : out[t];  // a later K pass, same thread
                        }
                }
                continue;
            }
            // stage the partial tile once this CTA is done with the previous one and
            // every receiver took the previous slices (which also means those copies
            // have finished reading xout)
            if (!warp_wait(xread, (gi & 1) ^ 1, abort)) break;
            if (!warp_wait<true>(xempty, (gi & 1) ^ 1, abort)) break;
            float4 *dst = reinterpret_cast<float4 *>(xout + r * 16);
#pragma unroll
            for (int i = 0; i < 4; ++i) dst[i] = make_float4(out[4 * i], out[4 * i + 1], out[4 * i + 2], out[4 * i + 3]);
            fence_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(xstage);
            bool sent = true;
            if (et == 0) {
                sent = mbar_wait(xstage, gi & 1, abort);  // all four warps staged
                if (sent)
                    for (int k = 0; k < a.GS; ++k) {
                        if (k == (int)rank) continue;
                        const int slot = (int)rank < k ? (int)rank : (int)rank - 1;  // this rank's slot at k
                        bulk_to_rank(map_rank(xbuf + slot * R * 16, (uint32_t)k), xout + k * R * 16, xslice,
                                     map_rank(xfull, (uint32_t)k));
                    }
            }
            if (!__shfl_sync(0xffffffffu, sent, 0)) break;  // whole warp
            // the other ranks' slices of this rank's rows arrived by bulk copy
            if (!warp_wait(xfull, gi & 1, abort)) break;
            const int lr = r - (int)rank * R;  // row within this rank's slice
            if (lr >= 0 && lr < R) {
                float sum[16];
                for (int j = 0; j < a.GS; ++j) {  // rank order
                    const float *src = j == (int)rank ? xout + r * 16 : xbuf + ((j < (int)rank ? j : j - 1) * R + lr) * 16;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float4 u = reinterpret_cast<const float4 *>(src)[i];
                        sum[4 * i] = j == 0 ? u.x : sum[4 * i] + u.x;
                        sum[4 * i + 1] = j == 0 ? u.y : sum[4 * i + 1] + u.y;
                        sum[4 * i + 2] = j == 0 ? u.z : sum[4 * i + 2] + u.z;
                        sum[4 * i + 3] = j == 0 ? u.w : sum[4 * i + 3] + u.w;
                    }
                }
                const int n = 128 * g + r;
                if (n < a.N) {
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        if (t < a.M) {
                            float *yd = a.y + (int64_t)t * a.ld_y + n;
                            *yd = a.accumulate ? *yd + sum[t] : sum[t];  // a later K pass, same thread
                        }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(xread);
            if (more) {
                // re-arm the receive barrier, then tell every sender its slot here is free
                bool freed = true;
                if (et == 0) {
                    freed = mbar_wait(xread, gi & 1, abort);
                    if (freed) {
                        mbar_expect_tx(xfull, (uint32_t)(a.GS - 1) * xslice);
                        for (int k = 0; k < a.GS; ++k)
                            if (k != (int)rank) mbar_arrive_remote(xempty, (uint32_t)k);
                    }
                }
                if (!__shfl_sync(0xffffffffu, freed, 0)) break;  // whole warp
            }
        }
    }

    // No CTA leaves while a partner may still copy into or out of its memory:
    // every thread arrives once its own cluster traffic is done and waits only
    // before the CTA's exit.
    if (a.GS > 1 && !(warp >= 1 && warp < kWorkerWarp0)) cluster_wait();  // (the set-up phase)
    if (a.GS > 1) cluster_arrive();
    fence_before();
    __syncthreads();
    if (a.GS > 1) cluster_wait();
    if (warp == 0) {
        __syncwarp();
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

// ------------------------------------------------------------------ host side
// MMA stage sg of the plane layout covers slots [stage_lo(sg), stage_lo(sg+1)).
int stage_lo(const Plan &p, int sg) {
    return sg <= p.st4 ? std::min(4 * sg, p.n4) : std::min(p.n4 + 2 * (sg - p.st4), p.nb);
}

struct DecodeShape {
    int GS, max_mst, grid, workers;
    int bound[9];  // slots
    size_t smem;
    bool ok;
};

// Stage boundaries splitting stages [g0, g1) into `parts` ranges of about
// the same packed bytes (a 6/8-bit slot weighs about twice a 4-bit one);
// every range gets at least one stage.
bool split_stages(const Plan &p, int g0, int g1, int parts, int *gb) {
    if (parts > g1 - g0) return false;
    const int64_t base = slot_offset(p, stage_lo(p, g0)), total = slot_offset(p, stage_lo(p, g1)) - base;
    gb[0] = g0;
    for (int r = 1; r < parts; ++r) {
        int s = gb[r - 1] + 1;
        while (s < g1 - (parts - r) && (slot_offset(p, stage_lo(p, s)) - base) * parts < total * r) ++s;
        gb[r] = s;
    }
    gb[parts] = g1;
    return true;
}

size_t smem_bytes(int GS, int max_mst, int workers) {
    // partial tile + (GS-1) received slices of 128/GS rows
    const size_t xbytes = GS > 1 ? (size_t)kXBytes + (size_t)(GS - 1) * (kXBytes / GS) : 0;
    return 1024 + (size_t)workers * (kPlaneBytes + 512) + (size_t)max_mst * (kTokBytes + 512) + xbytes + 512;
}

DecodeShape shape_for(const Plan &p, int GS, int64_t G, int sms, int g0, int g1) {
    DecodeShape sh = {};
    sh.GS = GS;
    int gb[9];
    if (!split_stages(p, g0, g1, GS, gb)) return sh;
    for (int r = 0; r <= GS; ++r) sh.bound[r] = stage_lo(p, gb[r]);
    for (int r = 0; r < GS; ++r) sh.max_mst = std::max(sh.max_mst, gb[r + 1] - gb[r]);
    // as many workers as fit, up to one per stage
    sh.workers = std::min(kMaxWorkers, sh.max_mst);
    while (sh.workers > 1 && smem_bytes(GS, sh.max_mst, sh.workers) > 225 * 1024) --sh.workers;
    sh.smem = std::max<size_t>(kMinSmem, smem_bytes(GS, sh.max_mst, sh.workers));
    sh.ok = sh.max_mst <= kMaxStages && sh.smem <= 225 * 1024 && sh.workers >= std::min(4, sh.max_mst);
    sh.grid = (int)std::min<int64_t>(G, std::max(1, sms / GS));
    return sh;
}

// Choose the K split.  A CTA's time is about (groups it owns) x (stages a
// worker owns per group + a fixed cost per group), in units of one worker
// stage (~2.5 us, the latency of its loads).  In a cluster every group after
// the first also waits for the previous group's cross-rank exchange, which
// measured at 8-13 us on GB300 (q/gate/down projections of an 8B model, each
// cluster size forced in turn), so clusters pay off only when their CTAs own
// one group each.  Ties go to the smaller cluster.
DecodeShape pick_shape(const Plan &p, int64_t G, int sms, int g0, int g1) {
    DecodeShape best = {};
    double best_cost = 1e30;
    for (int GS = 1; GS <= 8 && GS <= g1 - g0; GS *= 2) {
        const DecodeShape sh = shape_for(p, GS, G, sms, g0, g1);
        if (!sh.ok) continue;
        const double rounds = (double)((G + sh.grid - 1) / sh.grid);
        const double cost = rounds * ((sh.max_mst + sh.workers - 1) / sh.workers + 1.0) +
                            (GS > 1 ? 0.3 + 8.0 * (rounds - 1.0) : 0.0);
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

}  // namespace

int64_t decode_workspace_bytes(const Plan &, int64_t, int64_t) { return 0; }

int launch_gemm_decode(const Plan &p, const void *codes, const uint8_t *scales, const void *act_planes,
                       const void *packed, int64_t M, int64_t N, float *y, int64_t ld_y, bool pdl, cudaStream_t st) {
    if (N > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
    DecodeArgs a = {};
    a.codes = static_cast<const uint8_t *>(codes);
    a.scales = scales;
    a.w = static_cast<const uint8_t *>(packed);
    a.y = y;
    a.ld_y = ld_y;
    a.M = (int)M;
    a.N = (int)N;
    const WeightOffsets off = weight_offsets(p, N, false);
    a.G = (int)off.G;
    a.GB = off.GB;
    CUtensorMap map;
    std::memset(&map, 0, sizeof(map));
    if (act_planes) {
        const int rc = make_plane_map(&map, act_planes, M, p.kp, 16);
        if (rc) return rc;
        a.tok_sf = static_cast<const uint8_t *>(act_planes) + align256(M * p.kp);
    }
    // One launch normally; a K range whose token operand does not fit one
    // cluster's shared memory runs as several passes, each adding into y.
    for (int passes = 1; passes <= 16 && passes <= p.nst; ++passes) {
        int win[17];
        split_stages(p, 0, p.nst, passes, win);
        DecodeShape plan[16];
        bool ok = true;
        for (int k = 0; k < passes && ok; ++k) {
            plan[k] = pick_shape(p, a.G, sm_count(), win[k], win[k + 1]);
            ok = plan[k].ok;
        }
        if (!ok) continue;
        for (int k = 0; k < passes; ++k) {
            const DecodeShape &sh = plan[k];
            a.GS = sh.GS;
            for (int i = 0; i < 9; ++i) a.bound[i] = i <= sh.GS ? sh.bound[i] : sh.bound[sh.GS];
            a.max_mst = sh.max_mst;
            a.workers = sh.workers;
            a.accumulate = k > 0;
            cudaError_t e =
                cudaFuncSetAttribute(gemm_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3((unsigned)sh.grid, (unsigned)sh.GS, 1);
            cfg.blockDim = dim3((unsigned)((kWorkerWarp0 + sh.workers) * 32), 1, 1);
            cfg.dynamicSmemBytes = sh.smem;
            cfg.stream = st;
            cudaLaunchAttribute attr[2];
            int na = 0;
            attr[na].id = cudaLaunchAttributeClusterDimension;
            attr[na].val.clusterDim.x = 1;
            attr[na].val.clusterDim.y = (unsigned)sh.GS;
            attr[na].val.clusterDim.z = 1;
            ++na;
            if (pdl && k == 0) {
                attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
                attr[na].val.programmaticStreamSerializationAllowed = 1;
                ++na;
            }
            cfg.attrs = attr;
            cfg.numAttrs = na;
            e = cudaLaunchKernelEx(&cfg, gemm_decode_kernel, p, a, map);
            if (e != cudaSuccess) return cuda_fail(e, "gemm_decode_kernel launch");
        }
        return MXS_OK;
    }
    return fail(MXS_ERR_SHAPE, "decode: no shared-memory plan for K=%d", 32 * p.nb);
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
