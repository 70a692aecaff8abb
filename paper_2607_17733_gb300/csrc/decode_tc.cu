// decode_tc.cu -- A4 for decode shapes of 2..16 tokens: the MXINT GEMM on the
// 5th-generation tensor cores over the activations' MMA planes.
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 with the per-block
// widths of Sec. 4.1.  The activations were quantized on the fly by
// mxs_quantize_act's kernel into their MMA planes (Appendix A.2); this kernel
// is that quantizer's programmatic dependent.
//
// Operand forms (the conventions of the planes and of gemm_decode.cu):
//   * a 4-bit block runs on the block-scaled FP8 MMA (kind::mxf8f6f4,
//     scale_vec::1X, K = 32): its weight code (s << 3) | m is fed as the e4m3
//     byte (s << 7) | m, worth m * 2^-9, with the weight scale byte raised by 7
//     (saturating) in the A scale tile; the token operand is the plane's e4m3
//     m/4 under the block's own scale byte;
//   * a 6/8-bit block runs on the bf16 MMA (kind::f16, two K = 16 MMAs): its
//     codes become the exact bf16 values m * 2^(Sw-127-(b-2)), the token plane
//     holds the activations' bf16 values the same way; every term is exact.
//
// Why a second tensor-core decode kernel.  gemm_decode.cu hands the tensor
// core one 128-byte K' stage (four 4-bit or two 6/8-bit slots) at a time from
// each of four converter quads, and that per-stage hand-off (converters ->
// MMA issuer -> tensor core -> converters) bounds it; the MMAs themselves
// cost ~50 cycles each at N = 16 (measured), a quarter of its time.  Here one
// stage is four plane stages (sixteen 4-bit or eight 6/8-bit slots, ~34 KB of
// weights): all sixteen converter warps fill one 128-column A tile in tensor
// memory, one thread issues its MMAs, and the hand-offs drop fourfold.
//
// Work split (as in gemv_decode.cu): each CTA streams an equal share of a
// problem's weight bytes, cut at plane-stage boundaries; row groups its range
// covers whole go straight to y, the partial ones at its ends leave per-row
// partial sums in the workspace for the last of the group's CTAs to arrive,
// which adds them in CTA order (tagged 64-bit arrival counters, as there: no
// workspace preparation); the sum for a CTA's final segment is done by all
// its threads once every role is done.
//
// Roles (800 threads, one CTA per SM, all of tensor memory):
//   warp 0      producer: lane 0 the weight bytes of each stage (bulk copy,
//               before the wait for the quantizer: weights are static),
//               lanes 1-4 its token tiles (a TMA each), lane 5 their scale
//               tiles (bulk copy), after it;
//   warps 1-4   issuers: lane 0 of warp 1 + j issues the MMAs of plane stage
//               j of each stage into accumulator j and commits them (an
//               issuing thread takes ~50 cycles per MMA, independently of the
//               others, measured: four issue four times as fast as one);
//   warps 5-8   epilogue: the four accumulators of each row group segment
//               out of tensor memory (lane quarter warp % 4), added in issuer
//               order, into y or the workspace hand-off;
//   warps 9-24  converters: quartet j converts plane stage j of a stage for
//               the 32 rows of its lane quarter.
// Every wait is bounded; on expiry the kernel records MXS_ERR_TIMEOUT
// (mxs_device_status), skips its remaining arithmetic and stores, drains its
// copies and frees tensor memory.
#include <algorithm>
#include <atomic>
#include <cstring>

#include "common.cuh"

namespace mxs {

__device__ int g_dtc_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

#ifndef MXS_DTC_WIN
#define MXS_DTC_WIN 4
#endif
constexpr int kWin = MXS_DTC_WIN;               // plane stages per stage: one issuer and one converter quartet each
constexpr int kIssWarp0 = 1, kEpiWarp0 = 1 + kWin, kConvWarp0 = kEpiWarp0 + 4, kConvWarps = 4 * kWin;
constexpr int kDThreads = (kConvWarp0 + kConvWarps) * 32;  // 800 (25 warps)
constexpr int kTokTile = 16 * 128;              // one plane stage of 16 token rows
constexpr int kSlotTok = kWin * kTokTile;       // token tiles of a stage (1024-aligned)
constexpr int kSlotSf = kWin * 512;             // their scale tiles
constexpr int kSlotW = 4 * kWin * 2176;         // >= 2 kWin x 4224: the weights
constexpr int kSlotBytes = kSlotTok + kSlotSf + kSlotW;  // 45056 = 44 KiB for four plane stages
static_assert(kSlotBytes % 1024 == 0 && kSlotW >= 2 * kWin * 4224, "ring slot");
constexpr int kDMaxProblems = 3;
constexpr int kDMaxCtas = 256;
constexpr int64_t kDMinCtaBytes = 65536;
constexpr long long kDWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock
// tensor-memory columns: A tiles 128 buf (kNA buffers), accumulators
// 256 + 64 ab + 16 j (one per issuer j), weight scale tiles 384 + 16 buf + 4 j,
// token scale tiles 416 + 16 buf + 4 j
#ifndef MXS_DTC_NA
#define MXS_DTC_NA 2
#endif
constexpr int kNA = MXS_DTC_NA;
constexpr uint32_t kACols = 32 * kWin;  // one A tile
constexpr uint32_t kAcc0 = kACols * kNA, kSfa0 = kAcc0 + 32 * kWin, kSfb0 = kSfa0 + 4 * kWin * kNA, kTmemCols = 512;
static_assert(kSfb0 + 4 * kWin * kNA <= kTmemCols, "tensor-memory columns");

struct DtcProblem {
    const uint8_t *w;              // packed weights (compact part)
    const uint8_t *tok_sf;         // the planes' token scale tiles (512 bytes per plane stage)
    float *y;
    unsigned long long *cnt;       // workspace: arrival counters [G]
    float *rec;                    // workspace: partial sums [ncta][2][M][128]
    int64_t ld_y, GB, W;
    int N, G, nb, n4, n6, st4, nst;
    int cta0, ncta;
};
struct DtcParams {
    DtcProblem prob[kDMaxProblems];
    int4 span[kDMaxCtas];          // per CTA: first group, its first slot, last group, end slot in it
    unsigned long long tag;        // this call's counter tag (48 bits, nonzero)
    int nprob, M;
    int starve;                    // test hook: > 0 makes every CTA skip the weight copy of its stage starve-1
};

__host__ __device__ __forceinline__ int64_t slot_off_d(int n4, int s) {
    return s < n4 ? 2176 * (int64_t)s : 2176 * (int64_t)n4 + 4224 * (int64_t)(s - n4);
}
__host__ __device__ __forceinline__ int slot_at_d(int n4, int64_t off) {
    const int64_t b4 = 2176 * (int64_t)n4;
    return off <= b4 ? (int)(off / 2176) : n4 + (int)((off - b4) / 4224);
}
#ifndef MXS_DTC_COST8
#define MXS_DTC_COST8 100
#endif
// the work split's weight of a 6/8-bit slot, in percent of its bytes (a
// 4-bit slot weighs its bytes): converting a 6/8-bit plane stage takes more
// instructions per byte than a 4-bit one, but on the 70B layers 130 and 160
// measured no better than the bytes alone (100)
constexpr int64_t kCost8 = MXS_DTC_COST8;
static_assert(kCost8 >= 50 && kCost8 <= 200, "split weight");
// start of CTA k's range: the first plane-stage boundary (four 4-bit slots,
// two 6/8-bit slots, the end of the 4-bit run, the group's end) at or after
// the weighted position k * C / ncta (C: the problem's total weight)
__host__ __device__ __forceinline__ int64_t dtc_start(int k, int ncta, int64_t W, int64_t GB, int n4, int nb) {
    if (k >= ncta) return W;
    const int64_t G = W / GB, w4 = 100 * 2176, w8 = kCost8 * 4224;
    const int64_t CG = w4 * n4 + w8 * (nb - n4), b = G * CG * k / ncta;
    const int64_t g = b / CG, rem = b - g * CG, c4 = w4 * n4;
    int64_t off;
    if (rem <= c4) {
        int64_t s = (rem + w4 - 1) / w4;
        s = (s + 3) / 4 * 4;
        if (s > n4) s = n4;
        off = 2176 * s;
    } else {
        int64_t t = (rem - c4 + w8 - 1) / w8;
        t = (t + 1) / 2 * 2;
        if (t > nb - n4) t = nb - n4;
        off = 2176 * (int64_t)n4 + 4224 * t;
    }
    return g * GB + off;
}
// the CTAs of a problem whose ranges meet group g: [first, last]
__host__ __device__ __forceinline__ int first_cta_d(const int4 *sp, int n, int g) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) / 2;
        if (sp[mid].x < g || (sp[mid].x == g && sp[mid].y == 0)) lo = mid; else hi = mid - 1;
    }
    return lo;
}
__host__ __device__ __forceinline__ int last_cta_d(const int4 *sp, int n, int g, int nb) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        const int mid = (lo + hi) / 2;
        if (sp[mid].z > g || (sp[mid].z == g && sp[mid].w == nb)) hi = mid; else lo = mid + 1;
    }
    return lo;
}

// A segment's stages: its 4-bit slots [sa, e4) by windows of four plane
// stages (plane stage s / 4), then its 6/8-bit slots [a8, sb) the same way
// (plane stage st4 + (s - n4) / 2).  Stage k: slots [lo, hi), plane stages
// [ps, ps + nps), and whether it is a 4-bit stage.
struct Stage {
    int lo, hi, ps, nps;
    bool b4;
};
__host__ __device__ __forceinline__ int stage_count_d(int sa, int sb, int n4) {
    const int e4 = max(sa, min(sb, n4)), a8 = max(sa, n4);
    const int p4 = e4 > sa ? (e4 + 3) / 4 - sa / 4 : 0;
    const int p8 = sb > a8 ? (sb - n4 + 1) / 2 - (a8 - n4) / 2 : 0;
    return (p4 + kWin - 1) / kWin + (p8 + kWin - 1) / kWin;
}
// the most plane stages any stage of a segment has (the first window of each
// width run is the fullest)
__host__ __device__ __forceinline__ int stage_npmax(int sa, int sb, int n4) {
    const int e4 = max(sa, min(sb, n4)), a8 = max(sa, n4);
    const int p4 = e4 > sa ? (e4 + 3) / 4 - sa / 4 : 0;
    const int p8 = sb > a8 ? (sb - n4 + 1) / 2 - (a8 - n4) / 2 : 0;
    return max(min(kWin, p4), min(kWin, p8));
}
__host__ __device__ __forceinline__ Stage stage_at(int sa, int sb, int n4, int st4, int k) {
    const int e4 = max(sa, min(sb, n4)), a8 = max(sa, n4);
    const int p4 = e4 > sa ? (e4 + 3) / 4 - sa / 4 : 0;
    const int k4 = (p4 + kWin - 1) / kWin;
    Stage s;
    if (k < k4) {
        const int ps = sa / 4 + kWin * k;
        s.b4 = true;
        s.ps = ps;
        s.nps = min(kWin, (e4 + 3) / 4 - ps);
        s.lo = max(sa, 4 * ps);
        s.hi = min(e4, 4 * (ps + s.nps));
    } else {
        const int q = (a8 - n4) / 2 + kWin * (k - k4);  // plane stage within the 6/8-bit run
        s.b4 = false;
        s.ps = st4 + q;
        s.nps = min(kWin, (sb - n4 + 1) / 2 - q);
        s.lo = max(a8, n4 + 2 * q);
        s.hi = min(sb, n4 + 2 * (q + s.nps));
    }
    return s;
}

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
__device__ __forceinline__ bool mbar_poll(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
#ifndef MXS_DTC_SUSPEND_NS
#define MXS_DTC_SUSPEND_NS 1000
#endif
// the same test, but a thread whose phase is not complete is suspended until it
// completes or `ns` nanoseconds pass: a waiting warp takes no issue slots from
// the converters (a spinning one took most of them)
__device__ __forceinline__ bool mbar_poll_sleep(uint64_t *bar, uint32_t parity, uint32_t ns) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity), "r"(ns)
        : "memory");
    return ok != 0;
}
// bounded wait; on expiry the CTA's abort flag and the sticky status are set
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (mbar_poll(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (mbar_poll_sleep(bar, parity, MXS_DTC_SUSPEND_NS)) return true;
        if (*abort) return false;
        if (clock64() - t0 > kDWaitCycles) {
            *abort = 1;
            atomicExch(&g_dtc_status, MXS_ERR_TIMEOUT);
            return false;
        }
    }
}
// whole-warp wait: every lane waits (its own acquiring test), and the warp goes
// on only if all of them saw the phase
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_poll(bar, parity) && clock64() - t0 < kDWaitCycles) {
    }
}
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     su32(dst)),
                 "l"(src), "r"(bytes), "r"(su32(bar))
                 : "memory");
}
// box (128 bytes of K', 16 token rows) of the planes at K' byte x
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
            su32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(su32(bar)), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
// named barrier over n threads (whole warps) that also ANDs a flag across them
__device__ __forceinline__ bool bar_and(int id, int n, bool v) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred pi, po;\n setp.ne.u32 pi, %1, 0;\n bar.red.and.pred po, %2, %3, pi;\n selp.u32 %0, 1, 0, po;\n}"
        : "=r"(r)
        : "r"((uint32_t)v), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// UMMA descriptors: a 128B-swizzled K-major tile (8-row atoms of 1024 B) and a
// 32 x 16 B scale tile; a byte offset d moves a descriptor by d >> 4
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t desc_sf(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)(128 >> 4) << 32) | ((uint64_t)1 << 46);
}
// kind::mxf8f6f4, e4m3 x e4m3, K-major, N = 16, UE8M0 scales, M = 128; scale
// byte sfa_id / sfb_id of each 32-bit scale column
constexpr uint32_t kIdescMx = ((uint32_t)(16 >> 3) << 17) | (1u << 23) | ((uint32_t)(128 >> 4) << 24);
__device__ __forceinline__ constexpr uint32_t idesc_mx(int sfa_id, int sfb_id) {
    return kIdescMx | ((uint32_t)sfb_id << 4) | ((uint32_t)sfa_id << 29);
}
// kind::f16, bf16 x bf16, K-major, N = 16, M = 128, f32 accumulator
constexpr uint32_t kIdescBf =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(16 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
__device__ __forceinline__ void mma_bf_t(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %4, p;\n}" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(accum), "r"(kIdescBf)
        : "memory");
}
__device__ __forceinline__ void mma_mx_t(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t id, uint32_t sfa,
                                         uint32_t sfb, uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%5], [%6], p;\n}" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(id), "r"(accum), "r"(sfa), "r"(sfb)
        : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
        "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
        "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_cp_sf(uint32_t taddr, uint64_t desc) {
    asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
                 : "memory");
}

// e4m3 bytes (sign << 7) | |m| of the four low / four high sign-magnitude
// nibbles (s << 3) | |m| held in a word
// (the low nibble's sign, bit 3, becomes bit 7 by adding 120 where it is set:
// n + 15 (n & 8) per byte never carries, n <= 15; an IMAD keeps the work off
// the busier integer pipe)
__device__ __forceinline__ uint32_t lo_nib(uint32_t w) { return (w & 0x0F0F0F0Fu) + (w & 0x08080808u) * 15u; }
__device__ __forceinline__ uint32_t hi_nib(uint32_t w) { return ((w >> 4) & 0x07070707u) | (w & 0x80808080u); }
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
// bf16 pair of two 7-bit sign-magnitude codes (s << 7) | m spread by prmt into
// the 16-bit lanes of t (the code in the low byte, its sign replicated in the
// high one): with eb = E in each lane's exponent field, (s | E | m) - (s | E)
// = +-m * 2^(E-134), exact (a NaN when eb holds the NaN pattern)
__device__ __forceinline__ uint32_t bf16_codes(uint32_t t, uint32_t eb) {
    const uint32_t y = (t & 0x807F807Fu) | eb;
    const uint32_t o = (t & 0x80008000u) | eb;
    uint32_t d;
    asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(o), "r"(0xBF80BF80u), "r"(y));  // y - o
    return d;
}

// A CTA's segments (group, slots [sa, sb), side) in processing order: its
// partial groups first (the tail of its first group, then the head of its
// last), so that their hand-off overlaps the whole groups that follow.
struct Segs {
    int n, np, gfull;
    int4 part0, part1;
};
__device__ __forceinline__ Segs segments_d(int4 sp, int nb) {
    Segs s;
    s.part0 = s.part1 = make_int4(0, 0, 0, 0);
    if (sp.x == sp.z) {
        const bool whole = sp.y == 0 && sp.w == nb;
        s.np = whole ? 0 : 1;
        s.part0 = make_int4(sp.x, sp.y, sp.w, 0);
        s.gfull = whole ? sp.x : sp.x + 1;
        s.n = 1;
        return s;
    }
    const bool lead = sp.y > 0, trail = sp.w < nb;
    const int4 head = make_int4(sp.x, sp.y, nb, 0), tail = make_int4(sp.z, 0, sp.w, 1);
    s.part0 = lead ? head : tail;
    s.part1 = tail;
    s.np = (lead ? 1 : 0) + (trail ? 1 : 0);
    s.gfull = sp.x + (lead ? 1 : 0);
    s.n = s.np + (sp.z - (trail ? 1 : 0)) - s.gfull + 1;
    return s;
}
__device__ __forceinline__ int4 segment_d(const Segs &s, int i, int nb) {
    if (i < s.np) return i == 0 ? s.part0 : s.part1;
    return make_int4(s.gfull + (i - s.np), 0, nb, 0);
}

// One arrival on a row group's counter word (tag << 16 | count) for the call
// tagged `tag` (the caller's release fence comes first); returns the
// arrival's count, 1-based, or 0 if the fallback ran out.  Tags grow call by
// call, so the maximum turns an earlier call's word into (tag, 0) and one add
// takes the count; a word that holds another tag even so (prior contents of
// a workspace) goes through compare-and-swap, which reads it as count 0.
__device__ __forceinline__ unsigned arrive_count(unsigned long long *cw, unsigned long long tag) {
    atomicMax(cw, tag << 16);
    unsigned long long cur = atomicAdd(cw, 1ull);
    if ((cur >> 16) == tag) return (unsigned)(cur & 0xFFFFull) + 1;
    cur += 1;  // the word after this add, as far as this thread knows
    for (int it = 0; it < (1 << 20); ++it) {
        const unsigned long long c = (cur >> 16) == tag ? (cur & 0xFFFFull) + 1 : 1;
        const unsigned long long prev = atomicCAS(cw, cur, (tag << 16) | c);
        if (prev == cur) return (unsigned)c;
        cur = prev;
    }
    return 0;
}

// The last of row group g's CTAs to arrive, at the end of the kernel: every
// contributor's partial sums (CTAs f..l, in CTA order) added for the group's
// rows and the M tokens by all of the CTA's threads, a few outputs each with
// the contributors' values in flight together.
__device__ __forceinline__ void final_sum(const DtcProblem &P, const int4 *pspan, int M, int g, int f, int l) {
    constexpr int kPer = (16 * 128 + kDThreads - 1) / kDThreads;  // outputs per thread
    constexpr int kBatch = 8;                                      // contributors in flight
    const int no = M * 128;
    float acc[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) acc[e] = 0.0f;
    for (int k0 = f; k0 <= l; k0 += kBatch) {
        float pv[kBatch][kPer];
#pragma unroll
        for (int d = 0; d < kBatch; ++d) {
            const int kk = k0 + d;
            const int sd = kk <= l && pspan[kk].x < g ? 1 : 0;  // g is that CTA's last group
            const float *src = P.rec + (size_t)(kk * 2 + sd) * no;
#pragma unroll
            for (int e = 0; e < kPer; ++e) {
                const int o = (int)threadIdx.x + e * kDThreads;
                pv[d][e] = kk <= l && o < no ? __ldcg(src + o) : 0.0f;
            }
        }
#pragma unroll
        for (int d = 0; d < kBatch; ++d)
#pragma unroll
            for (int e = 0; e < kPer; ++e)
                if (k0 + d <= l) acc[e] = k0 + d == f ? pv[d][e] : acc[e] + pv[d][e];
    }
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
        const int o = (int)threadIdx.x + e * kDThreads, n = 128 * g + (o & 127);
        if (o < no && n < P.N) P.y[(int64_t)(o >> 7) * P.ld_y + n] = acc[e];
    }
}

template <int NR>
__global__ void __launch_bounds__(kDThreads, 1) decode_tc_kernel(const __grid_constant__ DtcParams dp,
                                                                const __grid_constant__ CUtensorMap map0,
                                                                const __grid_constant__ CUtensorMap map1,
                                                                const __grid_constant__ CUtensorMap map2) {
    int pi = 0;
    while (pi + 1 < dp.nprob && (int)blockIdx.x >= dp.prob[pi + 1].cta0) ++pi;
    const DtcProblem &P = dp.prob[pi];
    const CUtensorMap *tok_map = pi == 0 ? &map0 : (pi == 1 ? &map1 : &map2);
    const int kc = (int)blockIdx.x - P.cta0;
    const int4 sp = dp.span[blockIdx.x];
    const Segs segs = segments_d(sp, P.nb);
    const int M = dp.M, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t sbase = su32(smem_raw);
    uint8_t *smem = smem_raw + (((sbase + 1023) & ~1023u) - sbase);  // 1024-aligned for the swizzled tiles
    uint8_t *ring = smem;                                            // NR slots: [tokens][token sf][weights]
    uint8_t *sfa = ring + (size_t)NR * kSlotBytes;                   // [kNA][kWin][512] weight scale tiles
    uint64_t *full_w = reinterpret_cast<uint64_t *>(sfa + kNA * kWin * 512);
    uint64_t *full_t = full_w + NR, *freeb = full_t + NR, *empty_w = freeb + NR;
    uint64_t *a_full = empty_w + NR, *a_free = a_full + kNA, *acc_full = a_free + kNA, *acc_empty = acc_full + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_empty + 2);
    // abort, last arriver, first and last CTA of its group, the final sum pending, its group
    volatile int *flags = reinterpret_cast<volatile int *>(tmem_slot + 1);
    volatile int *abort_flag = flags;

    if (threadIdx.x == 0) {
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        for (int i = 0; i < NR; ++i) {
            mbar_init(&full_w[i], 1);
            mbar_init(&full_t[i], 1);
            mbar_init(&freeb[i], kWin);        // each issuer's commit after the stage's MMAs: its token tiles are free
            mbar_init(&empty_w[i], kConvWarps);  // the converters have read the stage's weights
        }
        for (int i = 0; i < kNA; ++i) {
            mbar_init(&a_full[i], kConvWarps);
            mbar_init(&a_free[i], kWin);  // each issuer's commit
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], kWin);  // each issuer's commit at the segment's end
            mbar_init(&acc_empty[i], 4);    // the four epilogue warps
        }
        flags[0] = flags[1] = flags[2] = flags[3] = flags[4] = flags[5] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        __syncwarp();
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = *tmem_slot;

    int issued = 0;  // (producer lanes) copies issued, for the drain after an abort
    if (warp == 0) {
        // ---- producer: lane 0 the weights of each stage, lanes 1-4 its token
        // tiles (plane stage lane - 1 of the stage), lane 5 their scale tiles
        // (the planes may come from the kernel just before: those lanes wait
        // for it first).  Copies issued by one thread are served one after
        // another, so each stream has its own lane.  A slot is refilled once the
        // MMAs of its last stage have run.
        int pre = 0;
        if (lane == 0) {
            // the weights of the ring's first NR stages at once, before the
            // warp waits for the kernel before (a warp's lanes pass that wait
            // together): their slots are free and the weights are static, so
            // the converters fill the A tiles while the quantizer runs
            int gs = 0;
            for (int si = 0; si < segs.n && gs < NR && dp.starve != gs + 1; ++si) {
                const int4 sg = segment_d(segs, si, P.nb);
                const int nst = stage_count_d(sg.y, sg.z, P.n4);
                for (int k = 0; k < nst && gs < NR && dp.starve != gs + 1; ++k, ++gs) {
                    const Stage st = stage_at(sg.y, sg.z, P.n4, P.st4, k);
                    const int64_t off = slot_off_d(P.n4, st.lo);
                    const uint32_t bytes = (uint32_t)(slot_off_d(P.n4, st.hi) - off);
                    mbar_expect_tx(&full_w[gs], bytes);
                    bulk_load(ring + (size_t)gs * kSlotBytes + kSlotTok + kSlotSf, P.w + (int64_t)sg.x * P.GB + off,
                              bytes, &full_w[gs]);
                }
            }
            pre = issued = gs;
        }
        __syncwarp();
        if (lane <= kWin + 1) {
            asm volatile("griddepcontrol.wait;" ::: "memory");  // the planes: written by the kernel before
            int gs = 0;
            bool ok = true;
            for (int si = 0; si < segs.n && ok; ++si) {
                const int4 sg = segment_d(segs, si, P.nb);
                const int nst = stage_count_d(sg.y, sg.z, P.n4);
                for (int k = 0; k < nst; ++k, ++gs) {
                    if (gs < pre) continue;  // (lane 0: issued above)
                    const Stage st = stage_at(sg.y, sg.z, P.n4, P.st4, k);
                    const int s = gs % NR;
                    // the weights' part of a slot is free once the converters have read
                    // it, the tokens' part once the MMAs have
                    uint64_t *fb = lane == 0 ? &empty_w[s] : &freeb[s];
                    if ((lane == 0 && dp.starve == gs + 1) || *abort_flag ||
                        (gs >= NR && !mbar_wait(fb, (uint32_t)(gs / NR - 1) & 1, abort_flag))) {
                        ok = false;
                        break;
                    }
                    uint8_t *slot = ring + (size_t)s * kSlotBytes;
                    if (lane == 0) {
                        const int64_t off = slot_off_d(P.n4, st.lo);
                        const uint32_t bytes = (uint32_t)(slot_off_d(P.n4, st.hi) - off);
                        mbar_expect_tx(&full_w[s], bytes);
                        bulk_load(slot + kSlotTok + kSlotSf, P.w + (int64_t)sg.x * P.GB + off, bytes, &full_w[s]);
                    } else if (lane <= kWin) {
                        const int j = lane - 1;
                        if (j == 0) mbar_expect_tx(&full_t[s], (uint32_t)(st.nps * (kTokTile + (st.b4 ? 512 : 0))));
                        if (j < st.nps) tma_load_2d(slot + j * kTokTile, tok_map, &full_t[s], 128 * (st.ps + j), 0);
                    } else if (st.b4) {
                        bulk_load(slot + kSlotTok, P.tok_sf + (int64_t)st.ps * 512, (uint32_t)st.nps * 512, &full_t[s]);
                    }
                    issued = gs + 1;
                }
            }
        }
        __syncwarp();
    } else if (warp < kEpiWarp0) {
        // ---- the MMA issuers: issuer j (warp 1 + j, lane 0) issues the MMAs of
        // plane stage j of every stage into its own accumulator (an issuing
        // thread takes ~50 cycles per MMA whatever the other issuers do, so four
        // of them issue four times as fast)
        const int j = warp - kIssWarp0;
        int committed = -1;  // the last stage whose MMAs were committed
        if (lane == 0) {
            int gs = 0;
            bool ok = true;
            for (int si = 0; si < segs.n && ok; ++si) {
                const int4 sg = segment_d(segs, si, P.nb);
                const int nst = stage_count_d(sg.y, sg.z, P.n4), ab = si & 1;
                const uint32_t acc = tmem + kAcc0 + 16 * kWin * ab + 16 * j;
                bool first = true;
                for (int k = 0; k < nst; ++k, ++gs) {
                    const Stage st = stage_at(sg.y, sg.z, P.n4, P.st4, k);
                    const int s = gs % NR, buf = gs % kNA;
                    ok = mbar_wait(&a_full[buf], (uint32_t)(gs / kNA) & 1, abort_flag) &&
                         mbar_wait(&full_t[s], (uint32_t)(gs / NR) & 1, abort_flag) &&
                         (k > 0 || si < 2 || mbar_wait(&acc_empty[ab], (uint32_t)((si >> 1) - 1) & 1, abort_flag));
                    if (!ok) break;
                    if (j < st.nps) {
                        fence_after();
                        uint8_t *slot = ring + (size_t)s * kSlotBytes;
                        const uint64_t tj = desc_sw128(su32(slot)) + (uint64_t)(j * (kTokTile >> 4));
                        const uint32_t aT = tmem + kACols * buf + 32 * j;
                        if (st.b4) {
                            const uint32_t sfa_t = tmem + kSfa0 + 4 * kWin * buf + 4 * j;
                            const uint32_t sfb_t = tmem + kSfb0 + 4 * kWin * buf + 4 * j;
                            tmem_cp_sf(sfa_t, desc_sf(su32(sfa + (buf * kWin + j) * 512)));
                            tmem_cp_sf(sfb_t, desc_sf(su32(slot + kSlotTok + j * 512)));
                            const int base = 4 * (st.ps + j);
                            if (base >= st.lo && base + 4 <= st.hi) {  // all four slots: one straight run
                                const uint32_t a0 = first ? 0u : 1u;
                                mma_mx_t(acc, aT, tj, idesc_mx(0, 0), sfa_t, sfb_t, a0);
                                mma_mx_t(acc, aT + 8, tj + 2, idesc_mx(1, 1), sfa_t, sfb_t, 1u);
                                mma_mx_t(acc, aT + 16, tj + 4, idesc_mx(2, 2), sfa_t, sfb_t, 1u);
                                mma_mx_t(acc, aT + 24, tj + 6, idesc_mx(3, 3), sfa_t, sfb_t, 1u);
                                first = false;
                            } else {
#pragma unroll
                                for (int q = 0; q < 4; ++q) {
                                    if (base + q < st.lo || base + q >= st.hi) continue;
                                    mma_mx_t(acc, aT + 8 * q, tj + 2 * q, idesc_mx(q, q), sfa_t, sfb_t, first ? 0u : 1u);
                                    first = false;
                                }
                            }
                        } else {
                            const int base = P.n4 + 2 * (st.ps + j - P.st4);
                            if (base >= st.lo && base + 2 <= st.hi) {  // both slots
                                const uint32_t a0 = first ? 0u : 1u;
                                mma_bf_t(acc, aT, tj, a0);
                                mma_bf_t(acc, aT + 8, tj + 2, 1u);
                                mma_bf_t(acc, aT + 16, tj + 4, 1u);
                                mma_bf_t(acc, aT + 24, tj + 6, 1u);
                                first = false;
                            } else {
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    if (base + h < st.lo || base + h >= st.hi) continue;
                                    mma_bf_t(acc, aT + 16 * h, tj + 4 * h, first ? 0u : 1u);
                                    mma_bf_t(acc, aT + 16 * h + 8, tj + 4 * h + 2, 1u);
                                    first = false;
                                }
                            }
                        }
                    }
                    mma_commit(&a_free[buf]);  // the A tile and scale columns are free once read
                    mma_commit(&freeb[s]);     // and the slot's token tiles
                    if (k == nst - 1) mma_commit(&acc_full[ab]);  // this issuer's share of the segment is done
                    committed = gs;
                }
            }
            if (committed >= 0 && *abort_flag)  // drain: the last commit
                drain_wait(&a_free[committed % kNA], (uint32_t)(committed / kNA) & 1);
        }
        __syncwarp();
    } else if (warp < kConvWarp0) {
        // ---- epilogue: accumulator row (= weight row) 32 * qtr + lane, columns = tokens
        const int qtr = warp & 3, r = 32 * qtr + lane, et = threadIdx.x - 32 * kEpiWarp0;
        const int4 *pspan = dp.span + P.cta0;
        asm volatile("griddepcontrol.wait;" ::: "memory");  // y and the workspace after the kernels before
        for (int si = 0; si < segs.n; ++si) {
            const int4 sg = segment_d(segs, si, P.nb);
            const int g = sg.x, ab = si & 1, n = 128 * g + r;
            const bool whole = sg.y == 0 && sg.z == P.nb;
            int kf = 0, kl = 0;
            if (!whole && et == 0) {  // ahead of the wait: the group's contributors
                kf = first_cta_d(pspan, P.ncta, g);
                kl = last_cta_d(pspan, P.ncta, g, P.nb);
            }
            // the four warps agree on going on (one that gave up would leave the
            // others at the named barrier)
            if (!bar_and(3, 128, warp_wait(&acc_full[ab], (uint32_t)(si >> 1) & 1, abort_flag))) break;
            fence_after();
            // issuer j's accumulator holds MMAs of this segment when one of its
            // stages has more than j plane stages (each has a slot in every one)
            const int npmax = stage_npmax(sg.y, sg.z, P.n4);
            float v[16];
            {
                uint32_t u[16];
                tmem_ld16(tmem + ((uint32_t)(32 * qtr) << 16) + kAcc0 + 16 * kWin * ab, u);
#pragma unroll
                for (int t = 0; t < 16; ++t) v[t] = __uint_as_float(u[t]);
            }
            for (int jj = 1; jj < npmax; ++jj) {  // in issuer order: deterministic
                uint32_t u[16];
                tmem_ld16(tmem + ((uint32_t)(32 * qtr) << 16) + kAcc0 + 16 * kWin * ab + 16 * jj, u);
#pragma unroll
                for (int t = 0; t < 16; ++t) v[t] += __uint_as_float(u[t]);
            }
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[ab]);
            if (whole) {
                if (n < P.N && !*abort_flag)
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        if (t < M) P.y[(int64_t)t * P.ld_y + n] = v[t];
                continue;
            }
            // part of the group: this CTA's sums into the workspace, one arrival
            // (release: a fence after the stores); the last of the group's CTAs
            // to arrive adds all of them in CTA order (for the CTA's final
            // segment, with all its threads once every role is done)
            float *mine = P.rec + (size_t)(kc * 2 + sg.w) * M * 128;
#pragma unroll
            for (int t = 0; t < 16; ++t)
                if (t < M) mine[t * 128 + r] = v[t];
            named_sync(3, 128);
            if (et == 0) {
                int last = 0;
                if (!*abort_flag) {
                    unsigned long long *cw = P.cnt + g;
                    asm volatile("fence.acq_rel.gpu;" ::: "memory");
                    const unsigned c = arrive_count(cw, dp.tag);
                    if (c == 0) {
                        *abort_flag = 1;
                        atomicExch(&g_dtc_status, MXS_ERR_TIMEOUT);
                    }
                    last = c == (unsigned)(kl - kf + 1);
                    if (last) {
                        asm volatile("fence.acq_rel.gpu;" ::: "memory");
                        // (tag, 0): what a replay of this call expects to find
                        asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(cw), "l"(dp.tag << 16) : "memory");
                        flags[2] = kf;
                        flags[3] = kl;
                        if (si == segs.n - 1) {  // the CTA's final segment: summed at the end
                            flags[5] = g;
                            flags[4] = 1;
                            last = 0;
                        }
                    }
                }
                flags[1] = last;
            }
            named_sync(3, 128);
            if (flags[1] && n < P.N) {
                // contributors in CTA order, each one's tokens loaded together
                const int f = flags[2], l = flags[3];
                float sum[16];
                for (int kk = f; kk <= l; ++kk) {
                    const int sd = pspan[kk].x < g ? 1 : 0;  // g is that CTA's last group
                    const float *src = P.rec + (size_t)(kk * 2 + sd) * M * 128 + r;
                    float pv[16];
#pragma unroll
                    for (int t = 0; t < 16; ++t) pv[t] = t < M ? __ldcg(src + t * 128) : 0.0f;
#pragma unroll
                    for (int t = 0; t < 16; ++t) sum[t] = kk == f ? pv[t] : sum[t] + pv[t];
                }
#pragma unroll
                for (int t = 0; t < 16; ++t)
                    if (t < M) P.y[(int64_t)t * P.ld_y + n] = sum[t];
            }
            named_sync(3, 128);  // the flags are reused by the next segment
        }
    } else {
        // ---- converters: quartet j converts plane stage j of each stage for the
        // 32 rows of its lane quarter into the A tile (tensor memory) and, for a
        // 4-bit stage, the rows' scale bytes into the weight scale tile
        const int cw = warp - kConvWarp0, j = cw >> 2, qtr = warp & 3, r = 32 * qtr + lane;
        const uint32_t a_lane = (uint32_t)(32 * qtr) << 16;
        int gs = 0;
        bool ok = true;
        for (int si = 0; si < segs.n; ++si) {
            const int4 sg = segment_d(segs, si, P.nb);
            const int nst = stage_count_d(sg.y, sg.z, P.n4);
            for (int k = 0; k < nst; ++k, ++gs) {
                const Stage st = stage_at(sg.y, sg.z, P.n4, P.st4, k);
                const int s = gs % NR, buf = gs % kNA;
                if (ok) ok = warp_wait(&full_w[s], (uint32_t)(gs / NR) & 1, abort_flag);
                if (ok && gs >= kNA) ok = warp_wait(&a_free[buf], (uint32_t)(gs / kNA - 1) & 1, abort_flag);
                if (ok && j < st.nps) {
                    const uint8_t *wst = ring + (size_t)s * kSlotBytes + kSlotTok + kSlotSf;  // the stage's weights
                    uint32_t d[32];
                    if (st.b4) {
                        // plane stage ps: slots 4 ps .. 4 ps + 3 (those outside [lo, hi) are zeros),
                        // 2176 bytes apart in the stage
                        const int ps = st.ps + j;
                        const uint8_t *src0 = wst + 2176 * (4 * ps - st.lo);
                        uint4 v[4];
                        uint32_t sb = 0;
                        const bool whole = 4 * ps >= st.lo && 4 * ps + 4 <= st.hi;  // all four slots present
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int sl = 4 * ps + q;
                            v[q] = make_uint4(0, 0, 0, 0);
                            if (whole || (sl >= st.lo && sl < st.hi)) {
                                const uint8_t *src = src0 + 2176 * q;
                                v[q] = *reinterpret_cast<const uint4 *>(src + 16 * r);
                                // the code's fixed-point weight in the scale byte: +7, at most
                                // 254; 255 (NaN) stays
                                const uint32_t S = src[2048 + r];
                                sb |= (S == 255u ? 255u : min(S + 7u, 254u)) << (8 * q);
                            }
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            // word i: bytes hold elements 8i..8i+3 (low nibbles), 8i+4..8i+7 (high nibbles)
                            d[8 * q + 0] = lo_nib(v[q].x);
                            d[8 * q + 1] = hi_nib(v[q].x);
                            d[8 * q + 2] = lo_nib(v[q].y);
                            d[8 * q + 3] = hi_nib(v[q].y);
                            d[8 * q + 4] = lo_nib(v[q].z);
                            d[8 * q + 5] = hi_nib(v[q].z);
                            d[8 * q + 6] = lo_nib(v[q].w);
                            d[8 * q + 7] = hi_nib(v[q].w);
                        }
                        // scale tile: row r = 32 qtr + lane at lane `lane`, column qtr; byte q = slot q
                        *reinterpret_cast<uint32_t *>(sfa + (buf * kWin + j) * 512 + lane * 16 + qtr * 4) = sb;
                    } else {
                        // plane stage ps: slots n4 + 2 (ps - st4) + h, h = 0, 1, as bf16
                        // values m * 2^(Sw-127-(b-2)) (the scale inside)
                        const int q0 = P.n4 + 2 * (st.ps + j - P.st4);
                        const uint8_t *src0 = wst + 4224 * (q0 - st.lo);
                        const bool whole = q0 >= st.lo && q0 + 2 <= st.hi;  // both slots present
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int sl = q0 + h;
                            uint4 v0 = make_uint4(0, 0, 0, 0), v1 = v0;
                            uint32_t eb = (1u << 7) | (1u << 23);  // absent slot: zeros
                            if (whole || (sl >= st.lo && sl < st.hi)) {
                                const uint8_t *src = src0 + 4224 * h;
                                v0 = *reinterpret_cast<const uint4 *>(src + 32 * r);
                                v1 = *reinterpret_cast<const uint4 *>(src + 32 * r + 16);
                                const int Sw = src[4096 + r];
                                const int b = sl < P.n4 + P.n6 ? 6 : 8;
                                // exponent field E = Sw + 7 - (b - 2), so that m * 2^(E-134) is the value
                                const uint32_t E = (uint32_t)min(Sw + 9 - b, 254);
                                eb = Sw == 255 ? 0x7FC07FC0u : (E << 7) | (E << 23);
                            }
                            const uint32_t w[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
                            for (int i = 0; i < 8; ++i) {  // word i: elements 4i .. 4i+3
                                d[16 * h + 2 * i] = bf16_codes(prmt(w[i], 0u, 0x9180u), eb);
                                d[16 * h + 2 * i + 1] = bf16_codes(prmt(w[i], 0u, 0xB3A2u), eb);
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&empty_w[s]);  // the stage's weight bytes are in registers
                    tmem_st32(tmem + a_lane + kACols * buf + 32 * j, d);
                    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                    fence_async_smem();
                    fence_before();
                }
                __syncwarp();
                if (lane == 0) {
                    if (!(ok && j < st.nps)) mbar_arrive(&empty_w[s]);  // (a converting warp arrived above)
                    mbar_arrive(&a_full[buf]);  // every converter warp, every stage
                }
            }
        }
    }

    named_sync(1, kDThreads);  // every role is done
    if (flags[4] && !*abort_flag) final_sum(P, dp.span + P.cta0, M, flags[5], flags[2], flags[3]);
    if (warp == 0) {
        if (lane <= kWin + 1 && *abort_flag)  // drain: the last copies into each slot
            for (int s = 0; s < NR && s < issued; ++s) {
                const int last = s + (issued - 1 - s) / NR * NR;
                drain_wait(lane == 0 ? &full_w[s] : &full_t[s], (uint32_t)(last / NR) & 1);
            }
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

}  // namespace

// ------------------------------------------------------------------ host side
namespace {

int sms_dtc() {
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

int64_t planes_bytes(const Plan &p, int64_t M) { return align256(align256(M * p.kp) + (M + 127) / 128 * p.nst * 512); }
int64_t cnt_bytes_d(int64_t G) { return (8 * G + 255) / 256 * 256; }
int64_t rec_bytes_d(int ncta, int64_t M) { return (int64_t)ncta * 2 * M * 128 * 4; }

std::atomic<unsigned long long> g_dtc_tags{0};
std::atomic<int> g_dtc_starve{0};  // mxs_test_decode_arm_starve: the next launch's skipped stage (1-based)

}  // namespace

// CTAs per problem: one each, then one at a time to the problem with the most
// bytes per CTA, each keeping at least kDMinCtaBytes (and more than one plane
// stage, 8704 bytes) per CTA, and no more than its workspace holds partial
// sums for (cap[i]).
void dtc_split_ctas(const int64_t *W, const int *cap_ws, int count, int sms, int *ncta) {
    const int total = std::max(count, std::min(sms, kDMaxCtas));
    int64_t cap[kDMaxProblems];
    int used = 0;
    for (int i = 0; i < count; ++i) {
        cap[i] = std::max<int64_t>(1, std::min<int64_t>(W[i] / 8705, W[i] / kDMinCtaBytes));
        cap[i] = std::min<int64_t>(cap[i], std::max(1, cap_ws[i]));
        ncta[i] = 1;
        ++used;
    }
    while (used < total) {
        int best = -1;
        double bw = -1.0;
        for (int i = 0; i < count; ++i)
            if (ncta[i] < cap[i] && (double)W[i] / ncta[i] > bw) bw = (double)W[i] / ncta[i], best = i;
        if (best < 0) break;
        ++ncta[best];
        ++used;
    }
}

void dtc_span(int k, int n, int64_t W, int64_t GB, int n4, int nb, int *out) {
    const int64_t a = dtc_start(k, n, W, GB, n4, nb), b = dtc_start(k + 1, n, W, GB, n4, nb);
    const int64_t g0 = a / GB, g1 = (b - 1) / GB;
    out[0] = (int)g0;
    out[1] = slot_at_d(n4, a - g0 * GB);
    out[2] = (int)g1;
    out[3] = slot_at_d(n4, b - g1 * GB);
}

int64_t dtc_workspace_bytes(const Plan &p, int64_t M, int64_t N) {
    return planes_bytes(p, M) + cnt_bytes_d((N + 127) / 128) + rec_bytes_d(kDMaxCtas, M);
}

int dtc_status(int *status, int reset) {
    int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_dtc_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyFromSymbol(decode status)");
    *status = v;
    if (reset && v != 0) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_dtc_status, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyToSymbol(decode status)");
    }
    return MXS_OK;
}

void dtc_arm_starve(int stage) { g_dtc_starve.store(stage); }
int dtc_split_cost8() { return (int)kCost8; }

int launch_decode_tc(const Plan *const *plans, void *const *ws, const size_t *ws_bytes, const void *const *packed,
                     const int64_t *N, float *const *y, const int64_t *ld_y, int count, int64_t M, bool pdl,
                     cudaStream_t st) {
    if (count < 1 || count > kDMaxProblems) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d)", count, kDMaxProblems);
    if (M < 1 || M > 16) return fail(MXS_ERR_SHAPE, "the tensor-core decode path takes 1 <= M <= 16");
    int64_t G[kDMaxProblems], GB[kDMaxProblems], W[kDMaxProblems];
    int cap_ws[kDMaxProblems];
    for (int i = 0; i < count; ++i) {
        if (N[i] > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
        const WeightOffsets wo = weight_offsets(*plans[i], N[i], false);
        G[i] = wo.G;
        GB[i] = wo.GB;
        W[i] = G[i] * GB[i];
        const int64_t room = (int64_t)ws_bytes[i] - planes_bytes(*plans[i], M) - cnt_bytes_d(G[i]);
        if (room < rec_bytes_d(1, M) || !ws[i])
            return fail(MXS_ERR_BUFFER, "problem %d: workspace of %lld bytes needed, %zu given", i,
                        (long long)(planes_bytes(*plans[i], M) + cnt_bytes_d(G[i]) + rec_bytes_d(1, M)), ws_bytes[i]);
        cap_ws[i] = (int)std::min<int64_t>(kDMaxCtas, room / rec_bytes_d(1, M));
    }
    int ncta[kDMaxProblems];
    dtc_split_ctas(W, cap_ws, count, sms_dtc(), ncta);
    static thread_local DtcParams dp;
    std::memset(&dp, 0, sizeof(dp));
    unsigned long long tag = 0;
    while (tag == 0) tag = (g_dtc_tags.fetch_add(1) + 1) & 0xFFFFFFFFFFFFull;
    dp.tag = tag;
    dp.nprob = count;
    dp.M = (int)M;
    dp.starve = g_dtc_starve.exchange(0);  // armed for this one launch
    CUtensorMap maps[kDMaxProblems];
    int cta = 0;
    for (int i = 0; i < count; ++i) {
        const Plan &p = *plans[i];
        DtcProblem &P = dp.prob[i];
        uint8_t *base = static_cast<uint8_t *>(ws[i]);
        P.w = static_cast<const uint8_t *>(packed[i]);
        P.tok_sf = base + align256(M * p.kp);
        P.y = y[i];
        P.cnt = reinterpret_cast<unsigned long long *>(base + planes_bytes(p, M));
        P.rec = reinterpret_cast<float *>(base + planes_bytes(p, M) + cnt_bytes_d(G[i]));
        P.ld_y = ld_y[i];
        P.GB = GB[i];
        P.W = W[i];
        P.N = (int)N[i];
        P.G = (int)G[i];
        P.nb = p.nb, P.n4 = p.n4, P.n6 = p.n6, P.st4 = p.st4, P.nst = p.nst;
        P.cta0 = cta;
        P.ncta = ncta[i];
        for (int k = 0; k < ncta[i]; ++k) {
            int sp[4];
            dtc_span(k, ncta[i], W[i], GB[i], p.n4, p.nb, sp);
            dp.span[cta + k] = make_int4(sp[0], sp[1], sp[2], sp[3]);
        }
        cta += ncta[i];
        std::memset(&maps[i], 0, sizeof(CUtensorMap));
        const int rc = make_plane_map(&maps[i], ws[i], M, p.kp, 16);
        if (rc) return rc;
    }
    for (int i = count; i < kDMaxProblems; ++i) maps[i] = maps[0];
#ifndef MXS_DTC_RING
#define MXS_DTC_RING 4
#endif
    constexpr int NR = MXS_DTC_RING;
    const size_t smem = 1024 + (size_t)NR * kSlotBytes + kNA * kWin * 512 + (4 * NR + 2 * kNA + 4) * 8 + 64;
    auto k = decode_tc_kernel<NR>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode_tc smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cta, 1, 1);
    cfg.blockDim = dim3(kDThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    int na = 0;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    e = cudaLaunchKernelEx(&cfg, k, dp, maps[0], maps[1], maps[2]);
    return cuda_fail(e, "decode_tc_kernel launch");
}

}  // namespace mxs

using namespace mxs;

int mxs_test_dtc_split(const int64_t *K, const uint8_t *const *bits, const int64_t *N, int count, int sms,
                       int32_t *ncta, int32_t *spans) {
    if (!K || !bits || !N || !ncta || !spans) return -fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (count < 1 || count > kDMaxProblems || sms < 1)
        return -fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d), sms=%d", count, kDMaxProblems, sms);
    int64_t W[kDMaxProblems], GB[kDMaxProblems];
    int cap_ws[kDMaxProblems];
    Plan plans[kDMaxProblems];
    for (int i = 0; i < count; ++i) {
        const int rc = build_plan(bits[i], K[i], &plans[i]);
        if (rc) return -rc;
        if (N[i] < 1 || N[i] > (int64_t)0x7FFFFFF0) return -fail(MXS_ERR_SHAPE, "N=%lld", (long long)N[i]);
        const WeightOffsets wo = weight_offsets(plans[i], N[i], false);
        GB[i] = wo.GB;
        W[i] = wo.G * wo.GB;
        cap_ws[i] = kDMaxCtas;  // a workspace sized by dtc_workspace_bytes
    }
    int n[kDMaxProblems];
    dtc_split_ctas(W, cap_ws, count, sms, n);
    int cta = 0;
    for (int i = 0; i < count; ++i) {
        ncta[i] = n[i];
        for (int k = 0; k < n[i]; ++k, ++cta) dtc_span(k, n[i], W[i], GB[i], plans[i].n4, plans[i].nb, spans + 4 * cta);
    }
    return cta;
}
