// gemm_decode.cu -- A4: the MXINT GEMM for decode shapes (M <= 16 tokens) on
// the 5th-generation tensor cores.
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea'+Ew') * (integer dot of the
// two blocks' mantissas): the MXINT product of Sec. 2 (fixed-point MACs under
// a shared power-of-two scale) with the per-block widths of Sec. 4.1.
//
// Decode reads every weight byte once, so the kernel streams the weights in
// their compact form (4-bit nibbles, 6/8-bit bytes) and does all arithmetic on
// the tensor core:
//   * 128 weight rows are the A operand -- in tensor memory -- and the <= 16
//     tokens the N = 16 B operand in shared memory; the sum over K stays in
//     fp32 tensor-memory accumulators;
//   * a 4-bit block runs on the block-scaled FP8 MMA (tcgen05.mma
//     kind::mxf8f6f4, scale_vec::1X): its weight code is fed as the e4m3 byte
//     (sign << 7) | |m|, whose value is |m| * 2^-9 (subnormals and the first
//     binade), with the code's fixed-point weight in the E8M0 scale byte (+7),
//     and the hardware applies the per-block scales;
//   * a 6/8-bit block runs on the bf16 MMA (kind::f16, two K = 16 MMAs): its
//     codes become the exact bf16 values m * 2^(Sw-127-(b-2)) (two integer
//     operations and one exact bf16 subtraction per two codes), and the
//     token operand holds the activations' bf16 values the same way; every
//     MMA term is exact.  (Two e4m3 digits per code on both sides, Sec. 6's
//     high/low split, took four FP8 MMAs per block: the MMA's fixed issue
//     cost makes two bf16 MMAs cheaper);
//   * the token operand is the activations' MMA-plane form (the layout the
//     prefill GEMM reads: e4m3 values m/4 under the block's own scale byte,
//     or bf16 values).  It is either loaded by TMA from planes
//     written by mxs_quantize_act -- the launch may then overlap the kernel
//     before it (programmatic dependent launch) -- or built in the prologue
//     from packed codes.
// Work: a CTA owns 128-row weight groups and (in a cluster) a K range of them,
// cut into MMA stages of 128 K'-bytes (four 4-bit slots or two 6/8-bit
// slots); two stages make one copy chunk.  One thread streams the chunks into
// a shared-memory ring with cp.async.bulk (about 17 KB per copy, up to eight
// in flight: the ring, not registers, holds the bytes in flight).  Four quads
// of four worker warps take the chunks round robin; each warp converts its 32
// rows (its tensor-memory lane quarter) of a stage and writes the e4m3 or
// bf16 values straight into the quad's A tile in tensor memory (tcgen05.st), the quad
// meets at a hardware named barrier, and one thread issues the stage's MMAs
// into the quad's accumulator.  Quads never wait for one another; the
// epilogue warps add the quads' partial accumulators in quad order (a fixed
// order: results are deterministic).  Warps 1-4 also load the token operand.
// K is split over the CTAs of a thread-block cluster when N alone cannot
// occupy the GPU.  The ranks then reduce-scatter through distributed shared
// memory: rank k receives rows [k*R, (k+1)*R) (R = 128/cluster size) of every
// other rank's partial tile by bulk copy, adds the partials in rank order and
// stores those rows.  A K range whose token operand does not fit shared
// memory runs as several passes, each adding into y.
// Every wait is bounded; on expiry the kernel records MXS_ERR_TIMEOUT, stops,
// drains what it issued and frees tensor memory.  The quads' named barrier
// carries an AND of the four warps' status, so a warp that gave up stops its
// quad at the next stage instead of leaving the others at the barrier.
// Weight scale bytes above 247 of a 4-bit block (|w| >= 2^120) saturate at
// 254 after the shift, as do those above 251 (6-bit) and 253 (8-bit) in the
// bf16 exponent.
#include <algorithm>
#include <cstring>
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace mxs {

__device__ int g_decode_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

constexpr int kQuads = 4;                                         // worker quads
constexpr int kQuadWarps = 5;                                     // four converters + one MMA issuer
constexpr int kWorkerWarp0 = 5;                                   // warps 5..24
constexpr int kThreads = (kWorkerWarp0 + kQuadWarps * kQuads) * 32;  // 800
constexpr int kTokBytes = 16 * 128;                       // 16 token rows x 128 bytes of K'
constexpr int kAccCols = 16;                              // one accumulator: 16 token columns
// tensor-memory columns: quad j's A tiles at kACol + 32 (2j + buf), its
// accumulators at kAccCol + 16 (2j + b), its weight / token scale columns at
// kSfaCol / kSfbCol + 4 (2j + buf)
constexpr int kACol = 0, kAccCol = 256, kSfaCol = 384, kSfbCol = 416, kTmemCols = 512;
constexpr int kXBytes = 128 * 16 * 4;  // one fp32 partial tile
constexpr int kMinSmem = 116 * 1024;   // one CTA per SM (each allocates all of tensor memory)
constexpr int kQuadBar0 = 8;           // named barriers 8..11: one per quad
constexpr int kCodesBar = 12;          // named barrier of the token prologue (codes mode)
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock
#ifndef MXS_POLL_SLEEP_NS
#define MXS_POLL_SLEEP_NS 64
#endif
// the producer warp's pause after a pass over its slots that moved nothing:
// its polling would otherwise take issue slots from the converter warps
constexpr unsigned kPollSleepNs = MXS_POLL_SLEEP_NS;

struct DecodeArgs {
    const uint8_t *codes;   // [M, row_bytes] packed activation codes (codes mode)
    const uint8_t *scales;  // [M, nb]
    const uint8_t *tok_sf;  // activation scale tiles of the planes buffer (planes mode), else NULL
    const uint8_t *w;       // packed weight buffer
    float *y;
    int64_t ld_y;
    int M, N, G;           // tokens, output features, 128-row groups
    int GS;                // CTAs per cluster along K
    int bound[9];          // rank r owns slots [bound[r], bound[r+1]) (stage-aligned)
    int max_mst;           // most MMA stages any rank holds (token operand carve)
    int ring, slot_bytes;  // copy chunks in flight, bytes per ring slot (a multiple of 1024)
    int w_off;             // weights' offset in a slot: after the streamed token tiles (planes mode), else 0
    int accumulate;        // add into y (a later K pass) instead of storing
    int starve;            // test hook: > 0 makes every CTA skip the weight copy of its chunk starve-1
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
// non-blocking test of a phase (try_wait may suspend the thread for a while
// when the phase is not complete: wrong for a loop that serves two barriers)
__device__ __forceinline__ bool test_phase(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
#ifndef MXS_DEC_SLEEP_NS
#define MXS_DEC_SLEEP_NS 0
#endif
template <bool kCluster = false>
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (poll<kCluster>(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (MXS_DEC_SLEEP_NS > 0) __nanosleep(MXS_DEC_SLEEP_NS);
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
// generic-proxy shared-memory writes -> visible to the tensor core / bulk copies
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
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
// relaxed: the barrier inits are published by fence.mbarrier_init.release.cluster,
// and the teardown only needs every rank's arrival (each receive barrier already
// proves that the copies into it have landed)
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory"); }
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
// kind::f16, bf16 x bf16, K-major, N = 16, M = 128, f32 accumulator
constexpr uint32_t kIdescF16 =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(16 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
// the bf16 MMA with the A operand in tensor memory (K-major: row i in lane i,
// two 16-bit elements per 32-bit column)
__device__ __forceinline__ void mma_f16_t(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %4, p;\n}" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(accum), "r"(kIdescF16)
        : "memory");
}
// the same with the A operand in tensor memory (K-major: row i in lane i, four
// 8-bit elements per 32-bit column)
__device__ __forceinline__ void mma_mx_t(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t id, uint32_t sfa,
                                         uint32_t sfb, uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%5], [%6], p;\n}" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(id), "r"(accum), "r"(sfa), "r"(sfb)
        : "memory");
}
// 32 consecutive 32-bit columns of this thread's lane
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

// e4m3 bytes (sign << 7) | |m| of the four low / four high
// sign-magnitude nibbles (s << 3) | |m| held in a word
__device__ __forceinline__ uint32_t lo_nib(uint32_t w) { return (w & 0x07070707u) | ((w << 4) & 0x80808080u); }
__device__ __forceinline__ uint32_t hi_nib(uint32_t w) { return ((w >> 4) & 0x07070707u) | (w & 0x80808080u); }
// bf16 pair of two 7-bit sign-magnitude codes (s << 7) | m spread by prmt
// into the 16-bit lanes of t (the code in the low byte, its sign replicated
// in the high one): with eb = E in each lane's exponent field, (s | E | m) -
// (s | E) = +-m * 2^(E-134), exact (a NaN when eb holds the NaN pattern)
__device__ __forceinline__ uint32_t bf16_codes(uint32_t t, uint32_t eb) {
    const uint32_t y = (t & 0x807F807Fu) | eb;
    const uint32_t o = (t & 0x80008000u) | eb;
    uint32_t d;
    asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(o), "r"(0xBF80BF80u), "r"(y));  // y - o
    return d;
}
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
// four scale bytes carrying their codes' fixed-point weights (shift per byte
// in `add`), saturating at 254; 255 (NaN) stays
__device__ __forceinline__ uint32_t shifted4(uint32_t S4, uint32_t add) {
    const uint32_t t = __vminu4(__vaddus4(S4, add), 0xFEFEFEFEu);
    return t | __vcmpeq4(S4, 0xFFFFFFFFu);
}

// y[t][n] for the M tokens.  The two cases are separate loops so that the
// plain store never waits for a read of y (a select between "y + v" and "v"
// would let the compiler load y for every store); a later K pass adds into
// the y that the same thread stored in the pass before.
__device__ __forceinline__ void store_y(const DecodeArgs &a, int n, const float (&v)[16]) {
    float *col = a.y + n;
    if (a.accumulate) {
#pragma unroll
        for (int t = 0; t < 16; ++t)
            if (t < a.M) col[(int64_t)t * a.ld_y] += v[t];
    } else {
#pragma unroll
        for (int t = 0; t < 16; ++t)
            if (t < a.M) col[(int64_t)t * a.ld_y] = v[t];
    }
}

// The counts of the grouping plan that the kernel reads.  The kernel's
// parameters hold these and the launch arguments side by side (a few hundred
// bytes): the first reads of a launch miss the constant cache, and the whole
// plan with its slot table would spread them over 4 KB.
struct PlanCounts {
    int nb, n4, n6, n8, n68;
    int st4, nst;
    int64_t row_bytes, kp;
};
// A launch holds up to kMaxProblems independent GEMMs (the projections of a
// decoder layer that share an input): problem i owns the CTAs
// [cta0, cta0 + ncta) along x, and a cluster (along y) never spans two.
constexpr int kMaxProblems = 3;
struct DecodeProblem {
    PlanCounts p;
    DecodeArgs a;
    int cta0, ncta;
};
struct DecodeParams {
    DecodeProblem prob[kMaxProblems];
    int nprob;
};

struct Stages {  // MMA stages of a CTA's K range [c0, c1): 4-bit ones (4 slots), then 6/8-bit ones (2 slots)
    int a4, e4, a8, e8, st4, n;
    __device__ void init(const PlanCounts &p, int c0, int c1) {
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

__global__ void __launch_bounds__(kThreads, 1) gemm_decode_kernel(const __grid_constant__ DecodeParams dp,
                                                                  const __grid_constant__ CUtensorMap map0,
                                                                  const __grid_constant__ CUtensorMap map1,
                                                                  const __grid_constant__ CUtensorMap map2) {
    // the problem this CTA serves, and its CTA index and count within it
    int pi = 0;
    while (pi + 1 < dp.nprob && (int)blockIdx.x >= dp.prob[pi + 1].cta0) ++pi;
    const PlanCounts &p = dp.prob[pi].p;
    const DecodeArgs &a = dp.prob[pi].a;
    const int bx = (int)blockIdx.x - dp.prob[pi].cta0, gx = dp.prob[pi].ncta;
    const CUtensorMap *tok_map = pi == 0 ? &map0 : (pi == 1 ? &map1 : &map2);
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sbase = su32(smem_raw);
    uint8_t *smem = smem_raw + (((sbase + 1023) & ~1023u) - sbase);  // 1024-aligned for the swizzled tiles
    // ring slot: [two token tiles (planes mode)][their two scale tiles][compact weight chunk]
    uint8_t *ring = smem;                                        // ring x slot_bytes
    uint8_t *tok = ring + (size_t)a.ring * a.slot_bytes;         // codes mode: max_mst x 2 KB resident token planes
    uint8_t *sfb = tok + (size_t)a.max_mst * kTokBytes;          // codes mode: max_mst x 512 token scale tiles
    uint8_t *sfa = sfb + (size_t)a.max_mst * 512;                // kQuads x 2 x 512 weight scale tiles
    // cluster reduce-scatter: rank k adds up rows [k*R, (k+1)*R) of the GS partial
    // tiles (R = 128/GS) and stores them; xout is this rank's whole partial tile,
    // xbuf the slices the other ranks send here (slot of sender j: j, or j-1 past k)
    const int R = 128 / a.GS;
    float *xout = reinterpret_cast<float *>(sfa + kQuads * 2 * 512);  // [128][16] (GS > 1)
    float *xbuf = xout + (a.GS > 1 ? 128 * 16 : 0);                                 // [GS-1][R][16]
    uint64_t *bars = reinterpret_cast<uint64_t *>(xbuf + (size_t)(a.GS - 1) * R * 16);
    // a ring slot's weight bytes (full_c / empty_c: the converters have loaded
    // them) and its token tiles (full_t / empty_t: the MMAs have read them) are
    // filled and released separately, so the next weights stream in while the
    // MMAs of the chunk before are still pending
    uint64_t *full_c = bars, *empty_c = full_c + a.ring, *full_t = empty_c + a.ring, *empty_t = full_t + a.ring;
    uint64_t *a_free = empty_t + a.ring;  // [kQuads][2] tcgen05.commit
    uint64_t *a_full = a_free + 2 * kQuads;  // [kQuads][2] the four converter warps
    uint64_t *acc_full = a_full + 2 * kQuads, *acc_empty = acc_full + 2;
    uint64_t *tok_full = acc_empty + 2;
    uint64_t *xfull = tok_full + 1, *xempty = xfull + 1, *xstage = xempty + 1, *xread = xstage + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(xread + 1);
    int *abort_flag = reinterpret_cast<int *>(tmem_slot + 1);
    volatile int *abort = abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = a.GS > 1 ? cg::this_cluster().block_rank() : 0;
    const int c0 = a.bound[rank], c1 = a.bound[rank + 1];
    const bool from_planes = a.tok_sf != nullptr;
    Stages S;
    S.init(p, c0, c1);
    const int nchunks = (S.n + 1) / 2;          // a copy chunk holds two MMA stages
    const int nq = min(kQuads, nchunks);        // quads with a chunk in every group
    const int ngroups = bx < a.G ? (a.G - 1 - bx) / gx + 1 : 0;
    const int total = ngroups * nchunks;        // chunks this CTA streams
    const uint32_t xslice = (uint32_t)(R * 16 * 4);
    const int sg0 = c0 < p.n4 ? c0 / 4 : p.st4 + (c0 - p.n4) / 2;  // the rank's first stage in the planes

    // chunk qc (in streaming order): group bx + (qc / nchunks) * gx,
    // stages 2k, 2k+1 with k = qc % nchunks; it goes to ring slot qc % ring and is
    // converted by quad qc % kQuads (ring is a multiple of kQuads, so each slot
    // has one consumer, which takes its slots in order)
    auto issue = [&](int qc) {
        if (a.starve == qc + 1) return;  // test hook: this chunk never arrives (its converters' wait runs out)
        const int gi = qc / nchunks, k = qc - gi * nchunks;
        const int s = qc % a.ring;
        int lo, hi, lo2, hi2;
        S.range(2 * k, lo, hi);
        if (2 * k + 1 < S.n) S.range(2 * k + 1, lo2, hi2); else hi2 = hi;
        const int64_t off = slot_offset(p, lo);
        const uint32_t bytes = (uint32_t)(slot_offset(p, hi2) - off);
        const uint8_t *wg = a.w + (int64_t)(bx + gi * gx) * a.GB;
        mbar_expect_tx(&full_c[s], bytes);
        bulk_load(ring + (size_t)s * a.slot_bytes + a.w_off, wg + off, bytes, &full_c[s]);
    };
    // planes mode: the token operand of chunk qc's stages, by TMA from the planes
    auto issue_tok = [&](int qc) {
        const int k = qc % nchunks, s = qc % a.ring;
        const int nst = min(2, S.n - 2 * k);
        uint8_t *slot = ring + (size_t)s * a.slot_bytes;
        mbar_expect_tx(&full_t[s], (uint32_t)nst * (kTokBytes + 512));
        for (int i = 0; i < nst; ++i) tma_load_2d(slot + i * kTokBytes, tok_map, &full_t[s], 128 * (sg0 + 2 * k + i), 0);
        bulk_load(slot + 2 * kTokBytes, a.tok_sf + (int64_t)(sg0 + 2 * k) * 512, (uint32_t)nst * 512, &full_t[s]);
    };

    // the next kernel on the stream may launch now (it waits for this grid
    // before it touches what this grid writes)
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (threadIdx.x == 0) {
        for (int i = 0; i < a.ring; ++i) {
            mbar_init(&full_c[i], 1);
            mbar_init(&empty_c[i], 4);  // the quad's four converter warps have loaded the chunk
            mbar_init(&full_t[i], 1);
            mbar_init(&empty_t[i], 1);  // tcgen05.commit after the chunk's MMAs
        }
        for (int i = 0; i < 2 * kQuads; ++i) {
            mbar_init(&a_free[i], 1);
            mbar_init(&a_full[i], 4);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], nq);  // each quad with a chunk in the group commits once
            mbar_init(&acc_empty[i], 4);  // the four epilogue warps
        }
        mbar_init(tok_full, from_planes ? 1 : 4);
        mbar_init(xfull, 1);                  // armed per tile with the bytes of GS-1 slices
        mbar_init(xempty, max(1, a.GS - 1));  // every receiver took this rank's previous slices (copies done)
        mbar_init(xstage, 4);                 // the four epilogue warps have staged the partial tile
        mbar_init(xread, 4);                  // the four epilogue warps are done with xout and xbuf
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (a.GS > 1) mbar_expect_tx(xfull, (uint32_t)(a.GS - 1) * xslice);  // the first tile's slices
    }
    if (warp == 0) {
        __syncwarp();
        // the weights are static (see mxs_linear_decode): fill the ring right away,
        // one chunk per lane
        if (lane < min(a.ring, total)) issue(lane);
        __syncwarp();
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
        // ------------------------------------------------------------ producer: the rest of the chunks
        if (from_planes) {
            // the planes may come from the kernel just before this one (programmatic
            // dependent launch): wait for it before the first token load
            asm volatile("griddepcontrol.wait;" ::: "memory");
            if (lane < min(a.ring, total)) issue_tok(lane);  // the first chunks' tokens, one per lane
        }
        // Refills.  Bulk copies issued by one thread are served one after
        // another (about 0.3 us each on GB300, whatever their size), so each
        // quad's chunks get their own issuing lane: lane j (< 4) sends the
        // weights of chunks qc = j mod 4 once the quad's converters have loaded
        // chunk qc - ring, lane 4 + j their token tiles once the MMAs of chunk
        // qc - ring have run.  The lanes poll in step without blocking; a stall
        // of kWaitCycles with no lane moving gives up.
        const int role = lane < 4 ? 0 : (lane < 8 && from_planes ? 1 : 2);  // 0 weights, 1 tokens, 2 idle
        int nx = a.ring + (lane & 3);  // the next chunk this lane refills
        if (role == 2) nx = total;
        long long t0 = clock64();
        while (__any_sync(0xffffffffu, nx < total)) {
            bool moved = false;
            if (nx < total) {
                const uint32_t par = ((nx / a.ring) & 1) ^ 1;
                if (role == 0 ? test_phase(&empty_c[nx % a.ring], par) : test_phase(&empty_t[nx % a.ring], par)) {
                    if (role == 0) issue(nx); else issue_tok(nx);
                    nx += kQuads;
                    moved = true;
                }
            }
            if (__any_sync(0xffffffffu, moved)) {
                t0 = clock64();
            } else if (*abort) {
                break;
            } else if (clock64() - t0 > kWaitCycles) {
                if (lane == 0) {
                    *abort = 1;
                    atomicExch(&g_decode_status, MXS_ERR_TIMEOUT);
                }
                break;
            } else if (kPollSleepNs > 0) {
                __nanosleep(kPollSleepNs);
            }
        }
        // copies still in flight land in shared memory before the CTA exits:
        // each lane waits for the latest chunk of each of its slots (its
        // residue's last ring / kQuads chunks that exist)
        if (role != 2)
            for (int qc = nx - kQuads, n = 0; qc >= 0 && n < a.ring / kQuads; qc -= kQuads, ++n)
                if (qc < total && !(role == 0 && a.starve == qc + 1))
                    drain_wait(role == 0 ? &full_c[qc % a.ring] : &full_t[qc % a.ring], (qc / a.ring) & 1);
    } else if (warp >= kWorkerWarp0) {
        // ------------------------------------------------------------ worker quads
        // quad j = warps 5+5j .. 9+5j: four converters (one per tensor-memory lane
        // quarter) and one MMA issuer; all five meet at the quad's barrier once per stage
        const int wq = warp - kWorkerWarp0;
        const int j = wq / kQuadWarps, role = wq % kQuadWarps;  // role 4: the issuer
        const int qtr = warp & 3;                                // a converter's lane quarter
        const int r = 32 * qtr + lane;                           // its weight row within the group
        const uint32_t a_lane = (uint32_t)(32 * qtr) << 16;
        uint8_t *sfa_q = sfa + j * 1024;  // two 512-byte tiles
        const uint64_t dB = desc_sw128(su32(tok)), dsfa = desc_sf(su32(sfa_q)), dsfb = desc_sf(su32(sfb));
        bool ok = true, tok_seen = false, stop = false;
        uint32_t qw = 0;  // stages this quad has issued (a_free phases)
        for (int qc = j; qc < total && !stop; qc += kQuads) {
            const int gi = qc / nchunks, k = qc - gi * nchunks, b = gi & 1;
            const int s = qc % a.ring;
            if (ok && role < 4) ok = warp_wait(&full_c[s], (qc / a.ring) & 1, abort);
            uint8_t *slot_base = ring + (size_t)s * a.slot_bytes;
            int clo, chi;
            S.range(2 * k, clo, chi);
            const uint8_t *chunk = slot_base + a.w_off - slot_offset(p, clo);  // + slot_offset(slot)
            const bool first_chunk = k < kQuads;           // the quad's first chunk of the group
            const bool last_chunk = k + kQuads >= nchunks;  // ... and its last
            const int st_end = min(2 * k + 2, S.n);
            for (int st = 2 * k; st < st_end; ++st, ++qw) {
                const int buf = qw & 1;
                if (role < 4) {
                    // the A tile and scale tile of this buffer are free once the MMAs of two stages ago ran
                    if (ok && qw >= 2) ok = warp_wait(&a_free[2 * j + buf], ((qw >> 1) - 1) & 1, abort);
                    if (ok) {
                        int lo, hi;
                        S.range(st, lo, hi);
                        const int nsl = hi - lo;                      // slots present in the stage
                        const uint8_t *s0 = chunk + slot_offset(p, lo);  // its first slot
                        uint32_t d[32], sfw;
                        if (st < S.st4) {
                            // all loads first: four 16-byte code words and four scale bytes of row r
                            uint4 v[4];
                            uint32_t sb = 0;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                v[q] = make_uint4(0, 0, 0, 0);
                                if (q < nsl) {
                                    v[q] = *reinterpret_cast<const uint4 *>(s0 + 2176 * q + 16 * r);
                                    sb |= (uint32_t)s0[2176 * q + 2048 + r] << (8 * q);
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
                            sfw = shifted4(sb, 0x07070707u);
                        } else {
                            // two 6/8-bit slots as bf16 values m * 2^(Sw-127-(b-2)) (the scale inside,
                            // no scale tile): row r's 32 codes of slot h at K' bytes 64h .. 64h+63
#pragma unroll
                            for (int h = 0; h < 2; ++h) {
                                uint4 v0 = make_uint4(0, 0, 0, 0), v1 = v0;
                                uint32_t eb = (1u << 7) | (1u << 23);  // absent slot: zeros
                                if (h < nsl) {
                                    v0 = *reinterpret_cast<const uint4 *>(s0 + 4224 * h + 32 * r);
                                    v1 = *reinterpret_cast<const uint4 *>(s0 + 4224 * h + 32 * r + 16);
                                    const int Sw = s0[4224 * h + 4096 + r];
                                    // exponent field E = Sw + 7 - (b - 2), so that m * 2^(E-134) is the value
                                    const uint32_t E = (uint32_t)min(Sw + 9 - slot_width(p, lo + h), 254);
                                    eb = Sw == 255 ? 0x7FC07FC0u : (E << 7) | (E << 23);
                                }
                                const uint32_t w[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
                                for (int i = 0; i < 8; ++i) {  // word i: elements 4i .. 4i+3
                                    d[16 * h + 2 * i] = bf16_codes(prmt(w[i], 0u, 0x9180u), eb);
                                    d[16 * h + 2 * i + 1] = bf16_codes(prmt(w[i], 0u, 0xB3A2u), eb);
                                }
                            }
                            sfw = 0;
                        }
                        if (st == st_end - 1) {
                            // the chunk's last stage is in registers: its weight bytes are free
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&empty_c[s]);
                        }
                        // absent slots: zero values (their scale bytes do not matter)
                        // the row's 128 K' bytes into its lane of the quad's A tile (32 columns)
                        tmem_st32(tmem + a_lane + kACol + 32 * (2 * j + buf), d);
                        // scale tile: row r = 32 qtr + lane at lane `lane`, column qtr; byte = sf id
                        *reinterpret_cast<uint32_t *>(sfa_q + buf * 512 + lane * 16 + qtr * 4) = sfw;
                        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                        fence_async_smem();
                        fence_before();
                    }
                }
                if (role < 4) {
                    // this warp's 32 rows of the stage are in tensor memory: tell the
                    // issuer, and go on to the next stage without waiting for it
                    __syncwarp();
                    if (ok && lane == 0) mbar_arrive(&a_full[2 * j + buf]);
                    if (!ok) {
                        stop = true;
                        break;
                    }
                } else {
                    if (lane == 0) {
                        // the four converter warps have written the stage
                        bool go = mbar_wait(&a_full[2 * j + buf], (qw >> 1) & 1, abort);
                        // planes mode: the chunk's token tiles have landed
                        if (go && from_planes && st == 2 * k) go = mbar_wait(&full_t[s], (qc / a.ring) & 1, abort);
                        if (go && !tok_seen && !from_planes) {
                            go = mbar_wait(tok_full, 0, abort);  // the resident token operand is built
                            tok_seen = true;
                        }
                        const bool first = first_chunk && st == 2 * k;
                        if (go && first) go = mbar_wait(&acc_empty[b], ((gi >> 1) & 1) ^ 1, abort);
                        if (go) {
                            fence_after();
                            const uint32_t sfa_t = tmem + kSfaCol + 4 * (2 * j + buf);
                            const uint32_t sfb_t = tmem + kSfbCol + 4 * (2 * j + buf);
                            if (st < S.st4) {
                                tmem_cp_sf(sfa_t, dsfa + 32 * buf);
                                // token scales: the chunk's tile (planes mode) or the resident one
                                tmem_cp_sf(sfb_t, from_planes ? desc_sf(su32(slot_base + 2 * kTokBytes)) +
                                                                    32 * (st - 2 * k)
                                                              : dsfb + 32 * st);
                            }
                            const uint32_t acc = tmem + kAccCol + kAccCols * (2 * j + b);
                            const uint32_t aT = tmem + kACol + 32 * (2 * j + buf);
                            const uint64_t db = from_planes
                                                    ? desc_sw128(su32(slot_base)) + (uint64_t)((st - 2 * k) * (kTokBytes >> 4))
                                                    : dB + (uint64_t)(st * (kTokBytes >> 4));
                            const uint32_t accum = first ? 0u : 1u;
                            if (st < S.st4) {
                                // slot q: weight values at columns 8q.. (K' bytes 32q..), token values at 32q..
                                mma_mx_t(acc, aT, db, idesc(0, 0), sfa_t, sfb_t, accum);
                                mma_mx_t(acc, aT + 8, db + 2, idesc(1, 1), sfa_t, sfb_t, 1u);
                                mma_mx_t(acc, aT + 16, db + 4, idesc(2, 2), sfa_t, sfb_t, 1u);
                                mma_mx_t(acc, aT + 24, db + 6, idesc(3, 3), sfa_t, sfb_t, 1u);
                            } else {
                                // two 6/8-bit slots as bf16 values on both sides (scales inside):
                                // four K = 16 MMAs over K' bytes 32q .. 32q+31
                                mma_f16_t(acc, aT, db, accum);
                                mma_f16_t(acc, aT + 8, db + 2, 1u);
                                mma_f16_t(acc, aT + 16, db + 4, 1u);
                                mma_f16_t(acc, aT + 24, db + 6, 1u);
                            }
                            mma_commit(&a_free[2 * j + buf]);  // A tile + scale tiles free once read
                            if (from_planes && st == st_end - 1) mma_commit(&empty_t[s]);  // token tiles free once read
                            if (last_chunk && st == st_end - 1) mma_commit(&acc_full[b]);  // the quad's share is issued
                        } else {
                            ok = false;
                        }
                    }
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        stop = true;
                        break;
                    }
                }
            }
        }
        if (role == 4 && lane == 0 && qw > 0) drain_wait(&a_free[2 * j + ((qw - 1) & 1)], ((qw - 1) >> 1) & 1);
    } else {
        // ------------------------------------------------------------ warps 1-4: token operand, epilogue
        const int et = threadIdx.x - 32;  // 0..127
        // codes mode: build the resident token operand (planes mode streams it with the chunks)
        if (!from_planes) {
            // the codes may come from the kernel just before this one
            asm volatile("griddepcontrol.wait;" ::: "memory");
            // zero the token planes and scale tiles of every stage, then fill them from the codes
            for (int i = et; i < S.n * (kTokBytes + 512) / 16; i += 128) {
                const int off = i * 16;
                uint8_t *dst = off < S.n * kTokBytes ? tok + off : sfb + (off - S.n * kTokBytes);
                *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
            }
            named_sync(kCodesBar, 128);
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
                // the plane form: m/4 (4-bit, block-scaled), or the bf16 values
                // m * 2^(Sa-127-(b-2)) (6/8-bit; NaN for a NaN block)
                uint32_t d0[8], d1[8];
                const float fv = b == 4 ? 0.25f : (Sa == 255 ? __int_as_float(0x7FC00000) : pow2f((int)Sa - 125 - b));
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (b == 4) {
                        d0[i] = e4m3x2(fv * m[4 * i], fv * m[4 * i + 1]) |
                                ((uint32_t)e4m3x2(fv * m[4 * i + 2], fv * m[4 * i + 3]) << 16);
                        d1[i] = 0;
                    } else {
                        d0[i] = bf16x2(fv * m[2 * i], fv * m[2 * i + 1]);            // elements 0..15
                        d1[i] = bf16x2(fv * m[16 + 2 * i], fv * m[17 + 2 * i]);      // elements 16..31
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

        // epilogue: accumulator row (= weight row) 32*qtr + lane, columns = tokens;
        // the quads' partial sums are added in quad order
        if (a.GS > 1) cluster_wait();
        const int qtr = warp & 3;
        const int r = 32 * qtr + lane;
        // cluster mode: the group whose slices the receive barrier is armed for
        // and this CTA has not yet taken (-1: none).  Partners may send them
        // whatever state this CTA is in, so a CTA that gives up waits (bounded)
        // for them before it leaves: no copy may land in a CTA that has exited.
        int rx_gi = a.GS > 1 ? 0 : -1;
        int gi = 0;
        for (int g = bx; g < a.G; g += gx, ++gi) {
            const int b = gi & 1;
            if (!warp_wait(&acc_full[b], (gi >> 1) & 1, abort)) break;
            fence_after();
            float out[16];
            bool first = true;
            for (int jq = 0; jq < kQuads; ++jq) {
                // quads holding a chunk of this group: (gi * nchunks + k) % kQuads for k < nq
                if (((jq - gi * nchunks) % kQuads + kQuads) % kQuads >= nq) continue;
                uint32_t v[16];
                tmem_ld16(tmem + ((uint32_t)(32 * qtr) << 16) + kAccCol + kAccCols * (2 * jq + b), v);
#pragma unroll
                for (int t = 0; t < 16; ++t) out[t] = first ? __uint_as_float(v[t]) : out[t] + __uint_as_float(v[t]);
                first = false;
            }
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);
            const bool more = g + gx < a.G;  // another group follows
            if (a.GS == 1) {
                const int n = 128 * g + r;
                if (n < a.N) store_y(a, n, out);
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
            rx_gi = -1;
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
                if (n < a.N) store_y(a, n, sum);
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
                rx_gi = gi + 1;
            }
        }
        // gave up with the receive barrier armed: the slices partners have sent
        // (or still send) land before this CTA exits
        if (rx_gi >= 0 && et == 0) drain_wait(xfull, rx_gi & 1);
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
    int GS, max_mst, most, grid, ring, slot_bytes, w_off;  // most: stages of the largest rank range
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

DecodeShape shape_for(const Plan &p, int GS, int64_t G, int sms, int g0, int g1, bool stream_tok) {
    DecodeShape sh = {};
    sh.GS = GS;
    int gb[9];
    if (!split_stages(p, g0, g1, GS, gb)) return sh;
    int max_copy = 0;
    for (int r = 0; r <= GS; ++r) sh.bound[r] = stage_lo(p, gb[r]);
    for (int r = 0; r < GS; ++r) {
        sh.max_mst = std::max(sh.max_mst, gb[r + 1] - gb[r]);
        for (int k = gb[r]; k < gb[r + 1]; k += 2) {  // chunks of two stages
            const int e = std::min(k + 2, gb[r + 1]);
            max_copy = std::max(max_copy, (int)(slot_offset(p, stage_lo(p, e)) - slot_offset(p, stage_lo(p, k))));
        }
    }
    // planes mode streams two token tiles and their scale tiles with every chunk;
    // codes mode keeps the rank's whole token operand resident
    sh.w_off = stream_tok ? 2 * (kTokBytes + 512) : 0;
    sh.slot_bytes = (sh.w_off + max_copy + 1023) / 1024 * 1024;
    const int resident = stream_tok ? 0 : sh.max_mst;
    // partial tile + (GS-1) received slices of 128/GS rows
    const size_t xbytes = GS > 1 ? (size_t)kXBytes + (size_t)(GS - 1) * (kXBytes / GS) : 0;
    const size_t fixed = 1024 + (size_t)resident * (kTokBytes + 512) + (size_t)kQuads * 1024 + xbytes + 512;
    // The ring holds 8 or 4 chunks: a multiple of kQuads, so that slot s is
    // only ever used by quad s % kQuads, which consumes its slots strictly in
    // order.  A slot shared by quads could be polled for its next phase while
    // its previous chunk is still in flight, and a parity wait would then
    // pass early.
    const size_t budget = 225 * 1024;
    sh.ring = fixed + 8 * (size_t)sh.slot_bytes <= budget ? 8 : (fixed + 4 * (size_t)sh.slot_bytes <= budget ? 4 : 0);
    sh.smem = std::max<size_t>(kMinSmem, fixed + (size_t)sh.ring * sh.slot_bytes + 32 * (size_t)sh.ring);
    sh.most = sh.max_mst;
    if (stream_tok) sh.max_mst = 0;  // no resident token operand
    sh.ok = sh.ring >= kQuads && sh.smem <= 225 * 1024 + 1024;
    sh.grid = (int)std::min<int64_t>(G, std::max(1, sms / GS));
    return sh;
}

// Choose the K split.  A CTA's time is about (groups it owns) x (copy chunks
// a quad converts per group + a fixed cost per group).  In a cluster every
// group after the first also waits for the previous group's cross-rank
// exchange, which measured at 8-13 us on GB300, so clusters pay off only when
// their CTAs own one group each.  Ties go to the smaller cluster.
DecodeShape pick_shape(const Plan &p, int64_t G, int sms, int g0, int g1, bool stream_tok) {
    DecodeShape best = {};
    double best_cost = 1e30;
    for (int GS = 1; GS <= 8 && GS <= g1 - g0; GS *= 2) {
        const DecodeShape sh = shape_for(p, GS, G, sms, g0, g1, stream_tok);
        if (!sh.ok) continue;
        const double rounds = (double)((G + sh.grid - 1) / sh.grid);
        const int nchunks = (sh.most + 1) / 2;
        const double cost = rounds * ((nchunks + kQuads - 1) / kQuads + 1.0) + (GS > 1 ? 0.3 + 8.0 * (rounds - 1.0) : 0.0);
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

PlanCounts counts_of(const Plan &p) {
    PlanCounts c;
    c.nb = p.nb, c.n4 = p.n4, c.n6 = p.n6, c.n8 = p.n8, c.n68 = p.n68;
    c.st4 = p.st4, c.nst = p.nst, c.row_bytes = p.row_bytes, c.kp = p.kp;
    return c;
}

// chunk rounds of a problem with `ncta` CTAs (the decode cost model: a CTA's
// groups one after another, four quads per group, the cluster exchange per
// extra group)
double problem_cost(const DecodeShape &sh, int64_t G, int ncta) {
    const double rounds = (double)((G + ncta - 1) / ncta);
    const int nchunks = (sh.most + 1) / 2;
    return rounds * ((nchunks + kQuads - 1) / kQuads + 1.0) + (sh.GS > 1 ? 0.3 + 8.0 * (rounds - 1.0) : 0.0);
}

}  // namespace

int64_t decode_workspace_bytes(const Plan &, int64_t, int64_t) { return 0; }

int launch_gemm_decode_group(const Plan *const *plans, const void *const *act_planes, const void *const *packed,
                             const int64_t *N, float *const *y, const int64_t *ld_y, int count, int64_t M, bool pdl,
                             cudaStream_t st) {
    if (count < 1 || count > kMaxProblems) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d)", count, kMaxProblems);
    const int sms = sm_count();
    int64_t G[kMaxProblems];
    for (int i = 0; i < count; ++i) {
        if (N[i] > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
        G[i] = weight_offsets(*plans[i], N[i], false).G;
    }
    // one cluster size for the launch; CTAs handed one at a time to the
    // problem whose share currently costs most
    double best_cost = 1e30;
    DecodeShape best_sh[kMaxProblems];
    int best_n[kMaxProblems] = {};
    for (int GS = 1; GS <= 8; GS *= 2) {
        DecodeShape sh[kMaxProblems];
        bool ok = sms / GS >= count;
        for (int i = 0; i < count && ok; ++i) {
            ok = GS <= plans[i]->nst;
            if (ok) sh[i] = shape_for(*plans[i], GS, G[i], sms, 0, plans[i]->nst, true);
            ok = ok && sh[i].ok;
        }
        if (!ok) continue;
        int n[kMaxProblems], used = count;
        for (int i = 0; i < count; ++i) n[i] = 1;
        while (used < sms / GS) {
            int worst = -1;
            double wc = -1.0;
            for (int i = 0; i < count; ++i)
                if (n[i] < G[i] && problem_cost(sh[i], G[i], n[i]) > wc) wc = problem_cost(sh[i], G[i], n[i]), worst = i;
            if (worst < 0) break;
            ++n[worst];
            ++used;
        }
        double cost = 0.0;
        for (int i = 0; i < count; ++i) cost = std::max(cost, problem_cost(sh[i], G[i], n[i]));
        if (cost < best_cost - 1e-9) {
            best_cost = cost;
            for (int i = 0; i < count; ++i) best_sh[i] = sh[i], best_n[i] = n[i];
        }
    }
    if (best_cost >= 1e29) return -1;  // no common plan: the caller launches the problems one by one
    DecodeParams dp = {};
    dp.nprob = count;
    CUtensorMap maps[kMaxProblems];
    size_t smem = 0;
    int cta = 0;
    for (int i = 0; i < count; ++i) {
        const Plan &p = *plans[i];
        const DecodeShape &sh = best_sh[i];
        DecodeArgs a = {};
        a.w = static_cast<const uint8_t *>(packed[i]);
        a.y = y[i];
        a.ld_y = ld_y[i];
        a.M = (int)M;
        a.N = (int)N[i];
        a.G = (int)G[i];
        a.GB = weight_offsets(p, N[i], false).GB;
        std::memset(&maps[i], 0, sizeof(CUtensorMap));
        const int rc = make_plane_map(&maps[i], act_planes[i], M, p.kp, 16);
        if (rc) return rc;
        a.tok_sf = static_cast<const uint8_t *>(act_planes[i]) + align256(M * p.kp);
        a.GS = sh.GS;
        for (int r = 0; r < 9; ++r) a.bound[r] = r <= sh.GS ? sh.bound[r] : sh.bound[sh.GS];
        a.max_mst = sh.max_mst;
        a.ring = sh.ring;
        a.slot_bytes = sh.slot_bytes;
        a.w_off = sh.w_off;
        a.accumulate = 0;
        dp.prob[i].p = counts_of(p);
        dp.prob[i].a = a;
        dp.prob[i].cta0 = cta;
        dp.prob[i].ncta = best_n[i];
        cta += best_n[i];
        smem = std::max(smem, sh.smem);
    }
    for (int i = count; i < kMaxProblems; ++i) maps[i] = maps[0];
    const int GS = best_sh[0].GS;
    cudaError_t e = cudaFuncSetAttribute(gemm_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cta, (unsigned)GS, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    int na = 0;
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = (unsigned)GS;
    attr[na].val.clusterDim.z = 1;
    ++na;
    if (pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    e = cudaLaunchKernelEx(&cfg, gemm_decode_kernel, dp, maps[0], maps[1], maps[2]);
    return cuda_fail(e, "gemm_decode_kernel launch");
}

int launch_gemm_decode(const Plan &p, const void *codes, const uint8_t *scales, const void *act_planes,
                       const void *packed, int64_t M, int64_t N, float *y, int64_t ld_y, bool pdl, cudaStream_t st,
                       int starve) {
    if (N > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
    DecodeArgs a = {};
    a.starve = starve;
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
            plan[k] = pick_shape(p, a.G, sm_count(), win[k], win[k + 1], act_planes != nullptr);
            ok = plan[k].ok;
        }
        if (!ok) continue;
        for (int k = 0; k < passes; ++k) {
            const DecodeShape &sh = plan[k];
            a.GS = sh.GS;
            for (int i = 0; i < 9; ++i) a.bound[i] = i <= sh.GS ? sh.bound[i] : sh.bound[sh.GS];
            a.max_mst = sh.max_mst;
            a.ring = sh.ring;
            a.slot_bytes = sh.slot_bytes;
            a.w_off = sh.w_off;
            a.accumulate = k > 0;
            cudaError_t e =
                cudaFuncSetAttribute(gemm_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(decode smem)");
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3((unsigned)sh.grid, (unsigned)sh.GS, 1);
            cfg.blockDim = dim3(kThreads, 1, 1);
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
            DecodeParams dp = {};
            dp.nprob = 1;
            dp.prob[0].p = counts_of(p);
            dp.prob[0].a = a;
            dp.prob[0].cta0 = 0;
            dp.prob[0].ncta = sh.grid;
            e = cudaLaunchKernelEx(&cfg, gemm_decode_kernel, dp, map, map, map);
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
