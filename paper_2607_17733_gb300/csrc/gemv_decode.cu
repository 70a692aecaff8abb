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
// Work split.  The packed weights of a problem are one stream of W bytes
// (128-row groups, each a run of 32-element slots).  Each CTA of the launch
// takes an equal share of the bytes -- the k-th of ncta ranges, cut at slot
// boundaries -- whatever the number of row groups, so that every SM streams
// the same bytes (a split by whole groups or by clusters along K leaves SMs
// idle whenever the groups do not divide the SM count).  A range covers whole
// groups, whose rows the CTA writes to y, and partial groups at its ends,
// whose per-row partial sums it writes to the caller's workspace; the last of
// a group's CTAs to arrive (an arrival counter in the workspace) adds the
// partials in CTA order and writes y: deterministic, independent of timing.
// A CTA takes its partial groups first and hands their sums to a hand-off
// warp (workspace stores, a release fence, one arrival, and for the last
// arriver the ordered sum), so that the latency of that exchange overlaps
// the streaming of the rest of its range.  (Measured on the 70B layers: with
// one CTA per SM and equal bytes, q/k/v, o, gate/up and down took 18.1, 15.9,
// 53.8 and 37.0 us against 19.7, 14.7, 53.8 and 38.5 us with whole groups
// per CTA split along K over thread-block clusters, whose counts cannot match
// 152 SMs for 64 or 80 row groups.)
//
// Per CTA.  Prologue: it quantizes the activations of the slots its range
// takes (x is bf16; the rule, bit for bit, of mxs_quantize_act; four threads
// per block, the block maximum by shuffles) into shared memory as int8 codes
// and scale bytes, its blocks of x prefetched into L2 before the wait for the
// kernel before.  One lane of a producer warp streams the range into a ring
// of shared-memory stages with cp.async.bulk (eighteen 4-bit slots, 39 KB, or
// six 6/8-bit slots, 25 KB, per stage; four stages in flight), starting
// before the wait for the kernel before (the weights are static).  Main loop:
// consumer thread t of six sets of 128 is weight row t % 128, and set t / 128
// takes the slots lo + t / 128 + 6j of a stage (a full stage without a test
// per slot); per slot it reads its row's
// codes (16 or 32 bytes) and scale byte from the stage, forms the integer dots
// with dp4a straight from the sign-magnitude codes and adds 2^(Ea'+Ew') * D
// into an fp32 accumulator per token (the product is exact: |D| < 2^20 times
// a power of two).  The sets' sums are added in set order.  Every wait on a
// stage is bounded: on expiry the kernel records MXS_ERR_TIMEOUT
// (mxs_device_status), skips the rest of its arithmetic and waits for its
// copies.
//
// Arrival counters are 64-bit words holding a 48-bit tag, a number the host
// draws afresh for every call (increasing), and a 16-bit count.  An arrival
// raises the word to (tag, 0) by an atomic maximum and takes its count by an
// atomic add (one round trip); a word that still holds another tag (a larger
// one: prior contents of the workspace) goes through compare-and-swap, which
// takes it for count zero.  The last arriver leaves (tag, 0), so the workspace
// needs no preparation: garbage, planes of an earlier call with M > 1, or the
// counters of an earlier call all read as zero (unless a stale word carries
// this call's 48-bit tag), and a CUDA graph that replays one call finds its
// own tag with count zero.
#include <algorithm>
#include <atomic>
#include <cstring>

#include "common.cuh"

namespace mxs {

__device__ int g_gemv_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

#ifndef MXS_GEMV_SETS
#define MXS_GEMV_SETS 6
#endif
constexpr int kGSets = MXS_GEMV_SETS;        // consumer sets; a set is 128 threads, one per weight row
constexpr int kSetWarps = 4;                 // warps per set
constexpr int kConsumers = kSetWarps * kGSets;  // consumer warps
constexpr int kCThreads = 32 * kConsumers;   // 768
constexpr int kGThreads = kCThreads + 64;    // + the producer warp and the hand-off warp
constexpr int kFixWarp = kConsumers + 1;
constexpr int kGMaxProblems = 3;
constexpr int kRing = 4;                     // shared-memory stages in flight (fewer when the tokens need the room)
#ifndef MXS_GEMV_PER4
#define MXS_GEMV_PER4 3
#endif
#ifndef MXS_GEMV_PER68
#define MXS_GEMV_PER68 1
#endif
constexpr int kSlots4 = MXS_GEMV_PER4 * kGSets;    // 4-bit slots per stage (18: three per set)
constexpr int kSlots68 = MXS_GEMV_PER68 * kGSets;  // 6/8-bit slots per stage (6: one per set)
constexpr int kStageBytes = 2176 * kSlots4 > 4224 * kSlots68 ? 2176 * kSlots4 : 4224 * kSlots68;  // 39168
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock
constexpr int64_t kMinCtaBytes = 32768;      // a CTA streams at least this much (and more than one slot)
constexpr int kGemvMaxCtas = 256;            // CTAs per launch at most (sizes the partial-sum area)

struct GemvProblem {
    const uint16_t *x;           // bf16 [M, K], row stride ld_x
    const uint8_t *w;            // packed weights (compact part)
    float *y;
    unsigned long long *cnt;     // workspace: arrival counters [G]
    float *rec;                  // workspace: partial sums [ncta][2][MT][128]
    int64_t ld_x, ld_y, GB, W;   // W = G * GB, the problem's weight bytes
    int N, G, nb, n4, n6;
    int cta0, ncta;              // the problem's CTAs [cta0, cta0 + ncta)
};
struct GemvParams {
    GemvProblem prob[kGMaxProblems];
    uint16_t slot_block[kGMaxProblems][kMaxNb];  // slot -> block of each problem's plan
    int4 span[kGemvMaxCtas];  // per CTA: first group, its first slot, last group, end slot in it
    unsigned long long tag;   // this call's counter tag (48 bits, nonzero)
    int nprob, M, rhaz;
    int starve;               // test hook: > 0 makes every CTA's producer skip the copy of its stage starve-1
};

__host__ __device__ __forceinline__ int64_t slot_off_g(int n4, int s) {
    return s < n4 ? 2176 * (int64_t)s : 2176 * (int64_t)n4 + 4224 * (int64_t)(s - n4);
}
// the slot that starts at byte `off` of a group (off a slot boundary, off <= GB)
__host__ __device__ __forceinline__ int slot_at(int n4, int64_t off) {
    const int64_t b4 = 2176 * (int64_t)n4;
    return off <= b4 ? (int)(off / 2176) : n4 + (int)((off - b4) / 4224);
}
#ifndef MXS_GEMV_COST4
#define MXS_GEMV_COST4 100
#endif
// the work split's weight of a 4-bit slot, in percent of its bytes (a 6/8-bit
// slot weighs its bytes; on the 70B layers 125 and 150 measured slower than
// the bytes alone, 100)
constexpr int64_t kCost4 = MXS_GEMV_COST4;
static_assert(kCost4 >= 50 && kCost4 <= 200, "split weight");
// start of CTA k's range: the first slot boundary at or after the weighted
// position k * C / ncta (C: the problem's total weight)
__host__ __device__ __forceinline__ int64_t cta_start(int k, int ncta, int64_t W, int64_t GB, int n4) {
    if (k >= ncta) return W;
    const int64_t G = W / GB, nb68 = (GB - 2176 * (int64_t)n4) / 4224, w4 = kCost4 * 2176, w8 = 100 * 4224;
    const int64_t CG = w4 * n4 + w8 * nb68, b = G * CG * k / ncta;
    const int64_t g = b / CG, rem = b - g * CG, c4 = w4 * n4;
    const int64_t off = rem <= c4 ? (rem + w4 - 1) / w4 * 2176 : 2176 * (int64_t)n4 + (rem - c4 + w8 - 1) / w8 * 4224;
    return g * GB + off;
}
// the CTAs of a problem whose ranges meet group g: [first, last] (sp: the
// problem's rows of the span table, n CTAs; nb slots per group)
__host__ __device__ __forceinline__ int first_cta(const int4 *sp, int n, int g) {
    int lo = 0, hi = n - 1;  // the last CTA that starts at or before the group's first byte
    while (lo < hi) {
        const int mid = (lo + hi + 1) / 2;
        if (sp[mid].x < g || (sp[mid].x == g && sp[mid].y == 0)) lo = mid; else hi = mid - 1;
    }
    return lo;
}
__host__ __device__ __forceinline__ int last_cta(const int4 *sp, int n, int g, int nb) {
    int lo = 0, hi = n - 1;  // the first CTA that ends at or after the group's last byte
    while (lo < hi) {
        const int mid = (lo + hi) / 2;
        if (sp[mid].z > g || (sp[mid].z == g && sp[mid].w == nb)) hi = mid; else lo = mid + 1;
    }
    return lo;
}
// stage k of a slot range [c0, c1), 4-bit slots [c0, e4): slots [lo, hi)
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
// shared memory: the sets' partial sums, the sums of the (at most two)
// partial segments for the hand-off warp, the barriers and flags, the stage
// ring (128-byte aligned), the token codes and scale bytes
__host__ __device__ __forceinline__ size_t off_fix(int MT) { return (size_t)kGSets * MT * 128 * 4; }
__host__ __device__ __forceinline__ size_t off_bars(int MT) { return off_fix(MT) + (size_t)2 * MT * 128 * 4; }
__host__ __device__ __forceinline__ size_t off_ring(int MT) {
    return (off_bars(MT) + (2 * kRing + 2) * 8 + 16 + 127) / 128 * 128;
}
__host__ __device__ __forceinline__ size_t off_tok(int MT, int nring) {
    return off_ring(MT) + (size_t)nring * kStageBytes;
}
__host__ __device__ __forceinline__ int64_t rec_bytes(int ncta, int MT) { return (int64_t)ncta * 2 * MT * 128 * 4; }
__host__ __device__ __forceinline__ int64_t cnt_bytes(int64_t G) { return (8 * G + 255) / 256 * 256; }

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
// whole-warp wait: every lane waits (its own acquiring test), and the warp goes
// on only if all of them saw the phase
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}
// the 128-byte lines of a 64-byte block (a hint: no data returns)
__device__ __forceinline__ void prefetch_l2(const uint16_t *p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p + 31));
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

// The token slots a CTA needs: its own slots [sp.y, sp.w) when its range
// lies in one group; [sp.y, nb) then [0, sp.w) when it ends in the next group
// before the slot it started at; else all.  Slot s is token slot
// (s - q0) mod nb of ns.
__host__ __device__ __forceinline__ void token_slots(int4 sp, int nb, int &q0, int &ns) {
    if (sp.x == sp.z) {
        q0 = sp.y, ns = sp.w - sp.y;
    } else if (sp.z == sp.x + 1 && sp.w <= sp.y) {
        q0 = sp.y, ns = nb - sp.y + sp.w;
    } else {
        q0 = 0, ns = nb;
    }
}

// A CTA's segments (group, slots [sa, sb)) in processing order: the partial
// groups first -- the tail of its first group, then the head of its last --
// so that their hand-off to the workspace overlaps the whole groups that
// follow; then the whole groups in order.
struct Segs {
    int n, np;         // segments; partial ones first
    int gfull;         // the first whole group
    int4 part0, part1;  // partial segments (group, sa, sb, side)
};
__device__ __forceinline__ Segs segments(int4 sp, int nb) {
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
__device__ __forceinline__ int4 segment(const Segs &s, int i, int nb) {
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

template <int MT, int NR>
__global__ void __launch_bounds__(kGThreads, 1) gemv_decode_kernel(const __grid_constant__ GemvParams gp) {
    int pi = 0;
    while (pi + 1 < gp.nprob && (int)blockIdx.x >= gp.prob[pi + 1].cta0) ++pi;
    const GemvProblem &P = gp.prob[pi];
    const uint16_t *sblk = gp.slot_block[pi];
    const int kc = (int)blockIdx.x - P.cta0;  // the CTA's index within its problem
    const int4 sp = gp.span[blockIdx.x];      // groups sp.x .. sp.z; slots from sp.y in the first, to sp.w in the last
    const Segs segs = segments(sp, P.nb);
    const int M = gp.M, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int q0, ns;
    token_slots(sp, P.nb, q0, ns);

    extern __shared__ __align__(128) uint8_t smem[];
    float *part = reinterpret_cast<float *>(smem);                           // [sets][MT][128]
    float *fixbuf = reinterpret_cast<float *>(smem + off_fix(MT));           // [2][MT][128]
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + off_bars(MT));       // [kRing]
    uint64_t *empty = full + kRing;                                           // [kRing]
    uint64_t *fix_ready = empty + kRing;                                      // [2]
    volatile int *flags = reinterpret_cast<volatile int *>(fix_ready + 2);    // abort
    uint8_t *ring = smem + off_ring(MT);                                     // [kRing][kStageBytes]
    constexpr int nring = NR;                                                // stages in the ring
    int8_t *tcode = reinterpret_cast<int8_t *>(smem + off_tok(MT, nring));   // [ns][MT][32] token codes
    uint8_t *tsc = reinterpret_cast<uint8_t *>(tcode) + (size_t)ns * MT * 32;  // [ns][MT] token scale bytes
    volatile int *abort_flag = flags;

    if (tid == 0) {
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        for (int i = 0; i < nring; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kConsumers);
        }
        mbar_init(&fix_ready[0], kSetWarps);  // the warps of set 0
        mbar_init(&fix_ready[1], kSetWarps);
        flags[0] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == kConsumers) {
        // ---- producer: the range's weight bytes, stage by stage (the weights
        // are static: no wait for the kernel before)
        int ctr = 0, ri = 0, rn = 0;  // copies issued; ring slot and its use count
        if (lane == 0) {
            bool ok = true;
            for (int si = 0; si < segs.n && ok; ++si) {
                const int4 sg = segment(segs, si, P.nb);
                const int sa = sg.y, sb = sg.z, e4 = max(sa, min(sb, P.n4));
                const int nst = stage_count(sa, e4, sb);
                const uint8_t *base = P.w + (int64_t)sg.x * P.GB;
                for (int k = 0; k < nst; ++k) {
                    int lo, hi;
                    stage_range(sa, e4, sb, k, lo, hi);
                    if (gp.starve == ctr + 1 || *abort_flag ||
                        (rn > 0 && !mbar_wait(&empty[ri], (uint32_t)(rn - 1) & 1, abort_flag))) {
                        ok = false;
                        break;
                    }
                    const int64_t off = slot_off_g(P.n4, lo);
                    const uint32_t bytes = (uint32_t)(slot_off_g(P.n4, hi) - off);
                    mbar_expect_tx(&full[ri], bytes);
                    bulk_load(ring + (size_t)ri * kStageBytes, base + off, bytes, &full[ri]);
                    ++ctr;
                    if (++ri == nring) ri = 0, ++rn;
                }
            }
        }
        __syncwarp();
        named_sync(2, kGThreads);  // the consumers are done
        if (lane == 0 && *abort_flag)  // drain: the last copy issued into each ring slot
            for (int i = 0; i < nring && i < ctr; ++i) {
                const int last = i + (ctr - 1 - i) / nring * nring;
                drain_wait(&full[i], (uint32_t)(last / nring) & 1);
            }
        return;
    }

    if (warp == kFixWarp) {
        // ---- the hand-off of the partial segments: this CTA's sums into the
        // workspace, one arrival on the group's counter (release: a fence
        // after the stores), and, for the last of the group's CTAs to arrive,
        // the sum of all of them in CTA order into y.  The consumers go on
        // with the next segment meanwhile.
        const int4 *pspan = gp.span + P.cta0;
        for (int pseg = 0; pseg < segs.np; ++pseg) {
            const int4 sg = pseg == 0 ? segs.part0 : segs.part1;
            const int g = sg.x;
            int kf = 0, kl = 0;
            if (lane == 0) {  // ahead of the wait: the group's contributors
                kf = first_cta(pspan, P.ncta, g);
                kl = last_cta(pspan, P.ncta, g, P.nb);
            }
            if (!warp_wait(&fix_ready[pseg], 0, abort_flag) || *abort_flag) break;
            for (int rr = lane; rr < 128; rr += 32)
#pragma unroll
                for (int t = 0; t < MT; ++t)
                    P.rec[((size_t)(kc * 2 + sg.w) * MT + t) * 128 + rr] = fixbuf[(pseg * MT + t) * 128 + rr];
            __syncwarp();
            int last = 0;
            if (lane == 0) {
                unsigned long long *cw = P.cnt + g;
                asm volatile("fence.acq_rel.gpu;" ::: "memory");
                const unsigned c = arrive_count(cw, gp.tag);
                if (c == 0) {
                    *abort_flag = 1;
                    atomicExch(&g_gemv_status, MXS_ERR_TIMEOUT);
                }
                last = c == (unsigned)(kl - kf + 1);
                if (last) {
                    asm volatile("fence.acq_rel.gpu;" ::: "memory");
                    // (tag, 0): what a replay of this call expects to find
                    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(cw), "l"(gp.tag << 16) : "memory");
                }
            }
            last = __shfl_sync(0xffffffffu, last, 0);
            kf = __shfl_sync(0xffffffffu, kf, 0);
            kl = __shfl_sync(0xffffffffu, kl, 0);
            if (!last) continue;
            // rows lane + 32u: every contributor's four rows in flight at once,
            // then added in CTA order
#pragma unroll
            for (int t = 0; t < MT; ++t) {
                if (t >= M) continue;
                float v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                for (int k0 = kf; k0 <= kl; k0 += 4) {
                    float pv[4][4];
#pragma unroll
                    for (int d = 0; d < 4; ++d) {
                        const int kk = k0 + d;
                        const int sd = kk <= kl && pspan[kk].x < g ? 1 : 0;  // g is that CTA's last group
                        const float *src = P.rec + ((size_t)(kk * 2 + sd) * MT + t) * 128 + lane;
#pragma unroll
                        for (int u = 0; u < 4; ++u) pv[d][u] = kk <= kl ? __ldcg(src + 32 * u) : 0.0f;
                    }
#pragma unroll
                    for (int d = 0; d < 4; ++d)
#pragma unroll
                        for (int u = 0; u < 4; ++u)
                            if (k0 + d <= kl) v[u] = k0 + d == kf ? pv[d][u] : v[u] + pv[d][u];
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int n = 128 * g + lane + 32 * u;
                    if (n < P.N) P.y[(int64_t)t * P.ld_y + n] = v[u];
                }
            }
        }
        named_sync(2, kGThreads);
        return;
    }

    // ---- consumers.  Prologue: the activations of the CTA's token slots as
    // int8 codes (mxs_quantize_act's rule), four threads per block of a
    // token; x may come from the kernel before (programmatic dependent launch)
    const int set = tid >> 7, r = tid & 127;
    // the blocks of x into L2 ahead of the wait: every write lands in L2, so a
    // block the kernel before still writes is read afresh after the wait,
    // and the loads below no longer queue behind the weight ring's first
    // copies in DRAM
    for (int jt = tid; jt < ns * MT; jt += kCThreads) {
        const int j = jt / MT, t = jt - j * MT;
        const int s = q0 + j < P.nb ? q0 + j : q0 + j - P.nb;
        if (t < M) prefetch_l2(P.x + (int64_t)t * P.ld_x + 32 * (int64_t)sblk[s]);
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int nq = ns * MT * 4;
    for (int base = 0; base < nq; base += kCThreads) {  // the same trip count in every thread
        const int i = base + tid;
        const int q = i & 3, jt = i >> 2, j = jt / MT, t = jt - j * MT;
        const int s = q0 + j < P.nb ? q0 + j : q0 + j - P.nb;
        const bool act = i < nq;
        uint4 u = make_uint4(0, 0, 0, 0);
        int b = 8;
        if (act) {
            b = s < P.n4 ? 4 : (s < P.n4 + P.n6 ? 6 : 8);
            if (t < M)
                u = __ldg(reinterpret_cast<const uint4 *>(P.x + (int64_t)t * P.ld_x + 32 * (int64_t)sblk[s]) + q);
        }
        const uint32_t h[8] = {u.x & 0xFFFFu, u.x >> 16, u.y & 0xFFFFu, u.y >> 16,
                               u.z & 0xFFFFu, u.z >> 16, u.w & 0xFFFFu, u.w >> 16};
        uint32_t mag = 0;
#pragma unroll
        for (int k = 0; k < 8; ++k) mag = max(mag, h[k] & 0x7FFFu);
        mag = max(mag, __shfl_xor_sync(0xffffffffu, mag, 1));  // the four threads of the block
        mag = max(mag, __shfl_xor_sync(0xffffffffu, mag, 2));
        const int S = (int)(mag >> 7);
        if (act) {
            uint32_t c0 = 0, c1 = 0;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int m0 = S == 255 ? 0 : quant_elem(h[k], S, b, gp.rhaz);
                const int m1 = S == 255 ? 0 : quant_elem(h[4 + k], S, b, gp.rhaz);
                c0 |= (uint32_t)(m0 & 0xFF) << (8 * k);
                c1 |= (uint32_t)(m1 & 0xFF) << (8 * k);
            }
            *reinterpret_cast<uint2 *>(tcode + (size_t)jt * 32 + 8 * q) = make_uint2(c0, c1);
            if (q == 0) tsc[jt] = (uint8_t)S;
        }
    }
    named_sync(1, kCThreads);

    bool aborted = false;
    int ri = 0, rn = 0;  // ring slot and its use count
    for (int si = 0; si < segs.n; ++si) {
        const int4 sg = segment(segs, si, P.nb);
        const int g = sg.x, sa = sg.y, sb = sg.z, e4 = max(sa, min(sb, P.n4));
        const int nst = stage_count(sa, e4, sb);
        const bool whole = sa == 0 && sb == P.nb;
        float acc[MT];
#pragma unroll
        for (int t = 0; t < MT; ++t) acc[t] = 0.0f;
        for (int k = 0; k < nst; ++k) {
            int lo, hi;
            stage_range(sa, e4, sb, k, lo, hi);
            const int i = ri;
            const uint32_t parity = (uint32_t)rn & 1;
            if (++ri == nring) ri = 0, ++rn;
            if (!aborted && !warp_wait(&full[i], parity, abort_flag)) aborted = true;
            if (!aborted) {
                const uint8_t *sb8 = ring + (size_t)i * kStageBytes;
                if (lo < P.n4) {
                    if (hi - lo == kSlots4) {  // a full stage: no per-slot test
#pragma unroll
                        for (int jj = 0; jj < kSlots4 / kGSets; ++jj) {
                            const int s = lo + set + kGSets * jj;
                            const int ts = s >= q0 ? s - q0 : s - q0 + P.nb;
                            slot4<MT>(sb8 + 2176 * (s - lo), r, tcode + (size_t)ts * MT * 32, tsc + ts * MT, acc);
                        }
                    } else
#pragma unroll
                    for (int jj = 0; jj < kSlots4 / kGSets; ++jj) {
                        const int s = lo + set + kGSets * jj;
                        const int ts = s >= q0 ? s - q0 : s - q0 + P.nb;
                        if (s < hi) slot4<MT>(sb8 + 2176 * (s - lo), r, tcode + (size_t)ts * MT * 32, tsc + ts * MT, acc);
                    }
                } else {
                    if (hi - lo == kSlots68) {  // a full stage: no per-slot test
#pragma unroll
                        for (int jj = 0; jj < kSlots68 / kGSets; ++jj) {
                            const int s = lo + set + kGSets * jj;
                            const int ts = s >= q0 ? s - q0 : s - q0 + P.nb;
                            slot68<MT>(sb8 + 4224 * (s - lo), r, s < P.n4 + P.n6 ? 6 : 8,
                                       tcode + (size_t)ts * MT * 32, tsc + ts * MT, acc);
                        }
                    } else
#pragma unroll
                    for (int jj = 0; jj < kSlots68 / kGSets; ++jj) {
                        const int s = lo + set + kGSets * jj;
                        const int ts = s >= q0 ? s - q0 : s - q0 + P.nb;
                        if (s < hi) slot68<MT>(sb8 + 4224 * (s - lo), r, s < P.n4 + P.n6 ? 6 : 8,
                                               tcode + (size_t)ts * MT * 32, tsc + ts * MT, acc);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[i]);
        }

        // ---- the sets' sums in set order
#pragma unroll
        for (int t = 0; t < MT; ++t) part[(set * MT + t) * 128 + r] = acc[t];
        named_sync(1, kCThreads);
        float val[MT];
        if (set == 0)
#pragma unroll
            for (int t = 0; t < MT; ++t) {
                float v = part[t * 128 + r];
#pragma unroll
                for (int k = 1; k < kGSets; ++k) v += part[(k * MT + t) * 128 + r];
                val[t] = v;
            }
        if (set == 0) {
            const int n = 128 * g + r;
            if (!whole) {  // part of the group: to the hand-off warp
#pragma unroll
                for (int t = 0; t < MT; ++t) fixbuf[(si * MT + t) * 128 + r] = val[t];
                __syncwarp();
                if (lane == 0) mbar_arrive(&fix_ready[si]);
            } else if (n < P.N && !*abort_flag) {  // the whole group: straight to y
#pragma unroll
                for (int t = 0; t < MT; ++t)
                    if (t < M) P.y[(int64_t)t * P.ld_y + n] = val[t];
            }
        }
        named_sync(1, kCThreads);  // `part` is reused by the next segment
    }
    named_sync(2, kGThreads);  // with the producer, which drains after an abort
}

// ------------------------------------------------------------------ host side
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

int mt_of(int64_t M) { return M == 1 ? 1 : (M == 2 ? 2 : 4); }

std::atomic<int> g_ring_override{0};  // mxs_test_gemv_ring: stages in the ring (0: chosen by size)
std::atomic<int> g_gemv_starve{0};    // mxs_test_decode_arm_starve: the next launch's skipped stage (1-based)

// CTAs per problem for a launch of `count` problems of W[i] weight bytes on
// `sms` SMs: one CTA each, then one at a time to the problem with the most
// bytes per CTA, each problem keeping at least kMinCtaBytes (and more than
// one 6/8-bit slot) per CTA.
void gemv_split_ctas(const int64_t *W, int count, int sms, int *ncta) {
    const int total = std::max(count, std::min(sms, kGemvMaxCtas));
    int64_t cap[kGMaxProblems];
    int used = 0;
    for (int i = 0; i < count; ++i) {
        cap[i] = std::max<int64_t>(1, std::min<int64_t>(W[i] / 4225, W[i] / kMinCtaBytes));
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

// the span of CTA k of n over a problem (groups of GB bytes, n4 4-bit slots
// of nb): first group, its first slot, last group, end slot in it
void gemv_span(int k, int n, int64_t W, int64_t GB, int n4, int nb, int *out) {
    (void)nb;
    const int64_t a = cta_start(k, n, W, GB, n4), b = cta_start(k + 1, n, W, GB, n4);
    const int64_t g0 = a / GB, g1 = (b - 1) / GB;
    out[0] = (int)g0;
    out[1] = slot_at(n4, a - g0 * GB);
    out[2] = (int)g1;
    out[3] = slot_at(n4, b - g1 * GB);
}

}  // namespace

int64_t gemv_workspace_bytes(int64_t M, int64_t N) {
    const int64_t G = (N + 127) / 128;
    return cnt_bytes(G) + rec_bytes(kGemvMaxCtas, mt_of(M));
}

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

void gemv_arm_starve(int stage) { g_gemv_starve.store(stage); }
int gemv_split_cost4() { return (int)kCost4; }

int launch_gemv_decode(const Plan *const *plans, const void *const *x, const int64_t *ld_x, const void *const *packed,
                       const int64_t *N, float *const *y, const int64_t *ld_y, void *const *ws,
                       const size_t *ws_bytes, int count, int64_t M, int rounding, bool pdl, cudaStream_t st) {
    if (count < 1 || count > kGMaxProblems) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d)", count, kGMaxProblems);
    if (M < 1 || M > kGemvMaxM) return fail(MXS_ERR_SHAPE, "the CUDA-core decode path takes 1 <= M <= %d", kGemvMaxM);
    const int MT = mt_of(M);
    int64_t G[kGMaxProblems], GB[kGMaxProblems], W[kGMaxProblems];
    for (int i = 0; i < count; ++i) {
        if (N[i] > (int64_t)0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "N too large");
        const WeightOffsets wo = weight_offsets(*plans[i], N[i], false);
        G[i] = wo.G;
        GB[i] = wo.GB;
        W[i] = G[i] * GB[i];
    }
    int ncta[kGMaxProblems];
    gemv_split_ctas(W, count, sms_now(), ncta);
    // the parameter block carries the slot tables and the spans (about 17 KB): built on the host
    static thread_local GemvParams gp;
    std::memset(&gp, 0, sizeof(gp));
    static std::atomic<unsigned long long> tags{0};
    unsigned long long tag = 0;
    while (tag == 0) tag = (tags.fetch_add(1) + 1) & 0xFFFFFFFFFFFFull;
    gp.tag = tag;
    gp.nprob = count;
    gp.M = (int)M;
    gp.rhaz = rounding == MXS_RHAZ;
    gp.starve = g_gemv_starve.exchange(0);  // armed for this one launch
    int cta = 0, max_ns = 0;
    for (int i = 0; i < count; ++i) {
        const Plan &p = *plans[i];
        const int64_t need = cnt_bytes(G[i]) + rec_bytes(ncta[i], MT);
        if ((int64_t)ws_bytes[i] < need || !ws[i])
            return fail(MXS_ERR_BUFFER, "problem %d: workspace of %lld bytes needed, %zu given", i, (long long)need,
                        ws_bytes[i]);
        GemvProblem &P = gp.prob[i];
        P.x = static_cast<const uint16_t *>(x[i]);
        P.w = static_cast<const uint8_t *>(packed[i]);
        P.y = y[i];
        P.cnt = static_cast<unsigned long long *>(ws[i]);
        P.rec = reinterpret_cast<float *>(static_cast<uint8_t *>(ws[i]) + cnt_bytes(G[i]));
        P.ld_x = ld_x[i];
        P.ld_y = ld_y[i];
        P.GB = GB[i];
        P.W = W[i];
        P.N = (int)N[i];
        P.G = (int)G[i];
        P.nb = p.nb, P.n4 = p.n4, P.n6 = p.n6;
        P.cta0 = cta;
        P.ncta = ncta[i];
        for (int k = 0; k < ncta[i]; ++k) {
            int sp[4];
            gemv_span(k, ncta[i], W[i], GB[i], p.n4, p.nb, sp);
            gp.span[cta + k] = make_int4(sp[0], sp[1], sp[2], sp[3]);
            int q0, ns;
            token_slots(make_int4(sp[0], sp[1], sp[2], sp[3]), p.nb, q0, ns);
            max_ns = std::max(max_ns, ns);
        }
        cta += ncta[i];
        std::memcpy(gp.slot_block[i], p.slot_block, sizeof(uint16_t) * (size_t)p.nb);
    }
    // four stages in flight, three or two when the token codes need the room
    const size_t tok = ((size_t)max_ns * MT * 33 + 15) / 16 * 16;
    int nring = kRing;
    while (nring > 2 && off_tok(MT, nring) + tok > (size_t)227 * 1024) --nring;
    const int forced = g_ring_override.load();
    if (forced >= 2 && forced < nring) nring = forced;
    const size_t smem = off_tok(MT, nring) + tok;
    if (smem > (size_t)227 * 1024)
        return fail(MXS_ERR_SHAPE, "decode: K too large for the CUDA-core path at M=%lld", (long long)M);
    using Kernel = void (*)(GemvParams);
    static const Kernel table[3][3] = {  // [MT 1, 2, 4][stages 2, 3, 4]
        {gemv_decode_kernel<1, 2>, gemv_decode_kernel<1, 3>, gemv_decode_kernel<1, 4>},
        {gemv_decode_kernel<2, 2>, gemv_decode_kernel<2, 3>, gemv_decode_kernel<2, 4>},
        {gemv_decode_kernel<4, 2>, gemv_decode_kernel<4, 3>, gemv_decode_kernel<4, 4>}};
    static_assert(kRing == 4, "the kernel table holds rings of 2..4 stages");
    const Kernel k = table[MT == 1 ? 0 : (MT == 2 ? 1 : 2)][nring - 2];
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(gemv smem)");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cta, 1, 1);
    cfg.blockDim = dim3(kGThreads, 1, 1);
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
    e = cudaLaunchKernelEx(&cfg, k, gp);
    return cuda_fail(e, "gemv_decode_kernel launch");
}

}  // namespace mxs

using namespace mxs;

int mxs_test_gemv_split(const int64_t *K, const uint8_t *const *bits, const int64_t *N, int count, int sms,
                        int32_t *ncta, int32_t *spans) {
    if (!K || !bits || !N || !ncta || !spans) return -fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (count < 1 || count > kGMaxProblems || sms < 1)
        return -fail(MXS_ERR_INVALID_ARG, "count=%d (1..%d), sms=%d", count, kGMaxProblems, sms);
    int64_t W[kGMaxProblems], GB[kGMaxProblems];
    Plan plans[kGMaxProblems];
    for (int i = 0; i < count; ++i) {
        const int rc = build_plan(bits[i], K[i], &plans[i]);
        if (rc) return -rc;
        if (N[i] < 1 || N[i] > (int64_t)0x7FFFFFF0) return -fail(MXS_ERR_SHAPE, "N=%lld", (long long)N[i]);
        const WeightOffsets wo = weight_offsets(plans[i], N[i], false);
        GB[i] = wo.GB;
        W[i] = wo.G * wo.GB;
    }
    int n[kGMaxProblems];
    gemv_split_ctas(W, count, sms, n);
    int cta = 0;
    for (int i = 0; i < count; ++i) {
        ncta[i] = n[i];
        for (int k = 0; k < n[i]; ++k, ++cta) gemv_span(k, n[i], W[i], GB[i], plans[i].n4, plans[i].nb, spans + 4 * cta);
    }
    return cta;
}

int mxs_test_gemv_ring(int stages) {
    if (stages != 0 && (stages < 2 || stages > kRing))
        return fail(MXS_ERR_INVALID_ARG, "stages=%d (0, or 2..%d)", stages, kRing);
    g_ring_override.store(stages);
    return MXS_OK;
}
