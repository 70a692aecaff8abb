// gemm_prefill.cu -- A3: the MXINT GEMM for prefill shapes on the 5th-generation
// tensor cores (tcgen05), M > 16 tokens.
//
// y[m,n] = sum over 32-element K-blocks of 2^(Ea+Ew) * sum_i (ma_i 2^-(b-2)) *
// (mw_i 2^-(b-2)): the MXINT product of Sec. 2 with the widths of Sec. 4.1.
// sm_103a has no integer tcgen05 MMA, so the integer mantissas enter the
// tensor core in exact floating-point forms, one accumulator for both:
//   4-bit block:    one e4m3 plane m/4 on the block-scaled FP8 MMA
//                   (kind::mxf8f6f4, one UE8M0 scale per 32 K-elements);
//   6/8-bit block:  its values m * 2^(E-(b-2)) in bf16 (|m| <= 127 has at
//                   most 7 significant bits, bf16 keeps 8 and fp32's exponent
//                   range) on the bf16 MMA (kind::f16): two K=16 MMAs per
//                   block, where high/low e4m3 digits would take four FP8
//                   MMAs (Sec. 6's high/low split, kept for decode).
// Every product is exact; the tensor core accumulates in fp32 TMEM.
//
// Structure (one 128x256 output tile per CTA, 320 threads):
//   warp 0     TMA producer: 128-byte K' stages of A and W planes (128B swizzle)
//              plus the scale tiles (1-D bulk copies), into a 4-stage ring;
//   warp 1     TMEM owner and MMA issuer: tcgen05.cp scales -> TMEM, then the
//              MMAs of the stage, tcgen05.commit frees the stage;
//   warps 2-9  epilogue: tcgen05.ld the fp32 accumulator (two warps per TMEM
//              lane quarter, 128 columns each), TMA-store y.
// Every mbarrier wait is bounded; on expiry the kernel records MXS_ERR_TIMEOUT
// in a device status word, stops issuing work, drains what it issued and frees
// its tensor memory before returning.
#include <cstring>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"

namespace mxs {

__device__ int g_prefill_status;  // sticky MXS_ERR_TIMEOUT, read by mxs_device_status

namespace {

// Output tiles of 128 x BN, BN = 256, or 128 when 256-wide tiles would leave
// SMs idle (fewer tiles than SMs).  Ring stages: 4 of 48 KB (BN = 256) or 6 of
// 32 KB (BN = 128).
constexpr int kBM = 128, kBK = 128;  // tile rows (A), K' bytes per stage
constexpr int kPrefillThreads = 320;  // producer, MMA issuer, 8 epilogue warps (two per TMEM lane quarter)
template <int BN> struct Tile {
    static constexpr int kStages = BN == 256 ? 4 : 6;
    static constexpr int kBBytes = BN * kBK;
    static constexpr int kSfbBytes = BN / 128 * 512;
    static constexpr int kSfCols = 4 + BN / 32;  // TMEM columns per stage: SFA 4, SFB 4 per 128 rows
};
constexpr int kBandM = 16;  // row tiles per band of the tile order
constexpr int kABytes = kBM * kBK;  // 16 KB
constexpr int kSfaBytes = 512;
constexpr int kTmemCols = 512;
constexpr int kAccCol = 0, kSfCol = 256;  // accumulator BN columns; scale factors from column 256
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock  // 2 s bound on any single wait

struct PrefillArgs {
    const uint8_t *sfa;  // scale tiles of A: [ceil(M/128)][nst][512]
    const uint8_t *sfb;  // scale tiles of W: [ceil(N/128)][nst][512]
    float *y;
    int64_t ld_y;
    int M, N, nst, st4, sfb_tiles;
    int starve;  // test hook: >0 makes the producer skip stage `starve-1` (the wait then times out)
    int tma_y;   // y is written by TMA stores through tmap_y (16-byte aligned rows), else by plain stores
};

template <int BN>
struct Smem {
    static constexpr int S = Tile<BN>::kStages;
    uint8_t a[S][kABytes];
    uint8_t b[S][Tile<BN>::kBBytes];
    uint8_t sfa[S][kSfaBytes];
    uint8_t sfb[S][Tile<BN>::kSfbBytes];
    uint8_t stage_y[8][32 * 64];  // per epilogue warp: a 32 x 16 fp32 output block (TMA store)
    uint64_t full[S], empty[S], acc_full, acc_empty;
    uint32_t tmem_base;
    int abort;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }


__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes) : "memory");
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
// Bounded wait: false if the CTA aborted or the wait ran out (then it aborts).
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63) == 0) {  // the bound is checked every 64 polls: reading a clock is not free
            if (*abort) return false;
            if (clock64() - t0 > kWaitCycles) {
                *abort = 1;
                atomicExch(&g_prefill_status, MXS_ERR_TIMEOUT);
                return false;
            }
        }
    }
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
            su32(dst)),
        "l"(map), "r"(su32(bar)), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     su32(dst)),
                 "l"(src), "r"(bytes), "r"(su32(bar))
                 : "memory");
}

// UMMA shared-memory descriptors (sm_100 family): start>>4 [0,14), LBO>>4 [16,30),
// SBO>>4 [32,46), version 1 [46,48), layout [61,64) (2 = 128B swizzle, 0 = none).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t desc_sf(uint32_t addr) {  // 32 rows x 16 B, no swizzle
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)(128 >> 4) << 32) | ((uint64_t)1 << 46);
}

// Instruction descriptor, kind::mxf8f6f4: A/B e4m3 (0), K-major, N>>3 at 17,
// UE8M0 scales (bit 23), M>>4 at 24, scale-factor byte ids at [4,6) (B) and [29,31) (A).
template <int BN>
__device__ __forceinline__ uint32_t idesc(int sfa_id, int sfb_id) {
    return ((uint32_t)(BN >> 3) << 17) | (1u << 23) | ((uint32_t)(kBM >> 4) << 24) | ((uint32_t)sfb_id << 4) |
           ((uint32_t)sfa_id << 29);
}

__device__ __forceinline__ void mma_mx(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t sfa, uint32_t sfb,
                                       uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"(accum), "r"(sfa), "r"(sfb)
        : "memory");
}
// Instruction descriptor, kind::f16: f32 accumulator (bits 4-5 = 1), A and B
// bf16 (bits 7-9, 10-12 = 1), K-major, N>>3 at 17, M>>4 at 24.
template <int BN>
__device__ __forceinline__ void mma_bf16(uint32_t d, uint64_t a, uint64_t b, uint32_t accum) {
    constexpr uint32_t id =
        (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %4, p;\n}" ::"r"(d),
        "l"(a), "l"(b), "r"(accum), "r"(id)
        : "memory");
}
__device__ __forceinline__ void tmem_cp_sf(uint32_t taddr, uint64_t desc) {
    asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
                 : "memory");
}
// smem -> global tile store through a tensor map (clipped at the tensor's edges)
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, const void *src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(map),
                 "r"(su32(src)), "r"(x), "r"(y)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// generic-proxy shared-memory writes -> visible to the bulk copy engine
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 128 consecutive 32-bit columns of this thread's lane
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t (&r)[128]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x128.b32 {"
        "%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,"
        "%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
        "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,"
        "%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,"
        "%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,"
        "%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,"
        "%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127"
        "}, [%128];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
          "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
          "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
          "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]),
          "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]),
          "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]),
          "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]),
          "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]),
          "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]),
          "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]),
          "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]),
          "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

template <int BN>
__global__ void __launch_bounds__(kPrefillThreads, 1) gemm_prefill_kernel(const __grid_constant__ CUtensorMap tmap_a,
                                                              const __grid_constant__ CUtensorMap tmap_b,
                                                              const __grid_constant__ CUtensorMap tmap_y,
                                                              const __grid_constant__ PrefillArgs a) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment for the 128B-swizzled operand tiles
    const uint32_t base = su32(smem_raw);
    constexpr int kStages = Tile<BN>::kStages;
    Smem<BN> &sm = *reinterpret_cast<Smem<BN> *>(smem_raw + (((base + 1023) & ~1023u) - base));

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // Persistent: CTA c takes tiles c, c + gridDim.x, ... of the tile order:
    // bands of kBandM row tiles, the band's row tiles fastest, so that the CTAs
    // running at a time share few weight tiles (each read from DRAM about once
    // per band) and the band's activation tiles stay in L2.  The producer runs
    // ahead into the next tile while the epilogue drains the accumulator.
    const int mt = (a.M + kBM - 1) / kBM, nt = (a.N + BN - 1) / BN, tiles = mt * nt;
    auto tile_origin = [&](int id, int &m0, int &n0) {
        const int band = id / (kBandM * nt);
        const int first = band * kBandM, gm = min(kBandM, mt - first);
        const int in = id - band * kBandM * nt;
        m0 = (first + in % gm) * kBM;
        n0 = (in / gm) * BN;
    };
    const int nst = a.nst;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        mbar_init(&sm.acc_full, 1);
        mbar_init(&sm.acc_empty, 4 * (BN / 128));  // the epilogue warps with columns have read them
        sm.abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&sm.tmem_base)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = sm.tmem_base;
    volatile int *abort = &sm.abort;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        // `it` counts the CTA's K' stages over all its tiles (ring slot it % kStages)
        if (lane == 0) {
            int it = 0, issued = 0;
            bool go = true;
            for (int id = blockIdx.x; id < tiles && go; id += gridDim.x) {
                int m0, n0;
                tile_origin(id, m0, n0);
                const int tile_a = m0 / 128, tile_b = n0 / 128;
                const bool two_b = BN == 256 && tile_b + 1 < a.sfb_tiles;
                const uint32_t tx = kABytes + Tile<BN>::kBBytes + kSfaBytes + (two_b ? 2 : 1) * 512;
                for (int ks = 0; ks < nst; ++ks, ++it) {
                    const int s = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!mbar_wait(&sm.empty[s], ph ^ 1, abort)) {
                        go = false;
                        break;
                    }
                    if (a.starve == it + 1) continue;  // test hook: this stage never arrives
                    mbar_expect_tx(&sm.full[s], tx);
                    tma_load_2d(sm.a[s], &tmap_a, &sm.full[s], ks * kBK, m0);
                    tma_load_2d(sm.b[s], &tmap_b, &sm.full[s], ks * kBK, n0);
                    bulk_load(sm.sfa[s], a.sfa + ((int64_t)tile_a * nst + ks) * 512, 512, &sm.full[s]);
                    bulk_load(sm.sfb[s], a.sfb + ((int64_t)tile_b * nst + ks) * 512, 512, &sm.full[s]);
                    if (two_b)
                        bulk_load(sm.sfb[s] + 512, a.sfb + ((int64_t)(tile_b + 1) * nst + ks) * 512, 512, &sm.full[s]);
                    issued = it + 1;
                }
            }
            // drain: every stage this thread issued must have landed before the CTA exits
            for (int k = (issued > kStages ? issued - kStages : 0); k < issued; ++k) {
                if (a.starve == k + 1) continue;
                const long long t0 = clock64();
                while (!mbar_try_wait(&sm.full[k % kStages], (k / kStages) & 1) && clock64() - t0 < kWaitCycles) {
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int it = 0, committed = 0, lt = 0;
            bool go = true;
            for (int id = blockIdx.x; id < tiles && go; id += gridDim.x, ++lt) {
                // the accumulator is free once the epilogue has read the previous tile
                if (lt > 0 && !mbar_wait(&sm.acc_empty, (lt - 1) & 1, abort)) break;
                fence_after();
                for (int ks = 0; ks < nst; ++ks, ++it) {
                    const int s = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!mbar_wait(&sm.full[s], ph, abort)) {
                        go = false;
                        break;
                    }
                    fence_after();
                    const uint32_t a_addr = su32(sm.a[s]), b_addr = su32(sm.b[s]);
                    if (ks < a.st4) {  // four 4-bit blocks, one e4m3 plane each, block-scaled
                        const uint32_t sfa_t = tmem + kSfCol + Tile<BN>::kSfCols * s, sfb_t = sfa_t + 4;
                        tmem_cp_sf(sfa_t, desc_sf(su32(sm.sfa[s])));
                        tmem_cp_sf(sfb_t, desc_sf(su32(sm.sfb[s])));
                        if (BN == 256) tmem_cp_sf(sfb_t + 4, desc_sf(su32(sm.sfb[s] + 512)));
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            mma_mx(tmem + kAccCol, desc_sw128(a_addr + 32 * q), desc_sw128(b_addr + 32 * q),
                                   idesc<BN>(q, q), sfa_t, sfb_t, (ks > 0 || q > 0) ? 1u : 0u);
                    } else {  // two 6/8-bit blocks as bf16 values (scales inside): four K=16 MMAs
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            mma_bf16<BN>(tmem + kAccCol, desc_sw128(a_addr + 32 * q), desc_sw128(b_addr + 32 * q),
                                         (ks > 0 || q > 0) ? 1u : 0u);
                    }
                    mma_commit(&sm.empty[s]);  // frees the stage once these MMAs have read it
                    committed = it + 1;
                }
                if (go) mma_commit(&sm.acc_full);  // the tile's accumulator is complete
            }
            // drain: wait (bounded) until the tensor core has finished what was issued
            if (committed > 0) {
                const int k = committed - 1;
                const long long t0 = clock64();
                while (!mbar_try_wait(&sm.empty[k % kStages], (k / kStages) & 1) && clock64() - t0 < kWaitCycles) {
                }
            }
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..9)
        // Warp w reads TMEM lane quarter w % 4 (the quarter a warp may access)
        // and columns [128 h, 128 h + 128), h = (w - 2) / 4: one 128-column
        // load, then the accumulator part is released and written out.
        const int quad = warp & 3, half = (warp - 2) >> 2;
        const bool vec = ((a.ld_y & 3) == 0) && ((reinterpret_cast<uintptr_t>(a.y) & 15) == 0);
        uint8_t *stg = sm.stage_y[warp - 2];
        int lt = 0;
        // (128-wide tiles: the warps of the second column half have no work)
        for (int id = half < BN / 128 ? (int)blockIdx.x : tiles; id < tiles; id += gridDim.x, ++lt) {
            int m0, n0;
            tile_origin(id, m0, n0);
            // one lane polls for the main loop, then every lane takes its own
            // acquiring test; the decision is warp-uniform (tcgen05.ld is .sync.aligned)
            bool ok = true;
            if (lane == 0) ok = mbar_wait(&sm.acc_full, lt & 1, abort);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            mbar_try_wait(&sm.acc_full, lt & 1);
            fence_after();
            const int row0 = m0 + 32 * quad, row = row0 + lane;
            float *yrow = a.y + (int64_t)row * a.ld_y;
            uint32_t r[128];
            tmem_ld128(tmem + ((uint32_t)(32 * quad) << 16) + kAccCol + 128 * half, r);
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.acc_empty);  // this part of the accumulator is in registers
#pragma unroll
            for (int cc = 0; cc < 8; ++cc) {
                const int n = n0 + 128 * half + 16 * cc;
                if (a.tma_y) {
                    // 32 rows x 16 columns through the staging block (row r at
                    // 64 r), one TMA store writes it as 64-byte row pieces
                    if (row0 < a.M && n < a.N) {
                        if (lane == 0) bulk_wait_read0();  // the previous store has read the block
                        __syncwarp();
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            *reinterpret_cast<uint4 *>(stg + lane * 64 + 16 * j) =
                                make_uint4(r[16 * cc + 4 * j], r[16 * cc + 4 * j + 1], r[16 * cc + 4 * j + 2],
                                           r[16 * cc + 4 * j + 3]);
                        fence_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tmap_y, stg, n, row0);
                            bulk_commit();
                        }
                    }
                } else if (row < a.M) {
                    if (vec && n + 16 <= a.N) {
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            *reinterpret_cast<uint4 *>(yrow + n + 4 * i) =
                                make_uint4(r[16 * cc + 4 * i], r[16 * cc + 4 * i + 1], r[16 * cc + 4 * i + 2],
                                           r[16 * cc + 4 * i + 3]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            if (n + i < a.N) yrow[n + i] = __uint_as_float(r[16 * cc + i]);
                    }
                }
            }
        }
        if (lane == 0) bulk_wait0();  // the stores have finished reading (and writing) before the CTA ends
    }

    fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

template <int BN>
int launch_tiles(const CUtensorMap &ta, const CUtensorMap &tb, const CUtensorMap &ty, const PrefillArgs &a,
                 int64_t tiles, int sms, cudaStream_t st) {
    const size_t smem = sizeof(Smem<BN>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(gemm_prefill_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(prefill smem)");
    dim3 grid((unsigned)std::min<int64_t>(tiles, std::max(1, sms)), 1);  // one persistent CTA per SM
    gemm_prefill_kernel<BN><<<grid, kPrefillThreads, smem, st>>>(ta, tb, ty, a);
    return cuda_fail(cudaGetLastError(), "gemm_prefill_kernel launch");
}

}  // namespace

int launch_gemm_prefill(const Plan &p, const void *act_planes, const void *packed_w, int64_t M, int64_t N, float *y,
                        int64_t ld_y, int starve, cudaStream_t st) {
    if (M > 0x7FFFFFF0 || N > 0x7FFFFFF0) return fail(MXS_ERR_SHAPE, "M or N too large");
    int dev = 0, sms = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return cuda_fail(e, "cudaDeviceGetAttribute(SM count)");
    // 256-wide tiles unless they would leave SMs idle
    const int64_t mt = (M + kBM - 1) / kBM;
    const int BN = mt * ((N + 255) / 256) >= sms ? 256 : 128;
    const int64_t tiles = mt * ((N + BN - 1) / BN);
    if (tiles > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "M x N too large for the prefill grid");
    const uint8_t *ap = static_cast<const uint8_t *>(act_planes);
    const uint8_t *wb = static_cast<const uint8_t *>(packed_w);
    const WeightOffsets off = weight_offsets(p, N, true);
    CUtensorMap ta, tb;
    int rc = make_plane_map(&ta, ap, M, p.kp, kBM);
    if (rc) return rc;
    rc = make_plane_map(&tb, wb + off.planes, N, p.kp, BN);
    if (rc) return rc;
    PrefillArgs a;
    a.sfa = ap + align256(M * p.kp);
    a.sfb = wb + off.sf;
    a.y = y;
    a.ld_y = ld_y;
    a.M = (int)M;
    a.N = (int)N;
    a.nst = p.nst;
    a.st4 = p.st4;
    a.sfb_tiles = (int)((N + 127) / 128);
    a.starve = starve;
    // y by TMA stores when its rows are 16-byte aligned (else plain stores)
    CUtensorMap ty;
    a.tma_y = ((ld_y & 3) == 0) && ((reinterpret_cast<uintptr_t>(y) & 15) == 0);
    if (a.tma_y) {
        rc = make_f32_out_map(&ty, y, M, N, ld_y);
        if (rc) return rc;
    } else {
        std::memcpy(&ty, &ta, sizeof(CUtensorMap));  // unused
    }
    return BN == 256 ? launch_tiles<256>(ta, tb, ty, a, tiles, sms, st) : launch_tiles<128>(ta, tb, ty, a, tiles, sms, st);
}

int prefill_status(int *status, int reset, cudaStream_t st) {
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int v = 0;
    e = cudaMemcpyFromSymbol(&v, g_prefill_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyFromSymbol(status)");
    *status = v;
    if (reset && v != 0) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_prefill_status, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyToSymbol(status)");
    }
    return MXS_OK;
}

}  // namespace mxs
