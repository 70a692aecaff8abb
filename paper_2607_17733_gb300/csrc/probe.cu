// probe.cu -- tensor-core rate probes (measurement only, not on the layer's
// path): the denominators of the GEMMs' rooflines and the per-instruction
// cost of the small MMAs the decode GEMM issues.
//
// One CTA per SM.  Thread 0 issues `iters` MMAs of one kind back to back into
// one tensor-memory accumulator (operands all zero, so no value can trap or
// slow a unit), commits them to an mbarrier and waits for it; the clock
// difference per CTA is written out.  The warp-level s8 kind runs the legacy
// mma.sync on four warps per CTA.  The caller times the launch with events:
// the FLOPs of a launch over its time is the instruction's throughput.
#include "common.cuh"

namespace mxs {
namespace {

constexpr int kProbeThreads = 128;
constexpr size_t kProbeSmem = 120 * 1024;  // > half of an SM's shared memory: one CTA per SM
constexpr long long kProbeWaitCycles = 4000000000ll;  // ~2 s at the maximum SM clock
constexpr uint32_t kAccCol = 0, kATmemCol = 256, kSfaCol = 288, kSfbCol = 292;

__device__ int g_probe_status;

struct ProbeSmem {
    uint8_t a[128 * 128];  // 128 rows x 128 K' bytes, 128-byte swizzle (all zero)
    uint8_t b[256 * 128];  // up to 256 rows
    uint8_t sfa[512], sfb[1024];
    uint64_t bar;
    uint32_t tmem;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t desc_sf(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)(128 >> 4) << 32) | ((uint64_t)1 << 46);
}
__device__ __forceinline__ bool bar_done(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(su32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// kind: 0 block-scaled e4m3 (A in shared memory), 1 the same with A in tensor
// memory, 2 bf16 (kind::f16), 3 mma.sync m16n8k32 s8.  Every MMA has M = 128
// (the block-scaled kinds have no M = 64 form with one CTA)
__global__ void __launch_bounds__(kProbeThreads, 1) probe_mma_kernel(int kind, int n, long long iters,
                                                                     long long *cycles) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t base = su32(smem_raw);
    ProbeSmem &sm = *reinterpret_cast<ProbeSmem *>(smem_raw + (((base + 1023) & ~1023u) - base));
    const int warp = threadIdx.x >> 5;
    if (kind == 3) {
        int c0 = 0, c1 = 0, c2 = 0, c3 = 0;
        const int a0 = 0, a1 = 0, a2 = 0, a3 = 0, b0 = 0, b1 = 0;
        const long long t0 = clock64();
        for (long long i = 0; i < iters; ++i)
            asm volatile(
                "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                "{%0,%1,%2,%3};"
                : "+r"(c0), "+r"(c1), "+r"(c2), "+r"(c3)
                : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        const long long t1 = clock64();
        if (threadIdx.x == 0 && cycles) cycles[blockIdx.x] = t1 - t0 + (c0 | c1 | c2 | c3);  // the sums are 0
        return;
    }
    // zero operands and scale tiles, visible to the tensor core's (async) proxy
    for (int i = threadIdx.x; i < (int)(sizeof(sm.a) + sizeof(sm.b) + sizeof(sm.sfa) + sizeof(sm.sfb)) / 16;
         i += kProbeThreads)
        reinterpret_cast<uint4 *>(sm.a)[i] = make_uint4(0, 0, 0, 0);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(su32(&sm.bar)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(su32(&sm.tmem))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = sm.tmem;
    if (kind == 1) {  // zero the A tile in tensor memory: each warp its lane quarter, 32 columns
        const uint32_t z = 0;
        const uint32_t taddr = tmem + ((uint32_t)(32 * warp) << 16) + kATmemCol;
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,"
            "%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1};" ::"r"(taddr),
            "r"(z)
            : "memory");
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (threadIdx.x == 0) {
        const uint64_t da = desc_sw128(su32(sm.a)), db = desc_sw128(su32(sm.b));
        const uint32_t d = tmem + kAccCol, sfa = tmem + kSfaCol, sfb = tmem + kSfbCol;
        if (kind != 2) {
            asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfa), "l"(desc_sf(su32(sm.sfa)))
                         : "memory");
            asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfb), "l"(desc_sf(su32(sm.sfb)))
                         : "memory");
            if (n > 128)
                asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfb + 4),
                             "l"(desc_sf(su32(sm.sfb + 512)))
                             : "memory");
        }
        const uint32_t id_mx = ((uint32_t)(n >> 3) << 17) | (1u << 23) | ((uint32_t)(128 >> 4) << 24);
        const uint32_t id_bf = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) |
                               ((uint32_t)(128 >> 4) << 24);
        const long long t0 = clock64();
        for (long long i = 0; i < iters; ++i) {
            const uint32_t acc = i > 0 ? 1u : 0u;
            if (kind == 0)
                asm volatile(
                    "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                    " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%5], "
                    "[%6], p;\n}" ::"r"(d),
                    "l"(da), "l"(db), "r"(id_mx), "r"(acc), "r"(sfa), "r"(sfb)
                    : "memory");
            else if (kind == 1)
                asm volatile(
                    "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                    " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%5], "
                    "[%6], p;\n}" ::"r"(d),
                    "r"(tmem + kATmemCol), "l"(db), "r"(id_mx), "r"(acc), "r"(sfa), "r"(sfb)
                    : "memory");
            else
                asm volatile(
                    "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
                    " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %4, p;\n}" ::"r"(d),
                    "l"(da), "l"(db), "r"(acc), "r"(id_bf)
                    : "memory");
        }
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                         su32(&sm.bar))
                     : "memory");
        const long long tw = clock64();
        bool done = false;
        while (!(done = bar_done(&sm.bar, 0)) && clock64() - tw < kProbeWaitCycles) {
        }
        if (!done) atomicExch(&g_probe_status, MXS_ERR_TIMEOUT);
        const long long t1 = clock64();
        if (cycles) cycles[blockIdx.x] = t1 - t0;
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    }
}

// Issue rate of the decode GEMMs' MMAs: NW warps per CTA (one thread each)
// issue `iters` MMAs back to back into four accumulators of their own, M = 128,
// N = 16, A in tensor memory, the A column and the scale byte varying as in
// the decode kernels.  KIND 0 block-scaled e4m3, 1 bf16, 2 kind 0 plus two
// scale-tile copies per four MMAs.  Operands are zero.  Each issuer records
// its cycles from its first MMA to its commit's completion.
template <int KIND, int NW>
__global__ void __launch_bounds__(kProbeThreads, 1) probe_issue_kernel(long long iters, long long *cycles) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t base = su32(smem_raw);
    ProbeSmem &sm = *reinterpret_cast<ProbeSmem *>(smem_raw + (((base + 1023) & ~1023u) - base));
    const int warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < (int)(sizeof(sm.a) + sizeof(sm.b) + sizeof(sm.sfa) + sizeof(sm.sfb)) / 16;
         i += kProbeThreads)
        reinterpret_cast<uint4 *>(sm.a)[i] = make_uint4(0, 0, 0, 0);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(&sm.bar)), "r"(NW) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(su32(&sm.tmem))
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = sm.tmem;
    {  // zero the A tile in tensor memory: each warp its lane quarter, 32 columns
        const uint32_t z = 0;
        const uint32_t taddr = tmem + ((uint32_t)(32 * warp) << 16) + kATmemCol;
        asm volatile(
            "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,"
            "%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1};" ::"r"(taddr),
            "r"(z)
            : "memory");
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if ((threadIdx.x & 31) == 0 && warp < NW) {
        const uint64_t db = desc_sw128(su32(sm.b)), dsa = desc_sf(su32(sm.sfa)), dsb = desc_sf(su32(sm.sfb));
        const uint32_t sfa = tmem + kSfaCol, sfb = tmem + kSfbCol, a = tmem + kATmemCol;
        const uint32_t acc0 = tmem + kAccCol + 64 * warp;  // four accumulators of 16 columns
        if (KIND != 1) {
            asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfa), "l"(dsa) : "memory");
            asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfb), "l"(dsb) : "memory");
        }
        constexpr uint32_t id_mx = ((uint32_t)(16 >> 3) << 17) | (1u << 23) | ((uint32_t)(128 >> 4) << 24);
        constexpr uint32_t id_bf =
            (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(16 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
        const long long t0 = clock64();
        for (long long i0 = 0; i0 < iters; i0 += 4) {
            if (KIND == 2) {
                asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfa), "l"(dsa) : "memory");
                asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(sfb), "l"(dsb) : "memory");
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t acc = i0 > 0 ? 1u : 0u;
                const uint32_t d = acc0 + 16 * q;
                if (KIND == 1)
                    asm volatile(
                        "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
                        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %4, p;\n}" ::"r"(d),
                        "r"(a + 8 * q), "l"(db + 2 * q), "r"(acc), "r"(id_bf)
                        : "memory");
                else
                    asm volatile(
                        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                        " tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, "
                        "[%5], [%6], p;\n}" ::"r"(d),
                        "r"(a + 8 * q), "l"(db + 2 * q), "r"(id_mx | ((uint32_t)q << 4) | ((uint32_t)q << 29)),
                        "r"(acc), "r"(sfa), "r"(sfb)
                        : "memory");
            }
        }
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                         su32(&sm.bar))
                     : "memory");
        const long long tw = clock64();
        bool done = false;
        while (!(done = bar_done(&sm.bar, 0)) && clock64() - tw < kProbeWaitCycles) {
        }
        if (!done) atomicExch(&g_probe_status, MXS_ERR_TIMEOUT);
        const long long t1 = clock64();
        if (cycles && warp == 0) cycles[blockIdx.x] = t1 - t0;
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    }
}

}  // namespace
}  // namespace mxs

using namespace mxs;

int mxs_probe_mma(int kind, int n, int64_t iters, int64_t *cycles, double *flop, void *stream) {
    if (kind < 0 || kind > 3) return fail(MXS_ERR_INVALID_ARG, "kind=%d (0..3)", kind);
    if (kind != 3 && (n < 16 || n > 256 || n % 16 != 0))
        return fail(MXS_ERR_INVALID_ARG, "n=%d must be a multiple of 16 in [16, 256]", n);
    if (iters < 1 || iters > (int64_t)1 << 32) return fail(MXS_ERR_INVALID_ARG, "iters=%lld", (long long)iters);
    if (!flop) return fail(MXS_ERR_INVALID_ARG, "flop is NULL");
    if (cycles && (reinterpret_cast<uintptr_t>(cycles) & 7)) return fail(MXS_ERR_ALIGN, "cycles must be 8-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute(SM count)");
    e = cudaFuncSetAttribute(probe_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kProbeSmem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(probe smem)");
    const double per = kind == 3 ? 2.0 * 16 * 8 * 32 * (kProbeThreads / 32) : 2.0 * 128 * n * (kind == 2 ? 16 : 32);
    *flop = per * (double)iters * sms;
    probe_mma_kernel<<<sms, kProbeThreads, kProbeSmem, static_cast<cudaStream_t>(stream)>>>(
        kind, n, (long long)iters, reinterpret_cast<long long *>(cycles));
    return cuda_fail(cudaGetLastError(), "probe_mma_kernel launch");
}

int mxs_probe_status(int *status, int reset) {
    if (!status) return fail(MXS_ERR_INVALID_ARG, "status is NULL");
    int rc = check_device();
    if (rc) return rc;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
    int v = 0;
    e = cudaMemcpyFromSymbol(&v, g_probe_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyFromSymbol(probe status)");
    *status = v;
    if (reset && v) {
        const int z = 0;
        e = cudaMemcpyToSymbol(g_probe_status, &z, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyToSymbol(probe status)");
    }
    return MXS_OK;
}

int mxs_probe_mma_issue(int kind, int issuers, int64_t iters, int64_t *cycles, void *stream) {
    if (kind < 0 || kind > 2) return fail(MXS_ERR_INVALID_ARG, "kind=%d (0..2)", kind);
    if (issuers != 1 && issuers != 2 && issuers != 4) return fail(MXS_ERR_INVALID_ARG, "issuers=%d (1, 2, 4)", issuers);
    if (iters < 4 || iters > (int64_t)1 << 32 || iters % 4) return fail(MXS_ERR_INVALID_ARG, "iters=%lld", (long long)iters);
    if (cycles && (reinterpret_cast<uintptr_t>(cycles) & 7)) return fail(MXS_ERR_ALIGN, "cycles must be 8-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute(SM count)");
    using K = void (*)(long long, long long *);
    static const K table[3][3] = {{probe_issue_kernel<0, 1>, probe_issue_kernel<0, 2>, probe_issue_kernel<0, 4>},
                                  {probe_issue_kernel<1, 1>, probe_issue_kernel<1, 2>, probe_issue_kernel<1, 4>},
                                  {probe_issue_kernel<2, 1>, probe_issue_kernel<2, 2>, probe_issue_kernel<2, 4>}};
    const K k = table[kind][issuers == 1 ? 0 : (issuers == 2 ? 1 : 2)];
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kProbeSmem);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(probe smem)");
    k<<<sms, kProbeThreads, kProbeSmem, static_cast<cudaStream_t>(stream)>>>((long long)iters,
                                                                         reinterpret_cast<long long *>(cycles));
    return cuda_fail(cudaGetLastError(), "probe_issue_kernel launch");
}

