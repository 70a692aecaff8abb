// calib.cu -- offline allocation on the GPU: column sensitivity (Alg. 1) and
// the column order and block widths of sensitivity-based allocation (Alg. 3,
// with the control parameter of Theorem 1).
//
// Column sensitivity (Sec. 3.1, Alg. 1): s_j += sum over the calibration rows
// of x_kj^2, the diagonal of X^T X.  HBM-bound: every bf16 is read once.  A
// CTA owns a strip of 64 columns and one eighth of the rows; the eight CTAs of
// a cluster split the rows of one strip and add their partial sums in rank
// order through distributed shared memory, so the result does not depend on
// timing and no workspace is needed.  A lane loads 16 B (8 columns) of a row;
// 32 lanes x 16 rows per step keep 64 KB of loads in flight per CTA.  The
// square of a bf16 value is exact in fp32 unless it under- or overflows, so
// each lane adds 16 rows of squares per column in fp32 (at most 16 roundings,
// relative error <= 2^-20) and adds that partial to an fp64 sum; a partial
// outside [2^-100, 2^100) is read again and added in fp64, so tiny and huge
// activations keep their exact squares.
//
// Column order (Alg. 3): the position of column i is the number of columns
// with a larger sensitivity, or an equal one and a smaller index (a stable
// descending sort), counted by one thread per column over all keys.  O(K^2)
// comparisons on integers that order the fp64 keys; K <= 65536.
#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace mxs {
namespace {

constexpr int kStrip = 64;   // columns per CTA
constexpr int kRanks = 8;    // CTAs per cluster: row ranges of one strip
constexpr int kCalThreads = 256;
constexpr int kSteps = 16;   // rows per lane between fp64 additions (16 x 32 rows per step)

__device__ __forceinline__ uint32_t map_rank(const void *p, uint32_t rank) {
    uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p)), r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    return r;
}
__device__ __forceinline__ double ld_cluster_f64(uint32_t addr) {
    double v;
    asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release;\n barrier.cluster.wait.acquire;" ::: "memory");
}

__global__ void __cluster_dims__(1, kRanks, 1) __launch_bounds__(kCalThreads, 2)
    column_sensitivity_kernel(const uint16_t *__restrict__ x, int64_t T, int64_t K, int64_t ld, double *s,
                              int accumulate) {
    __shared__ double red[kCalThreads / 8][kStrip];  // [row within a step][column]
    __shared__ double part[kStrip];                 // this CTA's sum of its rows
    uint32_t rank;
    asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
    const int c8 = threadIdx.x & 7;  // which 8 columns of the strip
    const int rs = threadIdx.x >> 3;  // which row of a 32-row step
    const int64_t col = (int64_t)blockIdx.x * kStrip + 8 * c8;
    const bool has = col < K;  // K is a multiple of 32, so col + 8 <= K
    const int64_t r0 = T * rank / kRanks, r1 = T * (rank + 1) / kRanks;

    double acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.0;
    for (int64_t row = r0 + rs; row < r1; row += 32 * kSteps) {
        uint4 v[kSteps];
#pragma unroll
        for (int u = 0; u < kSteps; ++u) {
            const int64_t rr = row + 32 * u;
            v[u] = (has && rr < r1) ? __ldg(reinterpret_cast<const uint4 *>(x + rr * ld + col)) : make_uint4(0, 0, 0, 0);
        }
        float p[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) p[e] = 0.0f;
#pragma unroll
        for (int u = 0; u < kSteps; ++u) {
            const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                const float lo = __uint_as_float(w[h] << 16), hi = __uint_as_float(w[h] & 0xFFFF0000u);
                p[2 * h] = fmaf(lo, lo, p[2 * h]);
                p[2 * h + 1] = fmaf(hi, hi, p[2 * h + 1]);
            }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (p[e] >= 0x1p-100f && p[e] < 0x1p100f) {
                acc[e] += (double)p[e];
            } else {  // an under- or overflowing square (or only zeros): read the run again, in fp64
                double q = 0.0;
                for (int u = 0; u < kSteps; ++u) {
                    const int64_t rr = row + 32 * u;
                    if (has && rr < r1) {
                        const double d = (double)__uint_as_float((uint32_t)__ldg(x + rr * ld + col + e) << 16);
                        q = fma(d, d, q);
                    }
                }
                acc[e] += q;
            }
        }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) red[rs][8 * c8 + e] = acc[e];
    __syncthreads();
    if (threadIdx.x < kStrip) {
        double t = 0.0;
        for (int r = 0; r < kCalThreads / 8; ++r) t += red[r][threadIdx.x];  // fixed order
        part[threadIdx.x] = t;
    }
    cluster_sync();  // every rank's partial sums are in its shared memory
    if (rank == 0 && threadIdx.x < kStrip) {
        double t = 0.0;
        for (uint32_t r = 0; r < kRanks; ++r) t += ld_cluster_f64(map_rank(&part[threadIdx.x], r));  // rank order
        const int64_t c = (int64_t)blockIdx.x * kStrip + threadIdx.x;
        if (c < K) s[c] = accumulate ? s[c] + t : t;
    }
    cluster_sync();  // rank 0 has read the others' shared memory
}

// fp64 -> unsigned integer with the same order (non-NaN keys); -0 counts as +0
__device__ __forceinline__ uint64_t order_key(double d) {
    uint64_t u = (uint64_t)__double_as_longlong(d == 0.0 ? 0.0 : d);
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}

__global__ void __launch_bounds__(256) column_order_kernel(const double *__restrict__ key, int K, int32_t *perm) {
    constexpr int kTile = 2048;
    __shared__ uint64_t tile[kTile];
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    const uint64_t ki = i < K ? order_key(key[i]) : 0;
    int rank = 0;
    for (int base = 0; base < K; base += kTile) {
        const int n = min(kTile, K - base);
        __syncthreads();
        for (int t = threadIdx.x; t < n; t += blockDim.x) tile[t] = order_key(key[base + t]);
        __syncthreads();
        if (i < K) {
            // keys before column i count when >= (ties by index), after it when >
            const int split = min(max(i - base, 0), n);
            for (int t = 0; t < split; ++t) rank += tile[t] >= ki;
            for (int t = split; t < n; ++t) rank += tile[t] > ki;
        }
    }
    if (i < K) perm[rank] = i;
}

}  // namespace
}  // namespace mxs

using namespace mxs;

extern "C" {

int mxs_column_sensitivity(const void *x, int64_t T, int64_t K, int64_t ld_x, double *s, int accumulate,
                           void *stream) {
    if (T < 0) return fail(MXS_ERR_SHAPE, "T=%lld < 0", (long long)T);
    if (K <= 0 || K % 32 != 0) return fail(MXS_ERR_SHAPE, "K=%lld must be a positive multiple of 32", (long long)K);
    if (!s) return fail(MXS_ERR_INVALID_ARG, "s is NULL");
    if (T > 0 && !x) return fail(MXS_ERR_INVALID_ARG, "x is NULL");
    if (ld_x < K || ld_x % 8 != 0)
        return fail(MXS_ERR_INVALID_ARG, "ld_x=%lld must be >= K and a multiple of 8", (long long)ld_x);
    if ((x && reinterpret_cast<uintptr_t>(x) % 16) || reinterpret_cast<uintptr_t>(s) % 8)
        return fail(MXS_ERR_ALIGN, "x must be 16-byte and s 8-byte aligned");
    int rc = check_device();
    if (rc) return rc;
    const int64_t strips = (K + kStrip - 1) / kStrip;
    if (strips > 0x7FFFFFFF) return fail(MXS_ERR_SHAPE, "K too large");
    column_sensitivity_kernel<<<dim3((unsigned)strips, kRanks, 1), kCalThreads, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint16_t *>(x), T, K, ld_x, s, accumulate ? 1 : 0);
    return cuda_fail(cudaGetLastError(), "column_sensitivity_kernel launch");
}

int mxs_allocation_r(int64_t n, const int64_t *d_in, const double *s_layer, double B, double *R) {
    if (n <= 0) return fail(MXS_ERR_SHAPE, "n=%lld layers", (long long)n);
    if (!d_in || !s_layer || !R) return fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (!std::isfinite(B)) return fail(MXS_ERR_INVALID_ARG, "B is not finite");
    double sum_d = 0.0, den = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        if (d_in[i] < 32 || d_in[i] % 32 != 0)
            return fail(MXS_ERR_SHAPE, "d_in[%lld]=%lld must be a positive multiple of 32", (long long)i,
                        (long long)d_in[i]);
        if (!(s_layer[i] >= 0.0 && s_layer[i] <= 1.0))
            return fail(MXS_ERR_INVALID_ARG, "s_layer[%lld]=%g is outside [0, 1]", (long long)i, s_layer[i]);
        sum_d += (double)d_in[i];
        den += 2.0 * s_layer[i] * (double)(d_in[i] - 32);
    }
    if (!(den > 0.0)) return fail(MXS_ERR_INVALID_ARG, "no layer can take 6-bit columns (sum of 2*S*(d-32) is 0)");
    const double r = ((B - 4.0) * sum_d - 4.0 * 32.0 * (double)n) / den;
    if (r < 0.0) return fail(MXS_ERR_INVALID_ARG, "B=%g is below the 8-bit block floor (R=%g < 0)", B, r);
    *R = r;
    return MXS_OK;
}

int mxs_allocate_layer(const double *s, int64_t K, double R, double s_layer, int32_t *perm, uint8_t *bits,
                       int64_t *n6, void *stream) {
    if (K < 32 || K % 32 != 0 || K > MXS_MAX_K)
        return fail(MXS_ERR_SHAPE, "K=%lld must be a multiple of 32 in [32, %d]", (long long)K, MXS_MAX_K);
    if (!s || !perm || !bits) return fail(MXS_ERR_INVALID_ARG, "NULL argument");
    if (!(R >= 0.0) || !std::isfinite(R)) return fail(MXS_ERR_INVALID_ARG, "R=%g", R);
    if (!(s_layer >= 0.0 && s_layer <= 1.0)) return fail(MXS_ERR_INVALID_ARG, "s_layer=%g is outside [0, 1]", s_layer);
    if (reinterpret_cast<uintptr_t>(s) % 8 || reinterpret_cast<uintptr_t>(perm) % 4)
        return fail(MXS_ERR_ALIGN, "s must be 8-byte and perm 4-byte aligned");
    // N6 = floor(R * S * (K - 32)) in [0, K - 32]; 6-bit columns in whole blocks
    const double v = std::floor(R * s_layer * (double)(K - 32));
    const int64_t c6 = (int64_t)std::min(std::max(v, 0.0), (double)(K - 32));
    const int64_t nb = K / 32, b6 = c6 / 32;
    for (int64_t b = 0; b < nb; ++b) bits[b] = b == 0 ? 8 : (b <= b6 ? 6 : 4);
    if (n6) *n6 = c6;
    int rc = check_device();
    if (rc) return rc;
    column_order_kernel<<<(unsigned)((K + 255) / 256), 256, 0, static_cast<cudaStream_t>(stream)>>>(s, (int)K, perm);
    return cuda_fail(cudaGetLastError(), "column_order_kernel launch");
}

}  // extern "C"
