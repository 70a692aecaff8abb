// host.cu -- the C ABI of libmxs (include/mxs.h): argument validation, the
// width-grouping plan (step A0), size queries and dispatch to the kernels.
// Validation happens before any CUDA call, so a bad argument is reported the
// same way with or without a GPU.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include <cudaTypedefs.h>

#include "common.cuh"

namespace mxs {

static thread_local char g_err[512] = "";

void set_error(const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
}

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char *what) {
    if (e == cudaSuccess) return MXS_OK;
    return fail(MXS_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Step A0: validate the map and partition block indices by width, keeping the
// original order inside each group (Sec. 4.1: one width per block; the 6/8-bit
// columns come in whole blocks, so every block has exactly one width).
int build_plan(const uint8_t *bits, int64_t K, Plan *p) {
    if (K <= 0 || K % kBlock != 0 || K > MXS_MAX_K)
        return fail(MXS_ERR_SHAPE, "K=%lld must be a positive multiple of 32 and <= %d", (long long)K,
                    MXS_MAX_K);
    if (!bits) return fail(MXS_ERR_INVALID_ARG, "bits is NULL");
    const int nb = (int)(K / kBlock);
    int counts[3] = {0, 0, 0};
    for (int kb = 0; kb < nb; ++kb) {
        const int b = bits[kb];
        if (b != 4 && b != 6 && b != 8) return fail(MXS_ERR_BITS, "bits[%d]=%d is not 4, 6 or 8", kb, b);
        counts[(b - 4) / 2]++;
    }
    p->nb = nb;
    p->n4 = counts[0];
    p->n6 = counts[1];
    p->n8 = counts[2];
    p->n68 = counts[1] + counts[2];
    p->st4 = (p->n4 + 3) / 4;
    p->nst = p->st4 + (p->n68 + 1) / 2;
    p->row_bytes = 16 * (int64_t)p->n4 + 32 * (int64_t)p->n68;
    p->kp = 128 * (int64_t)p->nst;
    int s = 0;
    for (int w = 4; w <= 8; w += 2)
        for (int kb = 0; kb < nb; ++kb)
            if (bits[kb] == w) p->slot_block[s++] = (uint16_t)kb;
    for (int i = nb; i < kMaxNb; ++i) p->slot_block[i] = 0;
    return MXS_OK;
}

int check_device() {
    static int cached[64];  // 0 unknown, 1 ok, 2 unsupported
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev >= 0 && dev < 64 && cached[dev] == 1) return MXS_OK;
    int major = 0, minor = 0;
    e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    const bool ok = major == 10 && minor == 3;
    if (dev >= 0 && dev < 64) cached[dev] = ok ? 1 : 2;
    if (!ok) return fail(MXS_ERR_UNSUPPORTED, "device %d is sm_%d%d; libmxs is built for sm_103a only", dev, major, minor);
    return MXS_OK;
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

int make_plane_map(CUtensorMap *map, const void *base, int64_t rows, int64_t kp, int box_rows) {
    auto fn = encode_fn();
    if (!fn) return fail(MXS_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
    cuuint64_t dims[2] = {(cuuint64_t)kp, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)kp};
    cuuint32_t box[2] = {128u, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(MXS_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return MXS_OK;
}

int make_f32_out_map(CUtensorMap *map, float *base, int64_t rows, int64_t cols, int64_t ld) {
    auto fn = encode_fn();
    if (!fn) return fail(MXS_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 4};
    cuuint32_t box[2] = {16u, 32u};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(MXS_ERR_CUDA, "cuTensorMapEncodeTiled(y) failed (%d)", (int)r);
    return MXS_OK;
}

static bool aligned16(const void *ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15) == 0; }

}  // namespace mxs

using namespace mxs;

extern "C" {

const char *mxs_last_error(void) { return g_err; }

int mxs_version(void) { return MXS_VERSION; }

int64_t mxs_act_row_bytes(int64_t K, const uint8_t *bits) {
    Plan p;
    const int rc = build_plan(bits, K, &p);
    return rc ? -rc : p.row_bytes;
}

int64_t mxs_act_codes_bytes(int64_t M, int64_t K, const uint8_t *bits) {
    if (M < 0) return -fail(MXS_ERR_SHAPE, "M=%lld < 0", (long long)M);
    Plan p;
    const int rc = build_plan(bits, K, &p);
    return rc ? -rc : M * p.row_bytes;
}

int64_t mxs_act_planes_bytes(int64_t M, int64_t K, const uint8_t *bits) {
    if (M < 0) return -fail(MXS_ERR_SHAPE, "M=%lld < 0", (long long)M);
    Plan p;
    const int rc = build_plan(bits, K, &p);
    return rc ? -rc : align256(align256(M * p.kp) + (M + 127) / 128 * p.nst * 512);
}

int64_t mxs_weight_bytes(int64_t N, int64_t K, const uint8_t *bits, int layout) {
    if (N < 0) return -fail(MXS_ERR_SHAPE, "N=%lld < 0", (long long)N);
    if (layout != MXS_W_COMPACT && layout != MXS_W_COMPACT_AND_PLANES)
        return -fail(MXS_ERR_INVALID_ARG, "layout=%d", layout);
    Plan p;
    const int rc = build_plan(bits, K, &p);
    return rc ? -rc : weight_offsets(p, N, layout == MXS_W_COMPACT_AND_PLANES).total;
}

int64_t mxs_linear_decode_workspace_bytes(int64_t M, int64_t K, int64_t N, const uint8_t *bits) {
    if (M < 0 || N < 0) return -fail(MXS_ERR_SHAPE, "M=%lld N=%lld", (long long)M, (long long)N);
    if (M >= 1 && M <= 16) {
        Plan p;
        const int rc = build_plan(bits, K, &p);
        if (rc) return -rc;
        if (M <= kGemvMaxM) return gemv_workspace_bytes(M, N);  // the CUDA-core path: counters, partial sums
        if (MXS_DECODE_TC) return dtc_workspace_bytes(p, M, N);  // planes, counters, partial sums
    }
    return mxs_act_planes_bytes(M, K, bits);
}

int64_t mxs_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K, const uint8_t *bits) {
    if (M < 0 || N < 0) return -fail(MXS_ERR_SHAPE, "M/N < 0");
    Plan p;
    const int rc = build_plan(bits, K, &p);
    if (rc) return -rc;
    return M <= 16 ? decode_workspace_bytes(p, M, N) : 0;
}

int mxs_quantize_act_permuted(const void *x, int64_t M, int64_t K, int64_t ld_x, const int32_t *perm,
                              const uint8_t *bits, int rounding, void *codes, uint8_t *scales, void *planes,
                              void *stream) {
    if (!perm) return fail(MXS_ERR_INVALID_ARG, "perm is NULL");
    if (!aligned16(perm)) return fail(MXS_ERR_ALIGN, "perm must be 16-byte aligned");
    return quantize_act_impl(x, M, K, ld_x, perm, bits, rounding, codes, scales, planes, stream);
}

int mxs_quantize_act(const void *x, int64_t M, int64_t K, int64_t ld_x, const uint8_t *bits, int rounding,
                     void *codes, uint8_t *scales, void *planes, void *stream) {
    return quantize_act_impl(x, M, K, ld_x, nullptr, bits, rounding, codes, scales, planes, stream);
}

int mxs_pack_weight_permuted(const void *w, int64_t N, int64_t K, int64_t ld_w, const int32_t *perm,
                             const uint8_t *bits, int rounding, int layout, void *packed, void *stream) {
    if (!perm) return fail(MXS_ERR_INVALID_ARG, "perm is NULL");
    if (!aligned16(perm)) return fail(MXS_ERR_ALIGN, "perm must be 16-byte aligned");
    return pack_weight_impl(w, N, K, ld_w, perm, bits, rounding, layout, packed, stream);
}

int mxs_pack_weight(const void *w, int64_t N, int64_t K, int64_t ld_w, const uint8_t *bits, int rounding,
                    int layout, void *packed, void *stream) {
    return pack_weight_impl(w, N, K, ld_w, nullptr, bits, rounding, layout, packed, stream);
}

}  // extern "C"

namespace mxs {

int quantize_act_impl(const void *x, int64_t M, int64_t K, int64_t ld_x, const int32_t *perm, const uint8_t *bits,
                      int rounding, void *codes, uint8_t *scales, void *planes, void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (M < 0) return fail(MXS_ERR_SHAPE, "M=%lld < 0", (long long)M);
    if (rounding != MXS_RNE && rounding != MXS_RHAZ) return fail(MXS_ERR_INVALID_ARG, "rounding=%d", rounding);
    if (!x) return fail(MXS_ERR_INVALID_ARG, "x is NULL");
    if (!codes && !planes) return fail(MXS_ERR_INVALID_ARG, "both codes and planes are NULL");
    if (!codes != !scales) return fail(MXS_ERR_INVALID_ARG, "codes and scales must be both set or both NULL");
    if (ld_x < K || ld_x % 8 != 0) return fail(MXS_ERR_INVALID_ARG, "ld_x=%lld must be >= K and a multiple of 8", (long long)ld_x);
    if (!aligned16(x) || (codes && !aligned16(codes)) || (planes && !aligned16(planes)))
        return fail(MXS_ERR_ALIGN, "x, codes and planes must be 16-byte aligned");
    if (M == 0) return MXS_OK;
    if ((rc = check_device())) return rc;
    return launch_quantize(p, x, M, ld_x, rounding, codes, scales, planes, static_cast<cudaStream_t>(stream), perm);
}

int pack_weight_impl(const void *w, int64_t N, int64_t K, int64_t ld_w, const int32_t *perm, const uint8_t *bits,
                     int rounding, int layout, void *packed, void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (N < 0) return fail(MXS_ERR_SHAPE, "N=%lld < 0", (long long)N);
    if (rounding != MXS_RNE && rounding != MXS_RHAZ) return fail(MXS_ERR_INVALID_ARG, "rounding=%d", rounding);
    if (layout != MXS_W_COMPACT && layout != MXS_W_COMPACT_AND_PLANES)
        return fail(MXS_ERR_INVALID_ARG, "layout=%d", layout);
    if (!w || !packed) return fail(MXS_ERR_INVALID_ARG, "w or packed is NULL");
    if (ld_w < K || ld_w % 8 != 0) return fail(MXS_ERR_INVALID_ARG, "ld_w=%lld must be >= K and a multiple of 8", (long long)ld_w);
    if (!aligned16(w) || !aligned16(packed)) return fail(MXS_ERR_ALIGN, "w and packed must be 16-byte aligned");
    if (N == 0) return MXS_OK;
    if ((rc = check_device())) return rc;
    return launch_pack_weight(p, w, N, ld_w, rounding, layout == MXS_W_COMPACT_AND_PLANES, packed,
                              static_cast<cudaStream_t>(stream), perm);
}

}  // namespace mxs

extern "C" {

int mxs_gemm_decode(const void *codes, const uint8_t *scales, const void *act_planes, const uint8_t *bits,
                    const void *packed_w, int64_t M, int64_t N, int64_t K, float *y, int64_t ld_y, void *ws,
                    size_t ws_bytes, void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (M < 0 || N < 0) return fail(MXS_ERR_SHAPE, "M=%lld N=%lld", (long long)M, (long long)N);
    if (M > 16) return fail(MXS_ERR_SHAPE, "decode path takes M <= 16 (M=%lld)", (long long)M);
    if (!packed_w || !y) return fail(MXS_ERR_INVALID_ARG, "NULL operand");
    if (act_planes ? (codes || scales) : (!codes || !scales))
        return fail(MXS_ERR_INVALID_ARG, "give either act_planes or codes and scales");
    if (ld_y < N) return fail(MXS_ERR_INVALID_ARG, "ld_y=%lld < N", (long long)ld_y);
    if ((codes && !aligned16(codes)) || (act_planes && !aligned16(act_planes)) || !aligned16(packed_w) ||
        (reinterpret_cast<uintptr_t>(y) & 3))
        return fail(MXS_ERR_ALIGN, "codes/act_planes/packed_w must be 16-byte aligned, y 4-byte aligned");
    const int64_t need = decode_workspace_bytes(p, M, N);
    if ((int64_t)ws_bytes < need || (need > 0 && !ws))
        return fail(MXS_ERR_BUFFER, "workspace of %lld bytes needed, %zu given", (long long)need, ws_bytes);
    if (M == 0 || N == 0) return MXS_OK;
    if ((rc = check_device())) return rc;
    return launch_gemm_decode(p, codes, scales, act_planes, packed_w, M, N, y, ld_y, false,
                              static_cast<cudaStream_t>(stream));
}

// the tensor-core decode kernel of decode_tc.cu takes the problems when every
// workspace holds, beyond its planes, the counters and one CTA's partial sums
static bool dtc_fits(const Plan *const *plans, const size_t *ws_bytes, const int64_t *N, int count, int64_t M) {
    for (int i = 0; i < count; ++i) {
        const Plan &p = *plans[i];
        const int64_t planes = align256(align256(M * p.kp) + (M + 127) / 128 * p.nst * 512);
        const int64_t counters = (8 * ((N[i] + 127) / 128) + 255) / 256 * 256;
        if ((int64_t)ws_bytes[i] < planes + counters + 2 * M * 128 * 4) return false;
    }
    return true;
}

int mxs_linear_decode_group(const mxs_decode_problem *probs, int count, int64_t M, int rounding, void *stream) {
    if (!probs || count < 1 || count > 3) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..3 problems)", count);
    if (M < 0) return fail(MXS_ERR_SHAPE, "M=%lld", (long long)M);
    if (M > 16) return fail(MXS_ERR_SHAPE, "the fused decode path takes M <= 16 (M=%lld)", (long long)M);
    if (rounding != MXS_RNE && rounding != MXS_RHAZ) return fail(MXS_ERR_INVALID_ARG, "rounding=%d", rounding);
    Plan plans[3];
    const Plan *pp[3];
    const void *planes[3], *packed[3];
    int64_t N[3], ld_y[3];
    float *y[3];
    bool empty = M == 0;
    for (int i = 0; i < count; ++i) {
        const mxs_decode_problem &q = probs[i];
        int rc = build_plan(q.bits, q.K, &plans[i]);
        if (rc) return rc;
        const Plan &p = plans[i];
        if (q.N < 0) return fail(MXS_ERR_SHAPE, "problem %d: N=%lld", i, (long long)q.N);
        if (!q.x || !q.packed_w || !q.y) return fail(MXS_ERR_INVALID_ARG, "problem %d: NULL operand", i);
        if (q.ld_x < q.K || q.ld_x % 8 != 0)
            return fail(MXS_ERR_INVALID_ARG, "problem %d: ld_x=%lld must be >= K and a multiple of 8", i, (long long)q.ld_x);
        if (q.ld_y < q.N) return fail(MXS_ERR_INVALID_ARG, "problem %d: ld_y=%lld < N", i, (long long)q.ld_y);
        // the one-token path's counters and sums; else the planes (the tensor-core
        // kernel fits its CTA count to what the workspace holds beyond them)
        const int64_t need = M >= 1 && M <= kGemvMaxM
                                 ? gemv_workspace_bytes(M, q.N)
                                 : align256(align256(M * p.kp) + (M + 127) / 128 * p.nst * 512);
        if ((int64_t)q.ws_bytes < need || (need > 0 && !q.workspace))
            return fail(MXS_ERR_BUFFER, "problem %d: workspace of %lld bytes needed, %zu given", i, (long long)need,
                        q.ws_bytes);
        if (!aligned16(q.x) || !aligned16(q.packed_w) || (q.workspace && !aligned16(q.workspace)) ||
            (reinterpret_cast<uintptr_t>(q.y) & 3))
            return fail(MXS_ERR_ALIGN, "problem %d: x/packed_w/workspace must be 16-byte aligned, y 4-byte aligned", i);
        for (int j = 0; j < i; ++j)
            if (probs[j].workspace == q.workspace)
                return fail(MXS_ERR_INVALID_ARG, "problems %d and %d share a workspace", j, i);
        empty = empty || q.N == 0;
        pp[i] = &plans[i];
        planes[i] = q.workspace;
        packed[i] = q.packed_w;
        N[i] = q.N;
        y[i] = q.y;
        ld_y[i] = q.ld_y;
    }
    if (empty) {  // nothing to compute for an empty problem: run the others one by one
        for (int i = 0; i < count; ++i) {
            const mxs_decode_problem &q = probs[i];
            const int rc = mxs_linear_decode(q.x, M, q.K, q.ld_x, q.bits, rounding, q.packed_w, q.N, q.y, q.ld_y,
                                             q.workspace, q.ws_bytes, stream);
            if (rc) return rc;
        }
        return MXS_OK;
    }
    int rc = check_device();
    if (rc) return rc;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const void *xs[3];
    int64_t lds[3];
    void *pls[3];
    size_t wsb[3];
    for (int i = 0; i < count; ++i)
        xs[i] = probs[i].x, lds[i] = probs[i].ld_x, pls[i] = probs[i].workspace, wsb[i] = probs[i].ws_bytes;
    if (M <= kGemvMaxM)  // one token: quantization fused into the CUDA-core GEMM (no planes)
        return launch_gemv_decode(pp, xs, lds, packed, N, y, ld_y, pls, wsb, count, M, rounding, true, st);
    rc = launch_quantize_group(pp, xs, lds, M, rounding, pls, count, st);  // one quantizer launch for the group
    if (rc) return rc;
    if (MXS_DECODE_TC && M > kGemvMaxM && dtc_fits(pp, wsb, N, count, M))
        return launch_decode_tc(pp, pls, wsb, packed, N, y, ld_y, count, M, true, st);
    rc = launch_gemm_decode_group(pp, planes, packed, N, y, ld_y, count, M, true, st);
    for (int i = 0; rc < 0 && i < count; ++i) {  // no grouped plan: one launch per problem
        const int r = launch_gemm_decode(plans[i], nullptr, nullptr, planes[i], packed[i], M, N[i], y[i], ld_y[i],
                                         true, st);
        if (r) return r;
        if (i == count - 1) rc = MXS_OK;
    }
    return rc;
}

int mxs_quantize_act_group(const mxs_quant_problem *probs, int count, int64_t M, int rounding, void *stream) {
    if (!probs || count < 1 || count > 3) return fail(MXS_ERR_INVALID_ARG, "count=%d (1..3 problems)", count);
    if (M < 0) return fail(MXS_ERR_SHAPE, "M=%lld", (long long)M);
    if (rounding != MXS_RNE && rounding != MXS_RHAZ) return fail(MXS_ERR_INVALID_ARG, "rounding=%d", rounding);
    Plan plans[3];
    const Plan *pp[3];
    const void *xs[3];
    int64_t lds[3];
    void *pls[3];
    for (int i = 0; i < count; ++i) {
        const mxs_quant_problem &q = probs[i];
        int rc = build_plan(q.bits, q.K, &plans[i]);
        if (rc) return rc;
        if (!q.x || !q.planes) return fail(MXS_ERR_INVALID_ARG, "problem %d: NULL x or planes", i);
        if (q.ld_x < q.K || q.ld_x % 8 != 0)
            return fail(MXS_ERR_INVALID_ARG, "problem %d: ld_x=%lld must be >= K and a multiple of 8", i, (long long)q.ld_x);
        if (!aligned16(q.x) || !aligned16(q.planes)) return fail(MXS_ERR_ALIGN, "problem %d: x and planes must be 16-byte aligned", i);
        const int64_t need = align256(align256(M * plans[i].kp) + (M + 127) / 128 * plans[i].nst * 512);
        if ((int64_t)q.planes_bytes < need)
            return fail(MXS_ERR_BUFFER, "problem %d: planes of %lld bytes needed, %zu given", i, (long long)need,
                        q.planes_bytes);
        for (int j = 0; j < i; ++j)
            if (probs[j].planes == q.planes) return fail(MXS_ERR_INVALID_ARG, "problems %d and %d share planes", j, i);
        pp[i] = &plans[i];
        xs[i] = q.x;
        lds[i] = q.ld_x;
        pls[i] = q.planes;
    }
    if (M == 0) return MXS_OK;
    const int rc = check_device();
    if (rc) return rc;
    return launch_quantize_group(pp, xs, lds, M, rounding, pls, count, static_cast<cudaStream_t>(stream));
}

int mxs_linear_decode(const void *x, int64_t M, int64_t K, int64_t ld_x, const uint8_t *bits, int rounding,
                      const void *packed_w, int64_t N, float *y, int64_t ld_y, void *ws, size_t ws_bytes,
                      void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (M < 0 || N < 0) return fail(MXS_ERR_SHAPE, "M=%lld N=%lld", (long long)M, (long long)N);
    if (M > 16) return fail(MXS_ERR_SHAPE, "the fused decode path takes M <= 16 (M=%lld)", (long long)M);
    if (rounding != MXS_RNE && rounding != MXS_RHAZ) return fail(MXS_ERR_INVALID_ARG, "rounding=%d", rounding);
    if (!x || !packed_w || !y) return fail(MXS_ERR_INVALID_ARG, "NULL operand");
    if (ld_x < K || ld_x % 8 != 0) return fail(MXS_ERR_INVALID_ARG, "ld_x=%lld must be >= K and a multiple of 8", (long long)ld_x);
    if (ld_y < N) return fail(MXS_ERR_INVALID_ARG, "ld_y=%lld < N", (long long)ld_y);
    const int64_t need = M >= 1 && M <= kGemvMaxM
                             ? gemv_workspace_bytes(M, N)
                             : align256(align256(M * p.kp) + (M + 127) / 128 * p.nst * 512);  // the planes
    if ((int64_t)ws_bytes < need || (need > 0 && !ws))
        return fail(MXS_ERR_BUFFER, "workspace of %lld bytes needed, %zu given", (long long)need, ws_bytes);
    if (!aligned16(x) || !aligned16(packed_w) || (ws && !aligned16(ws)) || (reinterpret_cast<uintptr_t>(y) & 3))
        return fail(MXS_ERR_ALIGN, "x/packed_w/workspace must be 16-byte aligned, y 4-byte aligned");
    if (M == 0 || N == 0) return MXS_OK;
    if ((rc = check_device())) return rc;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (M <= kGemvMaxM) {  // one token: quantization fused into the CUDA-core GEMM (no planes)
        const Plan *pp1 = &p;
        return launch_gemv_decode(&pp1, &x, &ld_x, &packed_w, &N, &y, &ld_y, &ws, &ws_bytes, 1, M, rounding, true,
                                  st);
    }
    rc = launch_quantize(p, x, M, ld_x, rounding, nullptr, nullptr, ws, st);
    if (rc) return rc;
    const Plan *pp = &p;
    if (MXS_DECODE_TC && dtc_fits(&pp, &ws_bytes, &N, 1, M))
        return launch_decode_tc(&pp, &ws, &ws_bytes, &packed_w, &N, &y, &ld_y, 1, M, true, st);
    return launch_gemm_decode(p, nullptr, nullptr, ws, packed_w, M, N, y, ld_y, true, st);
}

int mxs_gemm(const void *act_codes, const uint8_t *act_scales, const void *act_planes, const uint8_t *act_bits,
             const void *packed_w, int w_layout, const uint8_t *w_bits, int64_t M, int64_t N, int64_t K, float *y,
             int64_t ld_y, void *ws, size_t ws_bytes, void *stream) {
    Plan p;
    int rc = build_plan(act_bits, K, &p);
    if (rc) return rc;
    if (!w_bits) return fail(MXS_ERR_INVALID_ARG, "w_bits is NULL");
    if (act_bits != w_bits && std::memcmp(act_bits, w_bits, (size_t)p.nb) != 0)
        return fail(MXS_ERR_UNSUPPORTED, "activation and weight maps differ; one map per layer is supported");
    if (w_layout != MXS_W_COMPACT && w_layout != MXS_W_COMPACT_AND_PLANES)
        return fail(MXS_ERR_INVALID_ARG, "w_layout=%d", w_layout);
    if (M <= 16)  // over the planes when given, else over the packed codes
        return mxs_gemm_decode(act_planes ? nullptr : act_codes, act_planes ? nullptr : act_scales, act_planes,
                               act_bits, packed_w, M, N, K, y, ld_y, ws, ws_bytes, stream);
    if (w_layout != MXS_W_COMPACT_AND_PLANES)
        return fail(MXS_ERR_INVALID_ARG, "M > 16 needs a weight packed with MXS_W_COMPACT_AND_PLANES");
    return mxs_gemm_prefill(act_planes, act_bits, packed_w, M, N, K, y, ld_y, stream);
}

static int prefill_checked(const void *act_planes, const uint8_t *bits, const void *packed_w, int64_t M, int64_t N,
                           int64_t K, float *y, int64_t ld_y, int starve, void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (M < 0 || N < 0) return fail(MXS_ERR_SHAPE, "M=%lld N=%lld", (long long)M, (long long)N);
    if (M > 0 && M <= 16)  // such planes hold the decode GEMM's digit form of 6/8-bit blocks
        return fail(MXS_ERR_SHAPE, "the prefill path takes M > 16 (M=%lld): use the decode path", (long long)M);
    if (!act_planes || !packed_w || !y) return fail(MXS_ERR_INVALID_ARG, "NULL operand");
    if (ld_y < N) return fail(MXS_ERR_INVALID_ARG, "ld_y=%lld < N", (long long)ld_y);
    if (!aligned16(act_planes) || !aligned16(packed_w) || (reinterpret_cast<uintptr_t>(y) & 3))
        return fail(MXS_ERR_ALIGN, "act_planes/packed_w must be 16-byte aligned, y 4-byte aligned");
    if (M == 0 || N == 0) return MXS_OK;
    if ((rc = check_device())) return rc;
    return launch_gemm_prefill(p, act_planes, packed_w, M, N, y, ld_y, starve, static_cast<cudaStream_t>(stream));
}

int mxs_gemm_prefill(const void *act_planes, const uint8_t *bits, const void *packed_w, int64_t M, int64_t N,
                     int64_t K, float *y, int64_t ld_y, void *stream) {
    return prefill_checked(act_planes, bits, packed_w, M, N, K, y, ld_y, 0, stream);
}

int mxs_test_decode_starve(const void *act_planes, const uint8_t *bits, const void *packed_w, int64_t M, int64_t N,
                           int64_t K, float *y, int64_t ld_y, int chunk, void *stream) {
    Plan p;
    int rc = build_plan(bits, K, &p);
    if (rc) return rc;
    if (chunk < 1) return fail(MXS_ERR_INVALID_ARG, "chunk=%d must be >= 1", chunk);
    if (M < 1 || M > 16 || N < 1) return fail(MXS_ERR_SHAPE, "M=%lld (1..16), N=%lld", (long long)M, (long long)N);
    if (!act_planes || !packed_w || !y) return fail(MXS_ERR_INVALID_ARG, "NULL operand");
    if (ld_y < N) return fail(MXS_ERR_INVALID_ARG, "ld_y=%lld < N", (long long)ld_y);
    if (!aligned16(act_planes) || !aligned16(packed_w) || (reinterpret_cast<uintptr_t>(y) & 3))
        return fail(MXS_ERR_ALIGN, "act_planes/packed_w must be 16-byte aligned, y 4-byte aligned");
    if ((rc = check_device())) return rc;
    return launch_gemm_decode(p, nullptr, nullptr, act_planes, packed_w, M, N, y, ld_y, false,
                              static_cast<cudaStream_t>(stream), chunk);
}

int mxs_test_dtc_split_weight(int *cost4) {
    if (cost4) *cost4 = gemv_split_cost4();
    return dtc_split_cost8();
}

int mxs_test_decode_arm_starve(int kernel, int stage) {
    if ((kernel != 1 && kernel != 2) || stage < 0)
        return fail(MXS_ERR_INVALID_ARG, "kernel=%d (1 or 2), stage=%d (>= 0)", kernel, stage);
    if (kernel == 1)
        gemv_arm_starve(stage);
    else
        dtc_arm_starve(stage);
    return MXS_OK;
}

int mxs_test_prefill_starve(const void *act_planes, const uint8_t *bits, const void *packed_w, int64_t M, int64_t N,
                            int64_t K, float *y, int64_t ld_y, int stage, void *stream) {
    if (stage < 1) return fail(MXS_ERR_INVALID_ARG, "stage=%d must be >= 1", stage);
    return prefill_checked(act_planes, bits, packed_w, M, N, K, y, ld_y, stage, stream);
}

int mxs_device_status(int *status, int reset, void *stream) {
    if (!status) return fail(MXS_ERR_INVALID_ARG, "status is NULL");
    int rc = check_device();
    if (rc) return rc;
    int a = 0, b = 0, c = 0, d = 0;
    if ((rc = prefill_status(&a, reset, static_cast<cudaStream_t>(stream)))) return rc;
    if ((rc = decode_status(&b, reset))) return rc;
    if ((rc = gemv_status(&c, reset))) return rc;
    if ((rc = dtc_status(&d, reset))) return rc;
    *status = a ? a : (b ? b : (c ? c : d));
    return MXS_OK;
}

}  // extern "C"
