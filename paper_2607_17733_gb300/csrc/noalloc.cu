// noalloc.cu -- mxs_linear_decode for callers that cannot allocate device
// memory.
//
// mxs_linear_decode needs a scratch buffer (the activations' MMA planes, or
// for one token the arrival counters and partial sums of the CUDA-core path),
// which its caller allocates.  Some callers cannot: code that runs where
// cudaMalloc is not allowed or not wanted -- an allocator-free runtime that
// owns all device memory up front, a plug-in whose host framework forbids
// allocations on its hot path, or a real-time loop that must not block on
// the driver's allocator.  This file gives them one entry point whose scratch
// is a fixed array in the library's own device memory instead.  The paper has
// no counterpart; it is plumbing for such callers.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds kScratchBytes of it until the process exits.  Host code may
// not hand the array's name to a kernel (on the host that name is a stand-in,
// not a device address); the device address is looked up once per device
// with cudaGetSymbolAddress, with that device current.
#include <mutex>

#include "common.cuh"

namespace mxs {
namespace {

// Holds the MMA planes of M <= 16 tokens for K up to 49152 whatever the map
// (2560 bytes per 128-byte K' stage of 16 tokens).
constexpr size_t kScratchBytes = size_t(2) << 20;  // 2 MiB
constexpr int kMaxDevices = 64;

__device__ __align__(256) uint8_t g_scratch[kScratchBytes];

std::mutex g_scratch_mu;
void *g_scratch_ptr[kMaxDevices];  // device address of g_scratch, per device (nullptr: not looked up yet)

// The scratch's device address on the current device (looked up on first use).
int scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(MXS_ERR_UNSUPPORTED, "device %d: at most %d devices", dev, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void *ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_scratch);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(decode scratch)");
        g_scratch_ptr[dev] = ptr;
    }
    *out = g_scratch_ptr[dev];
    return MXS_OK;
}

}  // namespace
}  // namespace mxs

using namespace mxs;

int mxs_linear_decode_noalloc(const void *x, int64_t M, int64_t K, int64_t ld_x, const uint8_t *bits, int rounding,
                              const void *packed_w, int64_t N, float *y, int64_t ld_y, void *stream) {
    // the checks that need no device come first
    if (M > 16) return fail(MXS_ERR_SHAPE, "the fused decode path takes M <= 16 (M=%lld)", (long long)M);
    // one token: the CUDA-core path's counters and partial sums; more tokens:
    // the planes (the tensor-core kernel fits its CTA count to the rest)
    const int64_t need = M >= 1 && M <= kGemvMaxM ? mxs_linear_decode_workspace_bytes(M, K, N, bits)
                                                  : mxs_act_planes_bytes(M, K, bits);
    if (need < 0) return (int)-need;  // the size query has set the message
    if ((uint64_t)need > kScratchBytes)
        return fail(MXS_ERR_BUFFER,
                    "mxs_linear_decode_noalloc: M=%lld, K=%lld, N=%lld need %lld bytes of scratch; its built-in "
                    "scratch holds %zu (use mxs_linear_decode with a workspace)",
                    (long long)M, (long long)K, (long long)N, (long long)need, kScratchBytes);
    if (M == 0) return mxs_linear_decode(x, M, K, ld_x, bits, rounding, packed_w, N, y, ld_y, nullptr, 0, stream);
    int rc = check_device();
    if (rc) return rc;
    void *scratch = nullptr;
    rc = scratch_address(&scratch);
    if (rc) return rc;
    return mxs_linear_decode(x, M, K, ld_x, bits, rounding, packed_w, N, y, ld_y, scratch, kScratchBytes, stream);
}
