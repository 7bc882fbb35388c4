// noalloc.cu -- espace_linear_forward_noalloc: the projected forward for callers that must
// not allocate device memory during the call.
//
// Some callers cannot call cudaMalloc at the point where they run the layer: code running
// under a caller-managed memory budget or pool that forbids foreign allocations, inference
// servers that reserve all device memory up front, and hosts that only hand the library
// pre-allocated input and output buffers. espace_linear_forward grows a per-handle scratch
// buffer for the rank-L intermediate Z the first time it sees a larger batch, which is a
// cudaMalloc; this entry point instead keeps Z in one fixed-size array that is part of the
// loaded library image on each device, so the call itself allocates nothing.
//
// The array is shared by every call on a device and keeps the last call's contents.
// Nothing in it has to start at zero: the first kernel of each call overwrites the whole
// N x Lp region of Z that the second kernel reads. Two calls whose kernels overlap on the
// GPU (different streams, no ordering between them) race on the array.
//
// The first call on each device looks up the array's device address with
// cudaGetSymbolAddress (with that device current) and caches it; make that first call
// before any stream capture.
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include "../../include/espace.h"
#include "kernels.h"

namespace espace {
// Read-only view of a projection handle (defined with the handle in espace_api.cu).
struct ProjView {
    int64_t K, M, L, Lp;
    int device;
    const void* PT;
    const void* WfT;
    unsigned int* bar;
};
int proj_view(espace_proj_t p, ProjView* out);
void set_last_error(const char* msg);   // espace_last_error() text of the calling thread
}  // namespace espace

using namespace espace;

namespace {

// Z scratch of the no-allocation forward: ESPACE_NOALLOC_Z_ELEMS bf16 values (16 MiB),
// held by every device that loads the library until the process exits.
static __device__ __align__(256) uint16_t g_noalloc_z[ESPACE_NOALLOC_Z_ELEMS];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_z_addr[kMaxDevices] = {};

int fail(int code, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return code;
}

// Device address of g_noalloc_z on `device`, which must be current. In host code the name
// g_noalloc_z is only a host-side stand-in, so kernels are given this address instead.
int scratch_address(int device, void** out)
{
    if (device < 0 || device >= kMaxDevices)
        return fail(ESPACE_ERR_STATE, "espace_linear_forward_noalloc: device %d out of range", device);
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_z_addr[device] == nullptr) {
        void* ptr = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_z);
        if (e != cudaSuccess || ptr == nullptr)
            return fail(ESPACE_ERR_CUDA, "espace_linear_forward_noalloc: cudaGetSymbolAddress: %s",
                        cudaGetErrorString(e));
        g_z_addr[device] = ptr;
    }
    *out = g_z_addr[device];
    return ESPACE_OK;
}

}  // namespace

extern "C" int espace_linear_forward_noalloc(espace_proj_t p, const void* X_dev, int64_t N,
                                             void* Y_dev, void* stream)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "espace_linear_forward_noalloc: null handle");
    if (N < 0) return fail(ESPACE_ERR_SHAPE, "espace_linear_forward_noalloc: N < 0");
    if (N == 0) return ESPACE_OK;
    if (X_dev == nullptr || Y_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_linear_forward_noalloc: null pointer");
    if ((reinterpret_cast<uintptr_t>(X_dev) & 15u) || (reinterpret_cast<uintptr_t>(Y_dev) & 15u))
        return fail(ESPACE_ERR_ALIGN, "espace_linear_forward_noalloc: X/Y not 16-byte aligned");
    ProjView v{};
    int rc = proj_view(p, &v);
    if (rc != ESPACE_OK) return rc;
    const int64_t max_tokens = static_cast<int64_t>(ESPACE_NOALLOC_Z_ELEMS) / v.Lp;
    if (N > max_tokens)
        return fail(ESPACE_ERR_SHAPE,
                    "espace_linear_forward_noalloc: N=%lld tokens exceeds the fixed scratch of %d "
                    "bf16 values (at most %lld tokens at Lp=%lld)",
                    (long long)N, ESPACE_NOALLOC_Z_ELEMS, (long long)max_tokens, (long long)v.Lp);
    int cur = -1;
    if (cudaGetDevice(&cur) != cudaSuccess || cur != v.device)
        return fail(ESPACE_ERR_STATE,
                    "espace_linear_forward_noalloc: make device %d (the handle's) current first", v.device);
    void* Z = nullptr;
    rc = scratch_address(v.device, &Z);
    if (rc != ESPACE_OK) return rc;
    const int K = static_cast<int>(v.K), M = static_cast<int>(v.M), Lp = static_cast<int>(v.Lp);
    const int n = static_cast<int>(N);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, v.device) != cudaSuccess)
        return fail(ESPACE_ERR_CUDA, "espace_linear_forward_noalloc: device query failed");
    const bool small = N <= DECODE_MAX_TOKENS && decode_supported(n, K, Lp, M, sms);
    cudaError_t e;
    if (small) {
        e = launch_decode_forward(v.PT, v.WfT, X_dev, Z, Y_dev, K, Lp, M, n, v.bar, st);
    } else {
        e = launch_gemm_tn(X_dev, K, v.PT, K, n, Lp, K, Z, Lp, st);
        if (e == cudaSuccess) e = launch_gemm_tn(Z, Lp, v.WfT, Lp, n, M, Lp, Y_dev, M, st);
    }
    if (e != cudaSuccess)
        return fail(ESPACE_ERR_CUDA, "espace_linear_forward_noalloc: launch: %s", cudaGetErrorString(e));
    return ESPACE_OK;
}
