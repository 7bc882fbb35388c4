// selftest.cu -- test hooks that need no fault: (1) one thread waits on an mbarrier that
// nothing will ever arrive at, gives up after the limit and records ESPACE_ERR_TIMEOUT in
// the device status word, exactly as a stalled pipeline stage of the GEMM kernels would;
// (2) a kernel whose CTAs each hold one SM (shared memory too large for any other CTA of
// the library's kernels to share it) for a bounded time, so that a test can run a
// persistent kernel while part of the SMs are busy.
#include <cuda_runtime.h>

#include <atomic>

#include "../../include/espace.h"
#include "kernels.h"
#include "ptx.cuh"

namespace espace {

__global__ void wait_timeout_kernel(int* status, uint64_t limit_ns)
{
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
    // phase 0 never completes: no thread arrives
    mbar_wait(&bar, 0, &abort_flag, status, limit_ns, ESPACE_ERR_TIMEOUT);
}

cudaError_t launch_wait_timeout(uint64_t limit_ns, cudaStream_t stream)
{
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    wait_timeout_kernel<<<1, 1, 0, stream>>>(dev->status, limit_ns);
    return cudaGetLastError();
}

// Each CTA holds its SM until `hold_ns` after it started (global timer), then leaves.
__global__ void occupy_kernel(uint64_t hold_ns)
{
    extern __shared__ uint8_t hold_smem[];
    if (threadIdx.x == 0) {
        hold_smem[0] = 0;
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < hold_ns) __nanosleep(2000);
    }
}

constexpr int OCCUPY_SMEM = 200 * 1024;

cudaError_t launch_occupy(int ctas, uint64_t hold_ns, cudaStream_t stream)
{
    static std::atomic<bool> attr_set[64];
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return e;
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    if (!attr_set[device].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(occupy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, OCCUPY_SMEM);
        if (e != cudaSuccess) return e;
        attr_set[device].store(true, std::memory_order_release);
    }
    occupy_kernel<<<ctas, 32, OCCUPY_SMEM, stream>>>(hold_ns);
    return cudaGetLastError();
}

}  // namespace espace
