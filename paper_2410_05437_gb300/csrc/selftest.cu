// selftest.cu -- exercises the bounded-wait path of the kernels without any fault: one
// thread waits on an mbarrier that nothing will ever arrive at, gives up after the limit
// and records ESPACE_ERR_TIMEOUT in the device status word, exactly as a stalled pipeline
// stage of the GEMM kernels would.
#include <cuda_runtime.h>

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

}  // namespace espace
