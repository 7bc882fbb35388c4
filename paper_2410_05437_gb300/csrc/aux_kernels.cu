// aux_kernels.cu -- small element-wise kernels around the main ones: the per-token L2
// normalization used by the Cor. 1 calibration, and clearing an fp32 buffer.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "../../include/espace.h"
#include "kernels.h"

namespace espace {

__global__ void normalize_rows_kernel(const __nv_bfloat16* __restrict__ X, int64_t N, int K,
                                      __nv_bfloat16* __restrict__ Xn)
{
    // one warp per token row
    const int lane = threadIdx.x & 31;
    const int64_t row = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (row >= N) return;
    const __nv_bfloat16* x = X + row * K;
    float ss = 0.f;
    for (int k = lane; k < K; k += 32) {
        const float v = __bfloat162float(x[k]);
        ss = fmaf(v, v, ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = ss > 0.f ? rsqrtf(ss) : 0.f;
    for (int k = lane; k < K; k += 32)
        Xn[row * K + k] = __float2bfloat16_rn(__bfloat162float(x[k]) * inv);
}

cudaError_t launch_normalize_rows(const void* X, int64_t N, int K, void* Xn, cudaStream_t stream)
{
    if (N <= 0) return cudaSuccess;
    const int warps = 8;
    const int64_t blocks = (N + warps - 1) / warps;
    normalize_rows_kernel<<<static_cast<unsigned>(blocks), warps * 32, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(X), N, K, static_cast<__nv_bfloat16*>(Xn));
    return cudaGetLastError();
}

__global__ void zero_f32_kernel(float* __restrict__ dst, int64_t count)
{
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        dst[i] = 0.f;
}

cudaError_t launch_zero_f32(float* dst, int64_t count, cudaStream_t stream)
{
    if (count <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((count + 255) / 256, 4096);
    zero_f32_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(dst, count);
    return cudaGetLastError();
}

}  // namespace espace
