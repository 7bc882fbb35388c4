// aux_kernels.cu -- small kernels around the main ones: the per-token L2 normalization used
// by the Cor. 1 calibration, clearing an fp32 buffer, and the fp64 pieces of the Thm. 2
// (GO-MSE) calibration: expanding an upper-triangle fp32 sum to a full scaled fp64 matrix,
// and an fp64 K x K product.
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

// C[i][j] = scale * Su[min(i,j)][max(i,j)] (Su: fp32, upper triangle i <= j valid).
__global__ void sym_full_f64_kernel(const float* __restrict__ Su, int64_t K, double scale, double* __restrict__ C)
{
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < K * K;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = e / K, j = e - i * K;
        C[e] = scale * static_cast<double>(i <= j ? Su[i * K + j] : Su[j * K + i]);
    }
}

cudaError_t launch_sym_full_f64(const float* Su, int64_t K, double scale, double* C, cudaStream_t stream)
{
    if (K <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((K * K + 255) / 256, 65536);
    sym_full_f64_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(Su, K, scale, C);
    return cudaGetLastError();
}

__global__ void sym_split_bf16_kernel(const float* __restrict__ Su, int64_t K, float scale,
                                      __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo)
{
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < K * K;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = e / K, j = e - i * K;
        const float v = scale * (i <= j ? Su[i * K + j] : Su[j * K + i]);
        const __nv_bfloat16 h = __float2bfloat16_rn(v);
        hi[e] = h;
        // v - h is exact in fp32 (h is v rounded to 8 significant bits)
        lo[e] = __float2bfloat16_rn(v - __bfloat162float(h));
    }
}

cudaError_t launch_sym_split_bf16(const float* Su, int64_t K, float scale, void* hi, void* lo, cudaStream_t stream)
{
    if (K <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((K * K + 255) / 256, 65536);
    sym_split_bf16_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
        Su, K, scale, static_cast<__nv_bfloat16*>(hi), static_cast<__nv_bfloat16*>(lo));
    return cudaGetLastError();
}

__global__ void f32_to_bf16_kernel(const float* __restrict__ src, int64_t count, __nv_bfloat16* __restrict__ dst)
{
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < count;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x)
        dst[e] = __float2bfloat16_rn(src[e]);
}

cudaError_t launch_f32_to_bf16(const float* src, int64_t count, void* dst, cudaStream_t stream)
{
    if (count <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((count + 255) / 256, 65536);
    f32_to_bf16_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(src, count, static_cast<__nv_bfloat16*>(dst));
    return cudaGetLastError();
}

// T = A B for K x K row-major fp64 matrices: 64 x 64 output tiles, 256 threads with 4 x 4
// outputs each, 16-deep slices of A and B staged in shared memory; each output summed in
// k order.
__global__ void __launch_bounds__(256) gemm_f64_kernel(const double* __restrict__ A, const double* __restrict__ B,
                                                       int K, double* __restrict__ T)
{
    __shared__ double As[16][64 + 1];
    __shared__ double Bs[16][64 + 1];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int row0 = blockIdx.y * 64, col0 = blockIdx.x * 64;
    double acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += 16) {
        for (int e = threadIdx.x; e < 16 * 64; e += 256) {
            const int kk = e / 64, rr = e - kk * 64;
            const int ra = row0 + rr, ka = k0 + kk;
            As[kk][rr] = (ra < K && ka < K) ? A[static_cast<int64_t>(ra) * K + ka] : 0.0;
            const int cb = col0 + rr;
            Bs[kk][rr] = (ka < K && cb < K) ? B[static_cast<int64_t>(ka) * K + cb] : 0.0;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            double a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fma(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int r = row0 + ty * 4 + i, c = col0 + tx * 4 + j;
            if (r < K && c < K) T[static_cast<int64_t>(r) * K + c] = acc[i][j];
        }
}

cudaError_t launch_gemm_f64(const double* A, const double* B, int K, double* T, cudaStream_t stream)
{
    if (K <= 0) return cudaSuccess;
    const dim3 grid((K + 63) / 64, (K + 63) / 64);
    gemm_f64_kernel<<<grid, 256, 0, stream>>>(A, B, K, T);
    return cudaGetLastError();
}

}  // namespace espace
