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
// Symmetric expansion of an upper triangle: block (tj, ti) with ti <= tj reads the 64 x 64
// tile (ti, tj) of Su once, row by row in 16-byte pieces, and stores it together with its
// mirror (tj, ti) through shared memory, so that every global access runs along rows; below
// the diagonal of a diagonal tile the element comes from its transposed position.
// store(e, v) writes output elements e .. e + 3 (e = i K + j, j a multiple of 4), whose
// values are v[q] = S(i, j + q). K is a multiple of 4.
template <class Store>
__global__ void __launch_bounds__(256) sym_expand_kernel(const float* __restrict__ Su, int64_t K, Store store)
{
    __shared__ float t[64][65];
    const int64_t ti = blockIdx.y, tj = blockIdx.x;
    if (ti > tj) return;
    const int64_t r0 = ti * 64, c0 = tj * 64;
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
        const int r = e >> 4, c = (e & 15) * 4;
        const int64_t i = r0 + r, j = c0 + c;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i < K && j < K) v = *reinterpret_cast<const float4*>(Su + i * K + j);
        t[r][c] = v.x;
        t[r][c + 1] = v.y;
        t[r][c + 2] = v.z;
        t[r][c + 3] = v.w;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
        const int r = e >> 4, c = (e & 15) * 4;
        const int64_t i = r0 + r, j = c0 + c;
        if (i >= K || j >= K) continue;
        float v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) v[q] = (ti < tj || r <= c + q) ? t[r][c + q] : t[c + q][r];
        store(i * K + j, v);
    }
    if (ti == tj) return;
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
        const int r = e >> 4, c = (e & 15) * 4;
        const int64_t i = c0 + r, j = r0 + c;     // mirror tile: S(i, j) = S(j, i) = t[j - r0][i - c0]
        if (i >= K || j >= K) continue;
        float v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) v[q] = t[c + q][r];
        store(i * K + j, v);
    }
}

struct StoreF64 {
    double* C;
    double scale;
    __device__ void operator()(int64_t e, const float* v) const
    {
        double2* d = reinterpret_cast<double2*>(C + e);
        d[0] = make_double2(scale * static_cast<double>(v[0]), scale * static_cast<double>(v[1]));
        d[1] = make_double2(scale * static_cast<double>(v[2]), scale * static_cast<double>(v[3]));
    }
};

struct StoreSplitBf16 {
    __nv_bfloat16* hi;
    __nv_bfloat16* lo;
    float scale;
    __device__ void operator()(int64_t e, const float* v) const
    {
        __nv_bfloat16 h[4], l[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float x = scale * v[q];
            h[q] = __float2bfloat16_rn(x);
            // x - h is exact in fp32 (h is x rounded to 8 significant bits)
            l[q] = __float2bfloat16_rn(x - __bfloat162float(h[q]));
        }
        *reinterpret_cast<uint2*>(hi + e) = *reinterpret_cast<const uint2*>(h);
        *reinterpret_cast<uint2*>(lo + e) = *reinterpret_cast<const uint2*>(l);
    }
};

static dim3 sym_grid(int64_t K)
{
    const unsigned t = static_cast<unsigned>((K + 63) / 64);
    return dim3(t, t);
}

cudaError_t launch_sym_full_f64(const float* Su, int64_t K, double scale, double* C, cudaStream_t stream)
{
    if (K <= 0) return cudaSuccess;
    if (K % 4 != 0 || (K + 63) / 64 > 65535) return cudaErrorInvalidValue;
    sym_expand_kernel<<<sym_grid(K), 256, 0, stream>>>(Su, K, StoreF64{C, scale});
    return cudaGetLastError();
}

cudaError_t launch_sym_split_bf16(const float* Su, int64_t K, float scale, void* hi, void* lo, cudaStream_t stream)
{
    if (K <= 0) return cudaSuccess;
    if (K % 4 != 0 || (K + 63) / 64 > 65535) return cudaErrorInvalidValue;
    sym_expand_kernel<<<sym_grid(K), 256, 0, stream>>>(
        Su, K, StoreSplitBf16{static_cast<__nv_bfloat16*>(hi), static_cast<__nv_bfloat16*>(lo), scale});
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
