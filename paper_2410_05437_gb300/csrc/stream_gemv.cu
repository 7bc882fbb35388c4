// stream_gemv.cu -- bandwidth-bound kernels for decode-shaped (few-token) work.
//
// out[n][r] = sum_k B[n][k] A[r][k] for a handful of tokens n: the matrix A (P^T or W'^T,
// megabytes) is streamed from HBM exactly once with coalesced 16-byte loads, several in
// flight per lane; the few token rows B sit in shared memory; each warp owns whole rows of
// A and finishes them with a shuffle reduction. fp32 accumulation, bf16 output.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "../../include/espace.h"
#include "kernels.h"

namespace espace {

constexpr int GEMV_THREADS = 512;
constexpr int GEMV_UNROLL = 4;                      // 16-byte loads in flight per lane
constexpr int GEMV_MAX_SMEM = 200 * 1024;

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&f)[8])
{
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __bfloat1622float2(h[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

template <int NT>
__global__ void __launch_bounds__(GEMV_THREADS)
    stream_gemv_kernel(const __nv_bfloat16* __restrict__ A, int64_t lda,
                       const __nv_bfloat16* __restrict__ B, int64_t ldb, int nt, int R, int kdim,
                       __nv_bfloat16* __restrict__ out, int64_t ldo)
{
    extern __shared__ uint4 bs[];                   // [NT][kdim / 8] chunks of 8 bf16
    const int kc = kdim / 8;                        // 16-byte chunks per row
    for (int i = threadIdx.x; i < NT * kc; i += blockDim.x) {
        const int n = i / kc, c = i - n * kc;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (n < nt) v = *reinterpret_cast<const uint4*>(B + static_cast<int64_t>(n) * ldb + c * 8);
        bs[i] = v;
    }
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warps = blockDim.x >> 5;
    const int gwarp = blockIdx.x * warps + (threadIdx.x >> 5);
    const int nwarps = gridDim.x * warps;

    for (int r = gwarp; r < R; r += nwarps) {
        const uint4* arow = reinterpret_cast<const uint4*>(A + static_cast<int64_t>(r) * lda);
        float acc[NT];
#pragma unroll
        for (int n = 0; n < NT; ++n) acc[n] = 0.f;
        for (int c0 = lane; c0 < kc; c0 += 32 * GEMV_UNROLL) {
            uint4 a[GEMV_UNROLL];
#pragma unroll
            for (int u = 0; u < GEMV_UNROLL; ++u) {
                const int c = c0 + u * 32;
                a[u] = c < kc ? __ldg(arow + c) : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < GEMV_UNROLL; ++u) {
                const int c = c0 + u * 32;
                if (c >= kc) break;
                float af[8];
                bf16x8_to_f32(a[u], af);
#pragma unroll
                for (int n = 0; n < NT; ++n) {
                    float bf[8];
                    bf16x8_to_f32(bs[n * kc + c], bf);
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[n] = fmaf(af[e], bf[e], acc[n]);
                }
            }
        }
#pragma unroll
        for (int n = 0; n < NT; ++n) {
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) acc[n] += __shfl_xor_sync(0xffffffffu, acc[n], off);
        }
        if (lane < nt && lane < NT) {
            float v = 0.f;
#pragma unroll
            for (int n = 0; n < NT; ++n)
                if (n == lane) v = acc[n];
            out[static_cast<int64_t>(lane) * ldo + r] = __float2bfloat16_rn(v);
        }
    }
}

bool stream_gemv_supported(int nt, int kdim)
{
    if (nt < 1 || nt > 8 || kdim % 8 != 0) return false;
    const int ntp = nt <= 1 ? 1 : nt <= 2 ? 2 : nt <= 4 ? 4 : 8;
    return static_cast<int64_t>(ntp) * kdim * 2 <= GEMV_MAX_SMEM;
}

template <int NT>
static cudaError_t launch_nt(const void* A, int64_t lda, const void* B, int64_t ldb, int nt,
                             int R, int kdim, void* out, int64_t ldo, cudaStream_t stream,
                             int num_sms)
{
    const size_t smem = static_cast<size_t>(NT) * kdim * 2;
    auto kern = stream_gemv_kernel<NT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(std::max<size_t>(smem, 1)));
    if (e != cudaSuccess) return e;
    const int warps_per_block = GEMV_THREADS / 32;
    const int blocks_needed = (R + warps_per_block - 1) / warps_per_block;
    const int grid = std::max(1, std::min(blocks_needed, num_sms));
    kern<<<grid, GEMV_THREADS, smem, stream>>>(
        static_cast<const __nv_bfloat16*>(A), lda, static_cast<const __nv_bfloat16*>(B), ldb,
        nt, R, kdim, static_cast<__nv_bfloat16*>(out), ldo);
    return cudaGetLastError();
}

cudaError_t launch_stream_gemv(const void* A, int64_t lda, const void* B, int64_t ldb, int nt,
                               int R, int kdim, void* out, int64_t ldo, cudaStream_t stream)
{
    if (R <= 0 || nt <= 0) return cudaSuccess;
    if (!stream_gemv_supported(nt, kdim)) return cudaErrorInvalidValue;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (nt <= 1) return launch_nt<1>(A, lda, B, ldb, nt, R, kdim, out, ldo, stream, dev->num_sms);
    if (nt <= 2) return launch_nt<2>(A, lda, B, ldb, nt, R, kdim, out, ldo, stream, dev->num_sms);
    if (nt <= 4) return launch_nt<4>(A, lda, B, ldb, nt, R, kdim, out, ldo, stream, dev->num_sms);
    return launch_nt<8>(A, lda, B, ldb, nt, R, kdim, out, ldo, stream, dev->num_sms);
}

// ---------------------------------------------------------------------------- helpers

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
