// decode.cu -- the projected forward for decode-shaped batches (N <= 32 tokens), HBM-bound.
//
// One cooperative launch computes both products of Eq. 3:
//   phase 1  Z[n][l] = bf16( sum_k X[n][k] P^T[l][k] )   P^T streamed from HBM once
//   -------  grid barrier (bounded spin) --------------------------------------------
//   phase 2  Y[n][m] = bf16( sum_l Z[n][l] W'^T[m][l] )  W'^T streamed once
// (and, with one phase only, the dense decode product Y = X W^T).
//
// Streaming: at launch, each CTA asks the L2 to prefetch (cp.async.bulk.prefetch.L2, 64 KB
// per request) the rows it will read in phase 2, so the HBM stays busy across the grid
// barrier and phase 2 reads mostly from L2.
//
// Compute: each CTA owns a contiguous range of 16-row blocks of the streamed matrix A; its
// 16 warps split the reduction dimension into 16 segments of 32-wide chunks. A warp walks
// the (row block, chunk) units of its segment in batches, issuing all of a batch's 16-byte
// loads before its MMAs. The values feed mma.sync.m16n8k16 (bf16 in, fp32 accumulate)
// directly as A fragments: the reduction index is permuted inside each 32-wide chunk so
// that thread (g = lane / 4, t = lane % 4) loads elements 8t .. 8t+7 of rows g and g+8,
// which become the fragment positions {2t, 2t+1, 2t+8, 2t+9} of two consecutive k16 MMAs;
// the token operand (8 tokens per MMA) uses the same permutation, so the sum is unchanged.
// Partial results of the 16 warps meet in shared memory and each output is written once.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "../../include/espace.h"
#include "kernels.h"
#include "ptx.cuh"

namespace espace {

constexpr int DEC_THREADS = 512;
constexpr int DEC_WARPS = DEC_THREADS / 32;
constexpr int DEC_MAX_RB = 16;            // 16-row blocks per CTA and phase

struct DecodeArgs {
    const __nv_bfloat16* A[2];   // streamed matrix of each phase, [R][kdim]
    const __nv_bfloat16* B[2];   // tokens of each phase, [nt][kdim]
    __nv_bfloat16* out[2];       // [nt][ldo]
    int R[2], kdim[2], ldo[2];
    int phases;                  // 1 (dense) or 2 (projected)
    int nt;
    unsigned int* bar;           // grid barrier: [0] arrivals, [1] generation
    int* status;
    uint64_t wait_limit_ns;
};

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Read once: no L1 allocation.
__device__ __forceinline__ uint4 ldg_stream(const __nv_bfloat16* p)
{
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Grid-wide barrier for a cooperative launch. Returns false (and records a timeout) if the
// other CTAs did not arrive within the limit.
__device__ bool grid_barrier(unsigned int* bar, int* status, uint64_t limit_ns)
{
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        bool ok = true;
        volatile unsigned int* gen = bar + 1;
        const unsigned int my_gen = *gen;
        __threadfence();
        const unsigned int arrived = atomicAdd(bar, 1u);
        if (arrived == gridDim.x - 1) {
            atomicExch(bar, 0u);
            __threadfence();
            atomicAdd(bar + 1, 1u);
        } else {
            const uint64_t t0 = globaltimer_ns();
            while (*gen == my_gen) {
                if (globaltimer_ns() - t0 > limit_ns) {
                    atomicExch(status, ESPACE_ERR_TIMEOUT);
                    ok = false;
                    break;
                }
                __nanosleep(64);
            }
        }
        __threadfence();
        s_ok = ok ? 1 : 0;
    }
    __syncthreads();
    return s_ok != 0;
}

__device__ __forceinline__ void cta_blocks(int R, int& rb0, int& rb1)
{
    const int blocks = (R + 15) / 16;
    rb0 = static_cast<int>(static_cast<int64_t>(blocks) * blockIdx.x / gridDim.x);
    rb1 = static_cast<int>(static_cast<int64_t>(blocks) * (blockIdx.x + 1) / gridDim.x);
}

// L2 prefetch of this CTA's rows of A (contiguous), 64 KB per request.
__device__ __forceinline__ void prefetch_rows(const __nv_bfloat16* A, int R, int kdim)
{
    int rb0, rb1;
    cta_blocks(R, rb0, rb1);
    const int r_end = min(rb1 * 16, R);
    if (r_end <= rb0 * 16) return;
    const char* base = reinterpret_cast<const char*>(A + static_cast<int64_t>(rb0) * 16 * kdim);
    const int64_t bytes = static_cast<int64_t>(r_end - rb0 * 16) * kdim * 2;
    for (int64_t off = 0; off < bytes; off += 65536)
        prefetch_l2_bulk(base + off, static_cast<uint32_t>(bytes - off < 65536 ? bytes - off : 65536));
}

// One phase: out[n][r] = bf16(sum_k B[n][k] A[r][k]) for this CTA's row blocks. Tokens
// n < nt of B are read through the cache (`b_coherent`: through L2 only, for data written
// earlier in the same launch). acc_s: zeroed [DEC_MAX_RB * 16][NTP] fp32.
template <int NTILES, int BATCH>
__device__ void decode_phase(const __nv_bfloat16* __restrict__ A, const __nv_bfloat16* B, bool b_coherent,
                             int R, int kdim, int nt, float* acc_s, __nv_bfloat16* __restrict__ out, int ldo)
{
    constexpr int NTP = 8 * NTILES;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    int rb0, rb1;
    cta_blocks(R, rb0, rb1);
    const int chunks = (kdim + 31) / 32;
    const int per_warp = (chunks + DEC_WARPS - 1) / DEC_WARPS;
    const int c_begin = min(warp * per_warp, chunks);
    const int nch = min(c_begin + per_warp, chunks) - c_begin;     // chunks of this warp
    const int units = (rb1 - rb0) * nch;

    // token rows this thread feeds into the B fragments (rows past nt read as zero)
    const __nv_bfloat16* brow[NTILES];
    bool bvalid[NTILES];
#pragma unroll
    for (int j = 0; j < NTILES; ++j) {
        const int n = j * 8 + g;
        bvalid[j] = n < nt;
        brow[j] = B + static_cast<int64_t>(bvalid[j] ? n : 0) * kdim;
    }

    float c[NTILES][4];
#pragma unroll
    for (int j = 0; j < NTILES; ++j) c[j][0] = c[j][1] = c[j][2] = c[j][3] = 0.f;

    for (int u0 = 0; u0 < units; u0 += BATCH) {
        // every load of the batch (A rows and token rows) is issued before the first MMA
        uint4 lo[BATCH], hi[BATCH], bf[BATCH][NTILES];
#pragma unroll
        for (int i = 0; i < BATCH; ++i) {
            const int u = u0 + i;
            lo[i] = hi[i] = make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int j = 0; j < NTILES; ++j) bf[i][j] = make_uint4(0, 0, 0, 0);
            if (u < units) {
                const int rb = rb0 + u / nch;
                const int k = (c_begin + u % nch) * 32 + 8 * t;
                const int r_lo = rb * 16 + g, r_hi = r_lo + 8;
                if (k < kdim) {
                    if (r_lo < R) lo[i] = ldg_stream(A + static_cast<int64_t>(r_lo) * kdim + k);
                    if (r_hi < R) hi[i] = ldg_stream(A + static_cast<int64_t>(r_hi) * kdim + k);
#pragma unroll
                    for (int j = 0; j < NTILES; ++j)
                        if (bvalid[j])
                            bf[i][j] = b_coherent ? __ldcg(reinterpret_cast<const uint4*>(brow[j] + k))
                                                  : __ldg(reinterpret_cast<const uint4*>(brow[j] + k));
                }
            }
        }
#pragma unroll
        for (int i = 0; i < BATCH; ++i) {
            const int u = u0 + i;
            if (u >= units) break;                       // uniform across the warp
#pragma unroll
            for (int j = 0; j < NTILES; ++j) {
                mma_bf16_16816(c[j], lo[i].x, hi[i].x, lo[i].y, hi[i].y, bf[i][j].x, bf[i][j].y);
                mma_bf16_16816(c[j], lo[i].z, hi[i].z, lo[i].w, hi[i].w, bf[i][j].z, bf[i][j].w);
            }
            if ((u + 1) % nch == 0) {                    // last chunk of this row block
                float* slot = acc_s + (u / nch) * 16 * NTP;
#pragma unroll
                for (int j = 0; j < NTILES; ++j) {
                    atomicAdd(slot + g * NTP + 8 * j + 2 * t, c[j][0]);
                    atomicAdd(slot + g * NTP + 8 * j + 2 * t + 1, c[j][1]);
                    atomicAdd(slot + (g + 8) * NTP + 8 * j + 2 * t, c[j][2]);
                    atomicAdd(slot + (g + 8) * NTP + 8 * j + 2 * t + 1, c[j][3]);
                    c[j][0] = c[j][1] = c[j][2] = c[j][3] = 0.f;
                }
            }
        }
    }
    __syncthreads();
    const int rows = (rb1 - rb0) * 16;
    for (int i = threadIdx.x; i < rows * NTP; i += blockDim.x) {
        const int n = i / rows, rr = i - n * rows;           // token-major: coalesced stores
        const int r = rb0 * 16 + rr;
        if (n < nt && r < R) out[static_cast<int64_t>(n) * ldo + r] = __float2bfloat16_rn(acc_s[rr * NTP + n]);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < rows * NTP; i += blockDim.x) acc_s[i] = 0.f;
    __syncthreads();
}

template <int NTILES>
__global__ void __launch_bounds__(DEC_THREADS, 1) decode_kernel(const DecodeArgs a)
{
    constexpr int NTP = 8 * NTILES;
    constexpr int BATCH = NTILES == 1 ? 8 : NTILES == 2 ? 4 : 2;
    __shared__ float acc_s[DEC_MAX_RB * 16 * NTP];
    // rows of the second matrix towards L2 while the first one streams
    if (threadIdx.x == 0 && a.phases > 1) prefetch_rows(a.A[1], a.R[1], a.kdim[1]);
    for (int i = threadIdx.x; i < DEC_MAX_RB * 16 * NTP; i += blockDim.x) acc_s[i] = 0.f;
    __syncthreads();
    decode_phase<NTILES, BATCH>(a.A[0], a.B[0], false, a.R[0], a.kdim[0], a.nt, acc_s, a.out[0], a.ldo[0]);
    if (a.phases > 1) {
        if (!grid_barrier(a.bar, a.status, a.wait_limit_ns)) return;
        decode_phase<NTILES, BATCH>(a.A[1], a.B[1], true, a.R[1], a.kdim[1], a.nt, acc_s, a.out[1], a.ldo[1]);
    }
}

// ------------------------------------------------------------------------------ host side

namespace {

int ntiles_for(int nt) { return nt <= 8 ? 1 : nt <= 16 ? 2 : 4; }

template <int NTILES>
cudaError_t launch(DecodeArgs& a, const DeviceInfo* dev, cudaStream_t stream)
{
    auto kern = decode_kernel<NTILES>;
    static bool configured[64] = {};
    if (dev->device < 0 || dev->device >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev->device]) {
        int per_sm = 0;
        cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, DEC_THREADS, 0);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        configured[dev->device] = true;
    }
    if (a.phases == 1) {
        // no grid barrier: an ordinary launch
        kern<<<dev->num_sms, DEC_THREADS, 0, stream>>>(a);
        return cudaGetLastError();
    }
    void* params[] = {&a};
    return cudaLaunchCooperativeKernel(reinterpret_cast<void*>(kern), dim3(dev->num_sms), dim3(DEC_THREADS),
                                       params, 0, stream);
}

cudaError_t launch_any(DecodeArgs& a, const DeviceInfo* dev, cudaStream_t stream)
{
    const int nti = ntiles_for(a.nt);
    if (nti == 1) return launch<1>(a, dev, stream);
    if (nti == 2) return launch<2>(a, dev, stream);
    return launch<4>(a, dev, stream);
}

}  // namespace

bool decode_supported(int nt, int K, int Lp, int M, int num_sms)
{
    if (nt < 1 || nt > DECODE_MAX_TOKENS || K % 8 != 0 || Lp % 8 != 0 || num_sms < 1) return false;
    const int blocks = std::max((Lp + 15) / 16, (M + 15) / 16);
    return (blocks + num_sms - 1) / num_sms <= DEC_MAX_RB;
}

cudaError_t launch_decode_forward(const void* PT, const void* WfT, const void* X, void* Z, void* Y,
                                  int K, int Lp, int M, int nt, unsigned int* grid_bar,
                                  cudaStream_t stream)
{
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (!decode_supported(nt, K, Lp, M, dev->num_sms)) return cudaErrorInvalidValue;
    DecodeArgs a{};
    a.A[0] = static_cast<const __nv_bfloat16*>(PT);
    a.B[0] = static_cast<const __nv_bfloat16*>(X);
    a.out[0] = static_cast<__nv_bfloat16*>(Z);
    a.R[0] = Lp;
    a.kdim[0] = K;
    a.ldo[0] = Lp;
    a.A[1] = static_cast<const __nv_bfloat16*>(WfT);
    a.B[1] = static_cast<const __nv_bfloat16*>(Z);
    a.out[1] = static_cast<__nv_bfloat16*>(Y);
    a.R[1] = M;
    a.kdim[1] = Lp;
    a.ldo[1] = M;
    a.phases = 2;
    a.nt = nt;
    a.bar = grid_bar;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_any(a, dev, stream);
}

cudaError_t launch_decode_dense(const void* W, const void* X, void* Y, int K, int M, int nt,
                                cudaStream_t stream)
{
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (!decode_supported(nt, K, 8, M, dev->num_sms)) return cudaErrorInvalidValue;
    DecodeArgs a{};
    a.A[0] = static_cast<const __nv_bfloat16*>(W);
    a.B[0] = static_cast<const __nv_bfloat16*>(X);
    a.out[0] = static_cast<__nv_bfloat16*>(Y);
    a.R[0] = M;
    a.kdim[0] = K;
    a.ldo[0] = M;
    a.phases = 1;
    a.nt = nt;
    a.bar = nullptr;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_any(a, dev, stream);
}

}  // namespace espace
