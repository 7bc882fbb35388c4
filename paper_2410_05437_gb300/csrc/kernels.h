// kernels.h -- host-side launchers of the library's CUDA kernels (internal, not the ABI).
// Every launcher validates nothing: espace_api.cu checks shapes and pointers first.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace espace {

struct DeviceInfo {
    int device = -1;
    int num_sms = 0;
    int* status = nullptr;   // device status word (ESPACE_ERR_TIMEOUT after a failed wait)
};

// Per-device state, created on first use (the status word is the only allocation).
int device_info(DeviceInfo** out);

uint64_t wait_limit_ns();

// C[rows][cols] (bf16, leading dimension ldc) = A[rows][kdim] * B[cols][kdim]^T with fp32
// accumulation on tcgen05 tensor cores; A and B are bf16 with leading dimensions lda, ldb.
// kdim, lda, ldb and ldc must be multiples of 8 and the pointers 16-byte aligned.
cudaError_t launch_gemm_tn(const void* A, int64_t lda, const void* B, int64_t ldb, int rows,
                           int cols, int kdim, void* C, int64_t ldc, cudaStream_t stream);

// The projected forward Z = X P, Y = Z W' in one persistent launch of the CTA-pair kernel:
// work items drawn from an atomic ticket, Z tiles first, then Y tiles; a Y tile's producer
// waits (bounded) until the 256-row block of Z it reads is complete. ready: ceil(N / 256)
// zeroed ints, sched: two zeroed ints (ticket, exit counter), owned by the caller; the last
// CTA to leave zeroes them again, also after a launch that gave up waiting. One launch at
// a time may use them. Needs N, Lp > 128 to be worthwhile.
cudaError_t launch_forward_fused(const void* X, const void* PT, void* Z, const void* WfT, void* Y, int N,
                                 int K, int Lp, int M, int* ready, int* sched, cudaStream_t stream);

// Swapped product: out[n][r] (bf16, leading dimension ldo) = sum_k W[r][k] X[n][k], the
// weights as the 128-row tcgen05 operand, the tile stored transposed, token tiles of 128
// (ntok <= 128) or 256. The reduction splits over CTAs (ksplit > 1) when the tiles would
// leave more than half of the SMs idle and a workspace `part` of the plan's part_elems
// fp32 values (made with allow_split) is given; a second launch then adds the partials in
// split order. Used for few tokens (ntok <= SWAP_MAX_TOKENS), and for the rank-L product of
// a layer whose Z has too few 256 x 256 tiles to occupy the CTA pairs.
struct SwapPlan {
    int bn = 128, tiles = 0, kblocks = 0, ksplit = 1, kb_per_split = 0;
    int64_t ld_part = 0, part_elems = 0;
};
SwapPlan gemm_swap_plan(int rows, int ntok, int kdim, int num_sms, bool allow_split);
// pdl: launched with programmatic stream serialization, so that it may start while the
// preceding grid on the stream finishes: W is read before that grid has completed (it
// must not be written by it), X only after. Its own successor may start early likewise.
cudaError_t launch_gemm_swap(const void* W, int64_t ldw, const void* X, int64_t ldx, int rows, int ntok, int kdim,
                             void* out, int64_t ldo, float* part, cudaStream_t stream, bool pdl = false);
constexpr int SWAP_MAX_TOKENS = 256;

// Whether the CTA-pair kernels are enabled (ESPACE_DISABLE_PAIR_GEMM=1 turns them off).
bool pair_kernel_enabled();

// Block-diagonal product on CTA pairs (tensor-parallel ranks folded onto one GPU): output
// column block g, C[:, c0[g] .. c0[g] + cw[g]) (bf16, leading dimension ldc), is
// A[:, ak0[g] .. ak0[g] + kdim) (A: rows x a_cols bf16, leading dimension lda) times
// B[c0[g] .. c0[g] + cw[g])[0 .. kdim) transposed (B: [sum cw][kdim] bf16, rows contiguous).
// The blocks tile the columns in order (c0[0] = 0, c0[g + 1] = c0[g] + cw[g]); at most 8
// blocks; kdim and every ak0 are multiples of 64.
cudaError_t launch_gemm_tn_blocks(const void* A, int64_t lda, int a_cols, const void* B, int rows, int nblocks,
                                  const int* ak0, const int* c0, const int* cw, int kdim, void* C, int64_t ldc,
                                  cudaStream_t stream);

// C[rows][cols] (bf16, leading dimension ldc) = A[rows][kdim] B[kdim][cols] with B stored
// row-major (its columns contiguous: an M/N-major tcgen05 operand), on CTA pairs; A and B
// bf16 with leading dimensions lda, ldb (multiples of 8).
cudaError_t launch_gemm_nn(const void* A, int64_t lda, const void* B, int64_t ldb, int rows, int cols, int kdim,
                           void* C, int64_t ldc, cudaStream_t stream);
// out[R][C] (fp32, leading dimension ldo) += U^T V for token-major U[N][R], V[N][C] (bf16,
// rows contiguous): a reduction over tokens, as for weight gradients; atomics, so out is
// zeroed by the caller for a plain product. R and C multiples of 8.
cudaError_t launch_gemm_tn_tokens_f32(const void* U, int R, const void* V, int C, int64_t N, float* out,
                                     int64_t ldo, cudaStream_t stream);

// S's upper triangle += that of sum_q U_q^T V_q, one launch: U_q and V_q are the seg_rows x K
// blocks of Q ([q_rows][K] bf16, rows contiguous) that start at rows seg_u[q] and seg_v[q]
// (multiples of 64, as is seg_rows; rows of a block past its data must be zero). At most 6
// segments.
cudaError_t launch_syrk_segments_upper(const void* Q, int64_t q_rows, int K, int seg_rows, int nseg,
                                       const int* seg_u, const int* seg_v, float* S, cudaStream_t stream);
// S[K][K] (fp32, upper triangle i <= j) += X^T X for X[N][K] bf16, on tcgen05 tensor cores.
// sched: two ints of the caller, zero before the first launch and left zero by every launch
// (the pair kernel's wave counter and exit counter; nullptr: no wave pacing).
cudaError_t launch_syrk_upper(const void* X, int64_t N, int K, float* S, cudaStream_t stream,
                              int* sched = nullptr);
// Two independent SYRKs in one launch: Sx += X^T X and Sy += Y^T Y (upper triangles), or
// Sx = X^T X and Sy = Y^T Y with assign (the lower triangles are then left unset).
cudaError_t launch_syrk_upper_two(const void* X, const void* Y, int64_t N, int K, float* Sx, float* Sy,
                                  bool assign, cudaStream_t stream);
// The same kernel with two operands: S's upper triangle += that of X^T Y (X, Y [N][K] bf16).
cudaError_t launch_syrk_cross_upper(const void* X, const void* Y, int64_t N, int K, float* S, cudaStream_t stream,
                                    int* sched = nullptr);

// Token counts served by the decode kernels (when asked for), and chosen for them by the
// automatic paths: above these, the swapped tcgen05 products measured faster.
constexpr int DECODE_MAX_TOKENS = 32;
constexpr int DECODE_AUTO_TOKENS = 16;
constexpr int DECODE_DENSE_AUTO_TOKENS = 8;

// Decode-shaped forward (nt <= DECODE_MAX_TOKENS) in one cooperative launch: Z[nt][Lp] = X P
// from P^T [Lp][K], a grid barrier, then Y[nt][M] = Z W' from W'^T [M][Lp]; each matrix
// streamed from HBM once. grid_bar: one unsigned int owned by the caller, zero before the
// first launch and left at a multiple of 2^31 by every launch that completes (one launch at a
// time may use it).
cudaError_t launch_decode_forward(const void* PT, const void* WfT, const void* X, void* Z, void* Y,
                                  int K, int Lp, int M, int nt, unsigned int* grid_bar,
                                  cudaStream_t stream);
// Dense decode product Y[nt][M] = X W^T with W [M][K] streamed once (same kernel, one phase).
cudaError_t launch_decode_dense(const void* W, const void* X, void* Y, int K, int M, int nt,
                                cudaStream_t stream);
bool decode_supported(int nt, int K, int Lp, int M, int num_sms);
bool decode_dense_supported(int nt, int K, int M, int num_sms);

// Xn[t][k] = bf16(X[t][k] / ||x_t||) (0 for a zero token), fp32 norms.
cudaError_t launch_normalize_rows(const void* X, int64_t N, int K, void* Xn, cudaStream_t stream);

// One thread waits on an mbarrier that never completes; after limit_ns it records
// ESPACE_ERR_TIMEOUT in the status word and returns.
cudaError_t launch_wait_timeout(uint64_t limit_ns, cudaStream_t stream);
// `ctas` CTAs that each hold one SM (200 KB of shared memory) for hold_ns, then leave.
cudaError_t launch_occupy(int ctas, uint64_t hold_ns, cudaStream_t stream);

// C[K][K] (fp64) = scale * (the symmetric matrix whose upper triangle is Su, fp32).
cudaError_t launch_sym_full_f64(const float* Su, int64_t K, double scale, double* C, cudaStream_t stream);
// The symmetric matrix whose upper triangle is Su (fp32, K x K), times scale, split into two
// bf16 matrices: hi = bf16(v), lo = bf16(v - hi), so that hi + lo carries 16 significant bits.
cudaError_t launch_sym_split_bf16(const float* Su, int64_t K, float scale, void* hi, void* lo, cudaStream_t stream);
// T = A B for K x K row-major fp64 matrices.
cudaError_t launch_gemm_f64(const double* A, const double* B, int K, double* T, cudaStream_t stream);

// dst[i] = bf16(src[i]) (round to nearest even).
cudaError_t launch_f32_to_bf16(const float* src, int64_t count, void* dst, cudaStream_t stream);

// Fills dst[count] with zeros (fp32).
cudaError_t launch_zero_f32(float* dst, int64_t count, cudaStream_t stream);

}  // namespace espace
