/*
 * espace.h -- C ABI of the GB300 (sm_103a) library for ESPACE's projected linear layer.
 *
 * ESPACE (arXiv 2410.05437) replaces a linear layer Y = W^T X (Sec. 2.1, Eq. 1) by
 * Y = (P^T W)^T (P^T X) (Sec. 2.2, Eq. 3), where P (K x L) holds the L principal
 * eigenvectors of the activation autocorrelation C = E[x x^T] (Sec. 3.1, Eq. 4, Thm. 1)
 * and W' = P^T W is folded once before deployment (Sec. 2.2).
 *
 * Letters: K = input features, M = output features, N = tokens, L = rank (1 <= L <= K).
 * Storage is row-major and token-major, as PyTorch keeps activations:
 *   X  [N][K] bf16    input tokens, one per row
 *   W  [M][K] bf16    dense weight in nn.Linear layout (row m = output feature m)
 *   Y  [N][M] bf16    output tokens
 * In this layout Eq. 3 reads Z[N][L] = X P and Y = Z W'.
 *
 * Conventions shared by every call:
 *   - "bf16" buffers hold IEEE bfloat16 bit patterns (uint16_t); "_dev" pointers are CUDA
 *     device pointers of the current device and must be 16-byte aligned; K must be a
 *     multiple of 8 and M a multiple of 8 (16-byte row pitch, needed by the TMA engine).
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Calls
 *     marked "async" only enqueue work on it; the caller synchronizes before reading results.
 *   - The caller owns X, W, Y and streams. The library owns handles and the device memory
 *     behind them (S, P^T, W'^T, the Z scratch) and frees it in the *_destroy calls.
 *   - A handle's scratch and sums are shared by its calls: calls on one handle must be
 *     ordered on the GPU (one stream, or streams that wait on each other) and must not be
 *     made from two host threads at once; calls on different handles may overlap.
 *   - Every int-returning call returns ESPACE_OK (0) or one of the ESPACE_ERR_* codes below;
 *     nothing throws across the ABI, a rejected argument never launches a kernel, and
 *     espace_last_error() describes the most recent failure of the calling thread.
 *   - Device-side waits are bounded: a kernel that gives up records ESPACE_ERR_TIMEOUT in a
 *     per-device status word, which espace_check() reports (and clears).
 */
#ifndef ESPACE_H
#define ESPACE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ESPACE_OK            0
#define ESPACE_ERR_ARG       1   /* null pointer or value out of range */
#define ESPACE_ERR_SHAPE     2   /* sizes inconsistent with the handle or unsupported */
#define ESPACE_ERR_ALIGN     3   /* pointer not 16-byte aligned */
#define ESPACE_ERR_CUDA      4   /* a CUDA runtime / driver call failed */
#define ESPACE_ERR_TIMEOUT   5   /* a device-side wait exceeded its limit */
#define ESPACE_ERR_STATE     6   /* call not valid in the handle's state (e.g. no tokens) */
#define ESPACE_ERR_NOMEM     7   /* device or host allocation failed */
#define ESPACE_ERR_NUMERIC   8   /* the host eigen-solver did not converge */

typedef struct espace_calib_s* espace_calib_t;   /* autocorrelation accumulator (Eq. 4)   */
typedef struct espace_proj_s*  espace_proj_t;    /* calibrated P^T and folded W'^T (Eq. 3) */

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
int espace_version(void);

/* Text for the calling thread's most recent failure ("" if none). Valid until the next
 * failing call on the same thread. */
const char* espace_last_error(void);

/* ---------------------------------------------------------------------------------------
 * Calibration (Sec. 3.1, Eq. 4): C = X X^T / n summed over calibration tokens. The paper
 * averages per-batch means; the library keeps the running sum S and the token count n and
 * forms C = S / n, which is the same estimate for equal-size batches and the token-weighted
 * mean otherwise. No mean is subtracted: C is Sec. 3.1's autocorrelation E[x x^T], not a
 * covariance.
 * ------------------------------------------------------------------------------------- */

/* Creates an accumulator for K-dimensional activations with S = 0, n = 0. Allocates an
 * fp32 K x K device buffer. K: multiple of 8, 8 <= K <= 65536. */
int espace_calib_create(int64_t K, espace_calib_t* out);

/* Async. S += X^T X over the N rows of X_dev ([N][K] bf16) and n += N, on tcgen05 tensor
 * cores with fp32 accumulation; only the upper triangle of S is stored. N = 0 is a no-op.
 * The host-side counter n is updated when the call is enqueued. */
int espace_calib_accumulate(espace_calib_t h, const void* X_dev, int64_t N, void* stream);

/* Same, with each token first scaled to unit L2 norm (Cor. 1: the autocorrelation of
 * x / ||x|| whose eigenvectors minimize the normalized MSE of Eq. 7). Tokens of zero norm
 * add nothing but still count in n. Do not mix with espace_calib_accumulate on one handle. */
int espace_calib_accumulate_normalized(espace_calib_t h, const void* X_dev, int64_t N,
                                       void* stream);

/* Async. Thm. 2's NL-MSE calibration (Sec. 3.3, App. A.4): for one calibration sequence of
 * T tokens with activations X_dev ([T][K] bf16) and the loss gradients with respect to them
 * G_dev ([T][K] bf16), adds C_i = (A B + B A) / T^2, A = X^T X, B = G^T G, to the
 * accumulator and counts one sequence (the paper's per-sequence approximation; C = S / n is
 * then the mean over sequences). normalized != 0 takes the L2-normalized variant (every
 * token row of X and of G divided by its norm first). A and B are formed on the tensor
 * cores (fp32), each split into bf16 hi + lo halves, and the products accumulated as
 * A_hi B_hi + A_hi B_lo + A_lo B_hi (and the same for B A) in fp32: about 2^-16 relative.
 * Cannot be mixed with the other accumulations on one handle (ESPACE_ERR_STATE). The first
 * call allocates 8 K (K + Kp) bytes of scratch on the handle, Kp = K rounded up to a
 * multiple of 64 (4 T K bytes more when normalized). Four launches per call.
 * C may be indefinite: espace_build_projection then orders eigenvalues by magnitude. */
int espace_calib_accumulate_nl(espace_calib_t h, const void* X_dev, const void* G_dev, int64_t T,
                               int normalized, void* stream);

/* Synchronizes `stream`, then writes C = S / n as a full symmetric K x K fp64 matrix
 * (C_host may be NULL) and the token count (n_out may be NULL). ESPACE_ERR_STATE if n = 0
 * and C_host != NULL. */
int espace_calib_read(espace_calib_t h, double* C_host, int64_t* n_out, void* stream);

/* Checkpointing of the accumulator: export copies the raw upper-triangular fp32 sum S
 * (K*K floats, row-major, lower triangle unspecified) and n to the host after synchronizing
 * `stream`; import replaces them. Exported sums of several shards may be added and imported
 * into one handle (the all-reduce step of data-parallel calibration). */
int espace_calib_export(espace_calib_t h, float* S_host, int64_t* n_out, void* stream);
int espace_calib_import(espace_calib_t h, const float* S_host, int64_t n, void* stream);

/* Resets S = 0 and n = 0 (async on `stream`). */
int espace_calib_reset(espace_calib_t h, void* stream);

void espace_calib_destroy(espace_calib_t h);

/* ---------------------------------------------------------------------------------------
 * Projection and fold (Thm. 1, Sec. 2.2)
 * ------------------------------------------------------------------------------------- */

/* Synchronous. Builds the projected layer from a calibrated accumulator:
 *   1. C = S / n in fp64 on the host;
 *   2. symmetric eigen-decomposition of C in fp64 on the host cores (Householder
 *      tridiagonalization in panels, divide and conquer on the tridiagonal, only the L
 *      kept eigenvectors carried back), eigenvalues sorted decreasing (Sec. 3.1), or
 *      by decreasing magnitude when C is not positive semidefinite (smallest eigenvalue
 *      below -1e-6 of the largest magnitude; e.g. an NL-MSE matrix), as the paper does;
 *   3. P = the first L eigenvectors (Thm. 1), each column's largest-magnitude entry made
 *      positive (lowest index on ties), rounded to bf16;
 *   4. W'^T = W P rounded to bf16, i.e. W' = P^T W (Sec. 2.2), on the GPU with fp32
 *      accumulation, from W_dev ([M][K] bf16, read once; the caller may free it after).
 * The handle keeps P^T as [Lp][K] and W'^T as [M][Lp] bf16 with L rounded up to Lp, a
 * multiple of 64; the padding rows/columns are zero, which leaves Y unchanged. */
int espace_build_projection(espace_calib_t h, const void* W_dev, int64_t M, int64_t L,
                            void* stream, espace_proj_t* out);

/* Synchronous. As espace_build_projection, with Thm. 2's criterion (GO-MSE, Sec. 3.3): P
 * holds the L principal eigenvectors of C = C_X C_W + C_W C_X, where C_X = S / n is the
 * handle's autocorrelation (plain, or normalized for the GO-MSE variant with L2
 * normalization) and C_W = W^T W / M is the autocorrelation of the M weight rows (computed
 * on the tensor cores), taking weights and activations as independent. C_W is formed and
 * C_X C_W multiplied in fp64 on the device; C may be indefinite, so eigenvalues (and
 * espace_proj_eigenvalues) are ordered by magnitude, largest first, as the paper does.
 * Temporary device memory: 28 K^2 bytes. */
int espace_build_projection_go(espace_calib_t h, const void* W_dev, int64_t M, int64_t L,
                               void* stream, espace_proj_t* out);

/* Synchronous. Same as steps 3 (rounding only) and 4 above for a given fp64 P_host
 * ([K][L], row-major), with no eigen-solve: used to feed one projection to several
 * implementations. */
int espace_proj_from_host(int64_t K, int64_t M, int64_t L, const double* P_host,
                          const void* W_dev, void* stream, espace_proj_t* out);

/* Synchronous. Step 4 above for a projection already on the device in bf16: PT_dev is P_b^T
 * as [L][K] row-major bf16 (the L principal directions as rows, e.g. computed by the caller
 * on the GPU, as the paper does, App. B.1); it is copied into the handle (the caller keeps
 * its buffer) and W' = P_b^T W is folded on the device. Both pointers 16-byte aligned. */
int espace_proj_from_device(int64_t K, int64_t M, int64_t L, const void* PT_dev,
                            const void* W_dev, void* stream, espace_proj_t* out);

/* Shape of a projection: any output pointer may be NULL. */
int espace_proj_shape(espace_proj_t p, int64_t* K, int64_t* M, int64_t* L);

/* The K eigenvalues of C in decreasing order (only for handles made by
 * espace_build_projection; ESPACE_ERR_STATE otherwise). */
int espace_proj_eigenvalues(espace_proj_t p, double* dst);

/* Copies P as bf16 [K][L] (row-major) to the host. */
int espace_proj_read_P(espace_proj_t p, uint16_t* P_host);

/* Copies W' as bf16 [L][M] (row-major) to the host. */
int espace_proj_read_Wfold(espace_proj_t p, uint16_t* Wf_host);

/* Checkpointing of a projection: export writes P^T [Lp][K] and W'^T [M][Lp] bf16 and the
 * K eigenvalues (zeros if unknown) to host buffers sized from espace_proj_shape (Lp = L
 * rounded up to a multiple of 64); import rebuilds a handle from them. */
int espace_proj_export(espace_proj_t p, uint16_t* PT_host, uint16_t* WfT_host, double* evals);
int espace_proj_import(int64_t K, int64_t M, int64_t L, const uint16_t* PT_host,
                       const uint16_t* WfT_host, const double* evals, espace_proj_t* out);

void espace_proj_destroy(espace_proj_t p);

/* ---------------------------------------------------------------------------------------
 * Training view (Sec. 2.2): during training or fine-tuning the layer is
 * Y = W^T (P P^T X) with P static and W trainable. In token-major storage the order that
 * saves work is Z = X P (kept for the backward pass: N x L instead of N x K), Y = Z (W P)^T,
 * with W' = P^T W refolded after every weight update. All calls below are asynchronous on
 * the caller's stream and need a plain (not tensor-parallel) handle (ESPACE_ERR_STATE).
 * ------------------------------------------------------------------------------------- */

/* W'^T = W P_b again, rounded to bf16, from new weights W_dev ([M][K] bf16). */
int espace_proj_refold(espace_proj_t p, const void* W_dev, void* stream);

/* Z_dev ([N][Lp] bf16, caller-owned; Lp = L rounded up to 64, columns >= L come out zero)
 * = bf16(X P_b) and Y_dev ([N][M] bf16) = bf16(Z W'), the products of
 * espace_linear_forward with Z written where the caller keeps it. */
int espace_train_forward(espace_proj_t p, const void* X_dev, int64_t N, void* Z_dev, void* Y_dev,
                         void* stream);

/* The backward pass of the training view for one micro-batch: for the output gradient
 * dY_dev ([N][M] bf16) and the Z_dev of its forward pass, dX_dev ([N][K] bf16) =
 * bf16(bf16(dY W'^T) P_b^T), the gradient with respect to the input (through P P^T), and
 * (dW P)^T += Z^T dY into an fp32 accumulator of the handle ([Lp][M]): 2 L N (2 M + K)
 * flop against the dense layer's 4 N M K. Scratch on the handle: N Lp + 6 Lp M bytes (the
 * first call with a larger N grows it synchronously). */
int espace_train_backward(espace_proj_t p, const void* dY_dev, const void* Z_dev, int64_t N,
                          void* dX_dev, void* stream);

/* At the end of a step (after the micro-batches' backward passes): dW_dev ([M][K] fp32,
 * overwritten) = bf16(sum of dY^T Z) P_b^T, the gradient with respect to W (2 L M K flop,
 * once per step), and the accumulator is cleared for the next step. */
int espace_train_weight_grad(espace_proj_t p, float* dW_dev, void* stream);

/* The dense layer's backward pass (Eq. 1): dX_dev ([N][K] bf16) = bf16(dY W) and dW_dev
 * ([M][K] fp32) = dY^T X, or dW_dev += dY^T X when accumulate != 0 (micro-batches of one
 * step), for dY_dev [N][M], X_dev [N][K], W_dev [M][K]. */
int espace_dense_backward(const void* dY_dev, int64_t N, const void* X_dev, int64_t K,
                          const void* W_dev, int64_t M, void* dX_dev, float* dW_dev, int accumulate,
                          void* stream);

/* ---------------------------------------------------------------------------------------
 * Tensor-parallel layers folded onto one GPU (App. B.2, Table 2; latency method of App. B.4)
 *
 * Under tensor parallelism the paper applies ESPACE per rank, each rank r of tp with its
 * own projection P_r of L components. Folded onto one GPU the layer computes, for
 *   ESPACE_TP_COLUMN (column-parallel: QKV, FC1; rank r holds all K inputs and the output
 *   columns [r M/tp, (r+1) M/tp)):  Y[:, r M/tp ..] = bf16(X P_r) W'_r,  W'_r = P_r^T W_r^T
 *   with W_r the rank's M/tp rows of W (P_r: K x L);
 *   ESPACE_TP_ROW (row-parallel: attention projection, FC2; rank r holds the inputs
 *   [r K/tp, (r+1) K/tp) and all M outputs):  Y = sum_r bf16(X_r P_r) W'_r,
 *   W'_r = P_r^T W[:, r K/tp ..]^T (P_r: K/tp x L).
 * Both are two products: one dense and one block-diagonal with one block per rank (the
 * second for COLUMN, the first for ROW), each a tcgen05 launch on CTA pairs; Z ([N][tp L],
 * the ranks' intermediates side by side) is rounded to bf16 as in the plain layer.
 * Shapes: 1 <= tp <= 8; L a multiple of 64 with L <= K / tp (ROW) or L <= K (COLUMN);
 * COLUMN: M / tp a positive multiple of 8; ROW: K / tp a multiple of 64. The forward
 * calls (espace_linear_forward, _path with any path, _launches) accept these handles and
 * always run the two launches; espace_proj_read_P writes the tp bf16 projections as
 * [tp][Kr][L]; espace_proj_read_Wfold, _export and espace_linear_forward_noalloc return
 * ESPACE_ERR_STATE for them.
 * ------------------------------------------------------------------------------------- */
#define ESPACE_TP_COLUMN 1
#define ESPACE_TP_ROW    2

/* Synchronous. A tensor-parallel layer from tp given fp64 projections P_host, [tp][Kr][L]
 * row-major (Kr = K for COLUMN, K / tp for ROW), each rounded to bf16, and W_dev ([M][K]
 * bf16, read once): the ranks' W'_r are folded on the GPU (fp32 accumulation, bf16). */
int espace_proj_tp_from_host(int kind, int tp, int64_t K, int64_t M, int64_t L, const double* P_host,
                             const void* W_dev, void* stream, espace_proj_t* out);

/* Synchronous. As espace_build_projection (Thm. 1 per rank) for a tensor-parallel layer:
 * rank r's autocorrelation is that of its own inputs. ROW: the r-th diagonal K/tp x K/tp
 * block of C = S / n (tp eigen-solves of size K / tp; the handle's eigenvalues are the tp
 * ranks' K / tp values, each block decreasing). COLUMN: every rank sees all K inputs, so
 * the ranks' projections coincide and the call is espace_build_projection with the rank's
 * L (Table 2's per-rank L), returning a plain handle; only tp's range is checked. Needs a
 * plain or normalized activation accumulation (ESPACE_ERR_STATE after NL-MSE). */
int espace_build_projection_tp(espace_calib_t h, const void* W_dev, int64_t M, int64_t L, int kind, int tp,
                               void* stream, espace_proj_t* out);

/* The handle's tensor-parallel kind (0 for a plain layer) and rank count (1 for a plain
 * layer). Either pointer may be null. */
int espace_proj_tp_info(espace_proj_t p, int* kind, int* tp);

/* ---------------------------------------------------------------------------------------
 * Forward (Sec. 2.2, Eq. 3)
 * ------------------------------------------------------------------------------------- */

/* Async. Y = (P^T W)^T (P^T X) for the N tokens of X_dev ([N][K] bf16) into Y_dev
 * ([N][M] bf16): Z = X P is accumulated in fp32 and rounded to bf16 (the paper computes in
 * BF16, App. B.1), then Y = Z W' is accumulated in fp32 and rounded to bf16. N <= 16 runs
 * a bandwidth-bound kernel that streams P and W' once (when the layer fits it); N <= 256
 * runs one tcgen05 launch per product with the weights as the 128-row operand, a product
 * whose tiles would leave more than half of the SMs idle splitting its reduction over them
 * (one more launch adds the fp32 partials in a fixed order, so results are reproducible bit
 * for bit); larger N runs one persistent tcgen05 launch holding both products, except that
 * a layer with K >= 2 M whose Z has fewer 256 x 256 tiles than a quarter of the SMs runs
 * phase 1 as a split product and phase 2 on CTA pairs. The few-token and decode launches
 * (N <= 256) may start streaming the handle's P and W' while the kernel before them on the
 * stream finishes (programmatic dependent launch); they read X_dev only after it has
 * completed.
 * N = 0 is a no-op. The first call
 * with a larger N than any before on this handle allocates the Z scratch and the split
 * workspace (synchronously, so outside a stream capture); later calls allocate nothing. */
int espace_linear_forward(espace_proj_t p, const void* X_dev, int64_t N, void* Y_dev,
                          void* stream);

/* As espace_linear_forward with the kernel family chosen by the caller:
 *   0 automatic;
 *   1 tcgen05 tensor-core kernels: for N <= 256 one launch per product with the weights as
 *     the 128-row operand; above, one persistent launch holding both products when L and M
 *     exceed 128 (Z stays in L2 between them), else one launch per product;
 *   2 the decode-shaped streaming kernel (ESPACE_ERR_SHAPE if N > 32 or the layer is too
 *     large for it);
 *   3 tcgen05 kernels, always one launch per product (Z through the scratch buffer). */
#define ESPACE_PATH_AUTO         0
#define ESPACE_PATH_TENSOR       1
#define ESPACE_PATH_SMALL_N      2
#define ESPACE_PATH_TENSOR_SPLIT 3
int espace_linear_forward_path(espace_proj_t p, const void* X_dev, int64_t N, void* Y_dev,
                               void* stream, int path);

/* Number of kernel launches espace_linear_forward_path(p, ., N, ., ., path) makes (0 for
 * N = 0), or -1 for invalid arguments or a path that cannot take N. Host-only query. */
int espace_linear_forward_launches(espace_proj_t p, int64_t N, int path);

/* Synchronous. The forward of espace_linear_forward for X and Y in host memory: X_host
 * ([N][K] bf16) is copied to device staging owned by the handle, the products run on the
 * caller's stream, and Y ([N][M] bf16) is copied back into Y_host; the call returns with
 * Y_host filled (work already on the caller's stream runs first, and later work on it
 * waits for the copies). N is cut into up to 8 chunks of at least 512 tokens: the copy of
 * chunk j + 1 in, chunk j's products and the copy of chunk j - 1 out overlap, on two
 * streams of the handle. Pinned (page-locked) host buffers let the copies run
 * asynchronously; pageable ones still give the right result. The first call with a larger
 * N than any before allocates the staging (N (K + M) bf16 values). One call at a time per
 * handle. */
int espace_linear_forward_host(espace_proj_t p, const void* X_host, int64_t N, void* Y_host,
                               void* stream);

/* Async. espace_linear_forward_host without the final wait: the copies and products are
 * queued as described there (in up to 8 chunks of at least 8192 tokens), the caller's stream
 * is ordered after the last copy out, and the call returns. X_host must not change, and Y_host is not filled, until the caller's stream
 * reaches that point (synchronize it, or an event recorded on it after the call). Calls on
 * one handle must be ordered on one stream (they share the handle's staging); independent
 * layers on separate streams overlap one layer's copies with another's products. The first
 * call with a larger N than any before synchronizes the stream and allocates the staging
 * (outside a stream capture). An error after copies were queued waits for them before
 * returning, so no copy touches the host buffers after an error return. */
int espace_linear_forward_host_async(espace_proj_t p, const void* X_host, int64_t N, void* Y_host,
                                     void* stream);

/* Synchronous. The host-buffer forward of several independent layers in one pipeline:
 * layer i (handle layers[i]) maps X_host[i] ([N[i]][K_i] bf16) to Y_host[i] ([N[i]][M_i]
 * bf16) with the products of espace_linear_forward. The handles must be distinct and on
 * one device. Every copy in runs on one copy stream and every product on the caller's
 * stream, both in layer order, in token chunks of about 8192 (up to 8 per layer). The first
 * layer leads with chunks of 2048 and 4096 tokens, and the last layer ends with one of 2048,
 * where N leaves room. Every copy out runs on a second copy stream, so layer i + 1's tokens
 * are copied in while layer i computes and layer i's outputs are copied out while layer
 * i + 1 computes, with one product running at a time. Pinned host buffers let the copies overlap; pageable ones still give the right
 * result. Work already on the caller's stream runs first; the call returns with every
 * Y_host[i] filled. count <= ESPACE_HOST_MANY_MAX, and N[i] = 0 skips layer i. A handle's
 * first call with a larger N than any before allocates its staging, as
 * espace_linear_forward_host does. Errors (nothing is queued):
 *   ESPACE_ERR_ARG for null arrays, handles or buffers, a repeated handle, or handles on
 *     different devices;
 *   ESPACE_ERR_STATE for a tensor-parallel handle;
 *   ESPACE_ERR_SHAPE for a bad N[i]. */
#define ESPACE_HOST_MANY_MAX 16
int espace_linear_forward_host_many(int count, const espace_proj_t* layers, const void* const* X_host,
                                    const int64_t* N, void* const* Y_host, void* stream);

/* Capacity, in bf16 values, of the fixed scratch used by espace_linear_forward_noalloc:
 * 16 MiB, enough for N * Lp <= 8,388,608 (e.g. 4096 tokens at L = 2048). */
#define ESPACE_NOALLOC_Z_ELEMS 8388608

/* Async. The projected forward of espace_linear_forward, equal to it within the parity
 * tolerances, for callers that cannot
 * allocate device memory during the call -- for example code that runs inside a memory
 * budget or pool owned by someone else, or a server that reserved all device memory at
 * start-up. Instead of the handle's growable Z scratch it uses one fixed array of
 * ESPACE_NOALLOC_Z_ELEMS bf16 values that is part of the library image on every device
 * that loads the library (held until the process exits); the call itself allocates
 * nothing. The paper has no counterpart: it is an interface convenience of this library.
 *   - Kernels: the decode kernel for N <= 32 when the layer fits it (the automatic path
 *     takes it only up to 16 tokens), else one tcgen05 launch per product with Z through
 *     the fixed array (the automatic path may instead run both products in one launch, or
 *     split a reduction over the SMs); results can differ from espace_linear_forward's in
 *     the last bf16 bit, and the speed differs.
 *   - N * Lp (Lp = L rounded up to a multiple of 64) above ESPACE_NOALLOC_Z_ELEMS is
 *     rejected with ESPACE_ERR_SHAPE before anything is launched.
 *   - The handle's device must be current (ESPACE_ERR_STATE otherwise).
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress); make that first call before any stream capture.
 *   - All calls on a device share the array and it keeps the last call's contents (each
 *     call overwrites the part it reads); calls whose kernels overlap on the GPU, e.g. on
 *     two unordered streams, race on it. */
int espace_linear_forward_noalloc(espace_proj_t p, const void* X_dev, int64_t N, void* Y_dev,
                                  void* stream);

/* Async. The uncompressed layer of Eq. 1, Y = W^T X, as Y_dev[N][M] = X_dev[N][K] W_dev^T
 * with W_dev in [M][K] layout, with fp32 accumulation and bf16 output on the same kernel
 * families as the projected layer (N <= 8: the streaming kernel; N <= 256: tcgen05 with
 * the weights as the 128-row operand, the reduction split over the SMs in the same cases
 * as the projected layer's products, with fp32 partials in a per-device workspace that
 * the first such call allocates, or grows, and so must make outside a stream capture;
 * above: tcgen05): the baseline the projected layer is measured against. Calls that split
 * share the device's workspace: order them on the GPU (one stream, or streams that wait on
 * each other). For N <= 256 the product may start reading W_dev while the kernel
 * launched just before it on the stream finishes, when that kernel is one of this
 * library's few-token products (programmatic dependent launch); X_dev is read only after
 * that kernel completes. So W_dev must not be written by the call made just before on
 * the same stream. */
int espace_dense_forward(const void* X_dev, int64_t N, int64_t K, const void* W_dev,
                         int64_t M, void* Y_dev, void* stream);

/* Synchronizes `stream` and reports (then clears) the device status word: ESPACE_OK, or
 * ESPACE_ERR_TIMEOUT if a kernel gave up waiting since the last check, or ESPACE_ERR_CUDA
 * if the stream reported an error. */
int espace_check(void* stream);

/* Measurement hook: the next espace_linear_forward / espace_linear_forward_path call on
 * this thread records `event` (a cudaEvent_t) on its stream between the rank-L projection
 * kernel (Z = X P) and the folded-weight kernel (Y = Z W'), so that the two products of
 * Eq. 3 can be timed separately. One-shot: cleared by that call. NULL cancels. */
int espace_set_phase_event(void* event);

/* Test hook: upper bound in nanoseconds for every device-side wait of later launches
 * (default 4e9). 0 restores the default. */
int espace_set_wait_limit_ns(uint64_t ns);

/* Test hook for the bounded waits: launches (async) one thread that waits on a barrier
 * nothing completes, gives up after limit_ns (at most 1e9) and records ESPACE_ERR_TIMEOUT,
 * so that the next espace_check() reports it. Nothing faults and the context stays usable. */
int espace_debug_wait_timeout(uint64_t limit_ns, void* stream);

/* Test hook for persistent kernels sharing the GPU: launches (async) `ctas` CTAs (1 .. the
 * SM count), each holding one SM with 200 KB of shared memory for hold_ns (at most 1e9),
 * so that a kernel launched meanwhile on another stream finds only the other SMs free. */
int espace_debug_occupy(int ctas, uint64_t hold_ns, void* stream);

/* ---------------------------------------------------------------------------------------
 * Host-only helper (no GPU needed)
 * ------------------------------------------------------------------------------------- */

/* fp64 symmetric eigen-decomposition used by espace_build_projection (panel Householder
 * tridiagonalization, divide and conquer, compact-WY back-transformation): A_host is
 * K x K row-major symmetric (only read); w receives the eigenvalues in decreasing order and
 * V (K x K row-major, may be NULL) the unit eigenvectors as columns, with the sign
 * convention of espace_build_projection. ESPACE_ERR_NUMERIC if the implicit QR of a small
 * tridiagonal block does not converge. Uses up to `threads` host threads (0 = all cores;
 * a positive value sets the OpenMP thread count of the process). */
int espace_host_eigh(const double* A_host, int64_t K, double* w, double* V, int threads);

#ifdef __cplusplus
}
#endif

#endif /* ESPACE_H */
