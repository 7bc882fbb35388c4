/*
 * espace_oracle.c -- plain, slow fp64 reference of ESPACE's projected linear layer.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product library calls, links or includes this
 * file; only the tests, the smoke check and the benchmark's CPU-baseline leg use it. It
 * shares no code, header, table or constant with the CUDA path.
 *
 * Letters: K = input features, M = output features, N = tokens, L = rank. All matrices are
 * row-major fp64. Where the method rounds to bf16, the oracle rounds its fp64 value once,
 * to nearest with ties to even, and keeps the rounded value in fp64.
 *
 *   oracle_bf16_round        rounding of a real number to the nearest bf16 value
 *   oracle_autocorr_sum      S += sum_t x_t x_t^T                      (Sec. 3.1, Eq. 4)
 *   oracle_autocorr_rows     the same for selected rows of S            (Sec. 3.1, Eq. 4)
 *   oracle_jacobi_eigh       C = V D V^T, eigenvalues sorted decreasing (Sec. 3.1, Thm. 1)
 *   oracle_fold              W' = P^T W                                 (Sec. 2.2, Eq. 3)
 *   oracle_project           Z = P^T X (stored token-major as X P)      (Sec. 2.2, Eq. 3)
 *   oracle_contract          Y = W'^T Z                                 (Sec. 2.2, Eq. 3)
 *   oracle_reconstruct       x~ = sum_i <p_i, x> p_i                    (Sec. 3.2, Eq. 5)
 *   oracle_projection_mse    E ||x - x~||^2                             (Sec. 3.2, Eq. 6)
 *   oracle_dense             Y = W^T X                                  (Sec. 2.1, Eq. 1)
 *   oracle_autocorr_normalized_sum  sum_t (x_t/|x_t|)(x_t/|x_t|)^T     (Sec. 3.2, Cor. 1)
 *   oracle_go_combine        C = C_X C_W + C_W C_X                      (Sec. 3.3, Thm. 2)
 *
 * The OpenMP pragmas only split the outermost token / row loop across host cores; each
 * output element is still summed in the plain order of its definition.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* Nearest bf16 value of v, ties to even. bf16 keeps 8 significant bits (7 stored) and the
 * fp32 exponent range: normal numbers from 2^-126, subnormal spacing 2^-133, largest
 * finite value (2 - 2^-7) * 2^127; anything that rounds beyond it becomes infinity. */
double oracle_bf16_round(double v)
{
    if (v != v || v == 0.0 || isinf(v)) return v;
    double a = fabs(v);
    int e;
    frexp(a, &e);                 /* a = f * 2^e with 0.5 <= f < 1, so 2^(e-1) <= a < 2^e */
    int lsb_exp = (e - 1) - 7;    /* spacing of bf16 numbers in [2^(e-1), 2^e) */
    if (lsb_exp < -133) lsb_exp = -133;
    double q = ldexp(a, -lsb_exp);        /* exact: power-of-two scaling */
    double fl = floor(q);
    double rem = q - fl;                  /* exact */
    double r;
    if (rem > 0.5) r = fl + 1.0;
    else if (rem < 0.5) r = fl;
    else r = (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
    double out = ldexp(r, lsb_exp);
    const double max_finite = ldexp(255.0, 120);   /* (2 - 2^-7) * 2^127 */
    if (out > max_finite) out = INFINITY;
    return v < 0 ? -out : out;
}

void oracle_bf16_round_array(double* a, int64_t count)
{
    for (int64_t i = 0; i < count; ++i) a[i] = oracle_bf16_round(a[i]);
}

/* Eq. 4: X X^T = x_1 x_1^T + ... + x_n x_n^T, accumulated into the full K x K matrix S.
 * X is [n][K] (one token per row). The caller divides by the token count to get C. */
void oracle_autocorr_sum(const double* X, int64_t n, int64_t K, double* S)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < K; ++i) {
        for (int64_t t = 0; t < n; ++t) {
            const double xi = X[t * K + i];
            for (int64_t j = 0; j < K; ++j) S[i * K + j] += xi * X[t * K + j];
        }
    }
}

/* Eq. 4 restricted to the rows listed in `rows` (nrows of them): S[r][j] += sum_t
 * X[t][rows[r]] X[t][j], S being nrows x K. */
void oracle_autocorr_rows(const double* X, int64_t n, int64_t K, const int64_t* rows, int64_t nrows,
                          double* S)
{
    #pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < nrows; ++r) {
        const int64_t i = rows[r];
        for (int64_t t = 0; t < n; ++t) {
            const double xi = X[t * K + i];
            for (int64_t j = 0; j < K; ++j) S[r * K + j] += xi * X[t * K + j];
        }
    }
}

/* Corollary 1: the input-normalized autocorrelation sums (x/|x|)(x/|x|)^T. A token whose
 * norm is zero contributes nothing. */
void oracle_autocorr_normalized_sum(const double* X, int64_t n, int64_t K, double* S)
{
    for (int64_t t = 0; t < n; ++t) {
        double nrm2 = 0.0;
        for (int64_t j = 0; j < K; ++j) nrm2 += X[t * K + j] * X[t * K + j];
        if (nrm2 == 0.0) continue;
        for (int64_t i = 0; i < K; ++i)
            for (int64_t j = 0; j < K; ++j)
                S[i * K + j] += X[t * K + i] * X[t * K + j] / nrm2;
    }
}

/* Cyclic-by-row Jacobi eigenvalue iteration for a symmetric K x K matrix A (destroyed).
 * Each (p, q) step zeroes A[p][q] with the symmetric 2x2 Schur rotation
 *   tau = (a_qq - a_pp) / (2 a_pq),  t = sign(tau) / (|tau| + sqrt(1 + tau^2)),
 *   c = 1 / sqrt(1 + t^2),  s = t c,
 * applied as A <- J^T A J and V <- V J. Sweeps stop once the off-diagonal Frobenius norm is
 * at most tol * ||A||_F, or after max_sweeps. On return w holds the eigenvalues in
 * decreasing order (the order Sec. 3.1 assumes) and column i of V (row-major K x K) the
 * matching unit eigenvector. Returns the number of sweeps run. */
int oracle_jacobi_eigh(double* A, int64_t K, double* w, double* V, int max_sweeps, double tol)
{
    for (int64_t i = 0; i < K; ++i)
        for (int64_t j = 0; j < K; ++j) V[i * K + j] = (i == j) ? 1.0 : 0.0;
    double fro2 = 0.0;
    for (int64_t i = 0; i < K * K; ++i) fro2 += A[i] * A[i];
    int sweep = 0;
    for (; sweep < max_sweeps; ++sweep) {
        double off2 = 0.0;
        for (int64_t i = 0; i < K; ++i)
            for (int64_t j = 0; j < K; ++j)
                if (i != j) off2 += A[i * K + j] * A[i * K + j];
        if (off2 <= tol * tol * fro2) break;
        for (int64_t p = 0; p < K - 1; ++p) {
            for (int64_t q = p + 1; q < K; ++q) {
                double apq = A[p * K + q];
                if (apq == 0.0) continue;
                double tau = (A[q * K + q] - A[p * K + p]) / (2.0 * apq);
                double t = (tau >= 0.0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
                double c = 1.0 / sqrt(1.0 + t * t);
                double s = t * c;
                /* A <- A J : columns p and q */
                for (int64_t k = 0; k < K; ++k) {
                    double akp = A[k * K + p], akq = A[k * K + q];
                    A[k * K + p] = c * akp - s * akq;
                    A[k * K + q] = s * akp + c * akq;
                }
                /* A <- J^T A : rows p and q */
                for (int64_t k = 0; k < K; ++k) {
                    double apk = A[p * K + k], aqk = A[q * K + k];
                    A[p * K + k] = c * apk - s * aqk;
                    A[q * K + k] = s * apk + c * aqk;
                }
                /* V <- V J */
                for (int64_t k = 0; k < K; ++k) {
                    double vkp = V[k * K + p], vkq = V[k * K + q];
                    V[k * K + p] = c * vkp - s * vkq;
                    V[k * K + q] = s * vkp + c * vkq;
                }
            }
        }
    }
    for (int64_t i = 0; i < K; ++i) w[i] = A[i * K + i];
    /* selection sort into decreasing order, permuting the columns of V alongside */
    for (int64_t i = 0; i < K; ++i) {
        int64_t best = i;
        for (int64_t j = i + 1; j < K; ++j)
            if (w[j] > w[best]) best = j;
        if (best != i) {
            double tmp = w[i]; w[i] = w[best]; w[best] = tmp;
            for (int64_t k = 0; k < K; ++k) {
                double v = V[k * K + i]; V[k * K + i] = V[k * K + best]; V[k * K + best] = v;
            }
        }
    }
    return sweep;
}

/* W' = P^T W (Sec. 2.2: folded offline by associativity). P is K x L, W is stored [M][K]
 * (row m is output feature m, i.e. column m of the paper's K x M weight), and the result
 * Wf is L x M:  Wf[l][m] = sum_k P[k][l] W[m][k]. round_bf16 != 0 rounds each entry. */
void oracle_fold(const double* P, const double* W, int64_t K, int64_t M, int64_t L,
                 double* Wf, int round_bf16)
{
    #pragma omp parallel for schedule(static)
    for (int64_t l = 0; l < L; ++l) {
        for (int64_t m = 0; m < M; ++m) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) acc += P[k * L + l] * W[m * K + k];
            Wf[l * M + m] = round_bf16 ? oracle_bf16_round(acc) : acc;
        }
    }
}

/* Z = P^T X for tokens stored one per row: Z[t][l] = <p_l, x_t> = sum_k X[t][k] P[k][l].
 * X is N x K, P is K x L, Z is N x L. round_bf16 != 0 rounds each entry. */
void oracle_project(const double* X, const double* P, int64_t N, int64_t K, int64_t L,
                    double* Z, int round_bf16)
{
    #pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t) {
        for (int64_t l = 0; l < L; ++l) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) acc += X[t * K + k] * P[k * L + l];
            Z[t * L + l] = round_bf16 ? oracle_bf16_round(acc) : acc;
        }
    }
}

/* Y = (P^T W)^T (P^T X): Y[t][m] = sum_l Z[t][l] Wf[l][m]. Z is N x L, Wf is L x M. */
void oracle_contract(const double* Z, const double* Wf, int64_t N, int64_t L, int64_t M,
                     double* Y)
{
    #pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t) {
        for (int64_t m = 0; m < M; ++m) {
            double acc = 0.0;
            for (int64_t l = 0; l < L; ++l) acc += Z[t * L + l] * Wf[l * M + m];
            Y[t * M + m] = acc;
        }
    }
}

/* Eq. 1: Y = W^T X, per token Y[t][m] = sum_k W[m][k] X[t][k]. W stored [M][K]. */
void oracle_dense(const double* X, const double* W, int64_t N, int64_t K, int64_t M, double* Y)
{
    #pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t) {
        for (int64_t m = 0; m < M; ++m) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) acc += W[m * K + k] * X[t * K + k];
            Y[t * M + m] = acc;
        }
    }
}

/* Eq. 5: x~ = sum_{i<=L} <p_i, x> p_i for every token row of X (N x K); P is K x L. */
void oracle_reconstruct(const double* X, const double* P, int64_t N, int64_t K, int64_t L,
                        double* Xt)
{
    for (int64_t t = 0; t < N; ++t) {
        for (int64_t k = 0; k < K; ++k) Xt[t * K + k] = 0.0;
        for (int64_t i = 0; i < L; ++i) {
            double dot = 0.0;
            for (int64_t k = 0; k < K; ++k) dot += P[k * L + i] * X[t * K + k];
            for (int64_t k = 0; k < K; ++k) Xt[t * K + k] += dot * P[k * L + i];
        }
    }
}

/* Eq. 6: the sample mean of ||x - x~||^2 over the N token rows of X, with x~ from Eq. 5. */
double oracle_projection_mse(const double* X, const double* P, int64_t N, int64_t K, int64_t L)
{
    double total = 0.0;
    double xt[K > 0 ? K : 1];
    double dots[L > 0 ? L : 1];
    for (int64_t t = 0; t < N; ++t) {
        for (int64_t i = 0; i < L; ++i) {
            double dot = 0.0;
            for (int64_t k = 0; k < K; ++k) dot += P[k * L + i] * X[t * K + k];
            dots[i] = dot;
        }
        for (int64_t k = 0; k < K; ++k) {
            double acc = 0.0;
            for (int64_t i = 0; i < L; ++i) acc += dots[i] * P[k * L + i];
            xt[k] = acc;
        }
        double err = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            double d = X[t * K + k] - xt[k];
            err += d * d;
        }
        total += err;
    }
    return N > 0 ? total / (double)N : 0.0;
}

/* Thm. 2 (GO-MSE): C = C_X C_W + C_W C_X for K x K matrices, each entry summed in index
 * order. With C_X = E[x x^T] and C_W = E[w w^T] of independent x and w this is
 * E[x x^T w w^T + w w^T x x^T], the matrix whose principal eigenvectors minimize the bound
 * on the GEMM-output error of Prop. 1. */
void oracle_go_combine(const double* CX, const double* CW, int64_t K, double* C)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < K; ++i)
        for (int64_t j = 0; j < K; ++j) {
            double a = 0.0, b = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                a += CX[i * K + k] * CW[k * K + j];
                b += CW[i * K + k] * CX[k * K + j];
            }
            C[i * K + j] = a + b;
        }
}
