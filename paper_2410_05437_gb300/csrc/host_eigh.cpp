// host_eigh.cpp -- fp64 symmetric eigen-decomposition on the host for
// espace_build_projection (Thm. 1 needs the principal eigenvectors of the K x K
// autocorrelation; the paper runs this step off the hot path, App. B.1).
//
// Method:
//   1. Householder tridiagonalization A = Q T Q^T in panels (Golub & Van Loan, "Matrix
//      Computations", Sec. 8.3.1, with the panel form of Dongarra, Sorensen & Hammarling,
//      1989): NB columns are reduced against the trailing matrix as it was at the panel's
//      start, their effect on the later columns carried by two matrices V, W; the trailing
//      matrix is then updated once per panel, A -= V W^T + W V^T, as cache-blocked products.
//      The matrix-vector product with the trailing matrix reads its lower triangle once.
//   2. Eigenvalues and eigenvectors of T by divide and conquer (Cuppen, 1981; Golub & Van
//      Loan Sec. 8.4.4): T is torn into two halves plus a rank-one term, the halves are
//      solved recursively, and each join solves the secular equation of D + rho z z^T
//      (bisection in a variable shifted to the nearer pole, so that every difference d_j -
//      lambda is formed accurately), after deflating small z entries and close pairs of d.
//      The eigenvectors of the join come from the z recomputed from the roots (Gu &
//      Eisenstat, 1995), which keeps them orthogonal to working precision. Blocks of at most
//      32 rows use implicit QR steps with the Wilkinson shift.
//   3. The wanted eigenvectors of T are carried back through the reflectors, NB at a time
//      in compact WY form (I - V T V^T).
// All O(K^3) work is in cache-blocked, OpenMP-parallel loops; only the eigenvectors the
// caller selects (from all the eigenvalues) are formed at the last join and carried back.
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <functional>
#include <numeric>
#include <vector>

#include "../../include/espace.h"

namespace espace {

namespace {

constexpr double EPS = 2.220446049250313e-16;

inline int64_t imin(int64_t a, int64_t b) { return a < b ? a : b; }
inline int64_t imax(int64_t a, int64_t b) { return a > b ? a : b; }

// ============================================================================ products
// Column-major: X(i, j) = X[i + j * ld].

constexpr int MR = 8, NR = 4;
constexpr int64_t MC = 128, NC = 256, KC = 256;

// op(A) block rows [i0, i0 + mc) x columns [p0, p0 + kc), packed as MR-row slivers.
void pack_a(const double* A, int64_t lda, bool ta, int64_t i0, int64_t p0, int64_t mc, int64_t kc, double* dst)
{
    for (int64_t s = 0; s < mc; s += MR) {
        const int64_t rows = imin(MR, mc - s);
        double* out = dst + s * kc;
        for (int64_t p = 0; p < kc; ++p, out += MR) {
            const int64_t k = p0 + p;
            for (int64_t r = 0; r < MR; ++r) {
                const int64_t i = i0 + s + r;
                out[r] = r < rows ? (ta ? A[k + i * lda] : A[i + k * lda]) : 0.0;
            }
        }
    }
}

// op(B) block rows [p0, p0 + kc) x columns [j0, j0 + nc), packed as NR-column slivers.
void pack_b(const double* B, int64_t ldb, bool tb, int64_t p0, int64_t j0, int64_t kc, int64_t nc, double* dst)
{
    for (int64_t s = 0; s < nc; s += NR) {
        const int64_t cols = imin(NR, nc - s);
        double* out = dst + s * kc;
        for (int64_t p = 0; p < kc; ++p, out += NR) {
            const int64_t k = p0 + p;
            for (int64_t c = 0; c < NR; ++c) {
                const int64_t j = j0 + s + c;
                out[c] = c < cols ? (tb ? B[j + k * ldb] : B[k + j * ldb]) : 0.0;
            }
        }
    }
}

// C[0..mr) x [0..nr) += alpha * (packed a sliver) (packed b sliver)
inline void micro_kernel(int64_t kc, const double* a, const double* b, double* C, int64_t ldc, int64_t mr,
                         int64_t nr, double alpha)
{
    double acc[NR][MR];
    for (int c = 0; c < NR; ++c)
        for (int r = 0; r < MR; ++r) acc[c][r] = 0.0;
    for (int64_t p = 0; p < kc; ++p) {
        const double* ap = a + p * MR;
        const double* bp = b + p * NR;
        for (int c = 0; c < NR; ++c) {
            const double bv = bp[c];
            for (int r = 0; r < MR; ++r) acc[c][r] += ap[r] * bv;
        }
    }
    for (int64_t c = 0; c < nr; ++c)
        for (int64_t r = 0; r < mr; ++r) C[r + c * ldc] += alpha * acc[c][r];
}

// C[i0.., j0..] (mc x nc tile) += alpha op(A) op(B) over the whole k, sequential.
void gemm_tile(bool ta, bool tb, int64_t mc, int64_t nc, int64_t k, double alpha, const double* A, int64_t lda,
               int64_t i0, const double* B, int64_t ldb, int64_t j0, double* C, int64_t ldc, std::vector<double>& pa,
               std::vector<double>& pb)
{
    const int64_t mcp = (mc + MR - 1) / MR * MR, ncp = (nc + NR - 1) / NR * NR;
    pa.resize(static_cast<size_t>(mcp * KC));
    pb.resize(static_cast<size_t>(ncp * KC));
    for (int64_t p0 = 0; p0 < k; p0 += KC) {
        const int64_t kc = imin(KC, k - p0);
        pack_b(B, ldb, tb, p0, j0, kc, nc, pb.data());
        pack_a(A, lda, ta, i0, p0, mc, kc, pa.data());
        for (int64_t jr = 0; jr < nc; jr += NR)
            for (int64_t ir = 0; ir < mc; ir += MR)
                micro_kernel(kc, pa.data() + ir * kc, pb.data() + jr * kc, C + (i0 + ir) + (j0 + jr) * ldc, ldc,
                             imin(MR, mc - ir), imin(NR, nc - jr), alpha);
    }
}

// C (m x n) += alpha op(A) op(B) with op(A) m x k and op(B) k x n; OpenMP over C tiles.
void gemm(bool ta, bool tb, int64_t m, int64_t n, int64_t k, double alpha, const double* A, int64_t lda,
          const double* B, int64_t ldb, double* C, int64_t ldc)
{
    if (m <= 0 || n <= 0 || k <= 0) return;
    const int64_t tm = (m + MC - 1) / MC, tn = (n + NC - 1) / NC;
#pragma omp parallel if (tm * tn > 1 && m * n * k > 2000000)
    {
        std::vector<double> pa, pb;
#pragma omp for collapse(2) schedule(dynamic)
        for (int64_t a = 0; a < tm; ++a)
            for (int64_t b = 0; b < tn; ++b) {
                const int64_t i0 = a * MC, j0 = b * NC;
                gemm_tile(ta, tb, imin(MC, m - i0), imin(NC, n - j0), k, alpha, A, lda, i0, B, ldb, j0, C, ldc, pa,
                          pb);
            }
    }
}

// ============================================================================ tridiagonalization

constexpr int64_t NB = 32;   // panel width

// y = A(s.., s..) x for the trailing r x r block of the lower triangle (lda), each element of
// the triangle read once; per-thread partial sums.
void symv_lower(const double* A, int64_t lda, int64_t s, int64_t r, const double* x, double* y,
                std::vector<double>& part)
{
    const int nt = r > 256 ? omp_get_max_threads() : 1;
    part.assign(static_cast<size_t>(nt) * r, 0.0);
    // column ranges of about equal triangle area
    std::vector<int64_t> cut(nt + 1, r);
    cut[0] = 0;
    const double total = 0.5 * static_cast<double>(r) * (r + 1);
    for (int t = 1; t < nt; ++t) {
        const double target = total * t / nt;   // area of columns [0, c) = c r - c (c - 1) / 2
        const double c = (r + 0.5) - sqrt((r + 0.5) * (r + 0.5) - 2.0 * target);
        cut[t] = imin(r, imax(cut[t - 1], static_cast<int64_t>(c)));
    }
#pragma omp parallel num_threads(nt) if (nt > 1)
    {
        const int t = omp_get_thread_num();
        double* yt = part.data() + static_cast<size_t>(t) * r;
        for (int64_t c = cut[t]; c < cut[t + 1]; ++c) {
            const double* col = A + (s + c) * lda + s;
            const double xc = x[c];
            double dot = 0.0;
            for (int64_t i = c + 1; i < r; ++i) {
                yt[i] += col[i] * xc;
                dot += col[i] * x[i];
            }
            yt[c] += col[c] * xc + dot;
        }
    }
    for (int64_t i = 0; i < r; ++i) {
        double acc = 0.0;
        for (int t = 0; t < nt; ++t) acc += part[static_cast<size_t>(t) * r + i];
        y[i] = acc;
    }
}

// Lower triangle of the trailing block A(s.., s..) -= V W^T + W V^T, with V, W the rows s..
// of the panel's n x nb matrices (leading dimension ldv); 128 x 128 tiles in parallel.
void syr2k_lower(double* A, int64_t lda, int64_t s, int64_t r, int64_t nb, const double* V, const double* W,
                 int64_t ldv)
{
    constexpr int64_t TB = 128;
    const int64_t nblk = (r + TB - 1) / TB;
    std::vector<std::pair<int64_t, int64_t>> tiles;
    for (int64_t bj = 0; bj < nblk; ++bj)
        for (int64_t bi = bj; bi < nblk; ++bi) tiles.emplace_back(bi, bj);
    const int64_t ntile = static_cast<int64_t>(tiles.size());
#pragma omp parallel
    {
        std::vector<double> pa, pb;
#pragma omp for schedule(dynamic)
        for (int64_t t = 0; t < ntile; ++t) {
            const int64_t i0 = tiles[t].first * TB, j0 = tiles[t].second * TB;
            const int64_t mc = imin(TB, r - i0), nc = imin(TB, r - j0);
            double* C = A + s + s * lda;
            gemm_tile(false, true, mc, nc, nb, -1.0, V + s, ldv, i0, W + s, ldv, j0, C, lda, pa, pb);
            gemm_tile(false, true, mc, nc, nb, -1.0, W + s, ldv, i0, V + s, ldv, j0, C, lda, pa, pb);
        }
    }
}

// Reduces the symmetric A (n x n, column-major, lower triangle used, overwritten) to
// tridiagonal T = Q^T A Q: d = diagonal, e = subdiagonal, reflector j (j = 0 .. n-3) is
// H_j = I - tau[j] v v^T with v = (0 .. 0, 1 at row j+1, A(j+2.., j)).
void tridiagonalize(double* A, int64_t n, std::vector<double>& d, std::vector<double>& e, std::vector<double>& tau)
{
    d.assign(n, 0.0);
    e.assign(n > 1 ? n - 1 : 0, 0.0);
    tau.assign(n, 0.0);
    std::vector<double> V(static_cast<size_t>(n) * NB), W(static_cast<size_t>(n) * NB);
    std::vector<double> vw(NB), ww(NB), part, y(n);
    const int64_t lda = n;
    for (int64_t j0 = 0; j0 < n - 1; j0 += NB) {
        const int64_t nb = imin(NB, n - 1 - j0);
        std::fill(V.begin(), V.end(), 0.0);
        std::fill(W.begin(), W.end(), 0.0);
        for (int64_t i = 0; i < nb; ++i) {
            const int64_t j = j0 + i;
            double* col = A + j * lda;
            // column j of the panel, rows j.., brought up to date with the panel's columns
            // before it: A(j.., j) -= V(j.., 0..i) W(j, 0..i)^T + W(j.., 0..i) V(j, 0..i)^T
            for (int64_t t = 0; t < i; ++t) {
                const double wj = W[j + t * n], vj = V[j + t * n];
                const double* vt = &V[t * n];
                const double* wt = &W[t * n];
                for (int64_t r = j; r < n; ++r) col[r] -= vt[r] * wj + wt[r] * vj;
            }
            d[j] = col[j];
            // reflector zeroing rows j+2.. of the column
            const int64_t m = n - j - 1;   // length of x = A(j+1.., j)
            const double alpha = col[j + 1];
            double xn2 = 0.0;
            for (int64_t r = j + 2; r < n; ++r) xn2 += col[r] * col[r];
            double tj = 0.0, beta = alpha;
            if (xn2 > 0.0) {
                beta = -(alpha >= 0.0 ? 1.0 : -1.0) * sqrt(alpha * alpha + xn2);
                tj = (beta - alpha) / beta;
                const double scale = 1.0 / (alpha - beta);
                for (int64_t r = j + 2; r < n; ++r) col[r] *= scale;
            }
            e[j] = beta;
            tau[j] = tj;
            double* v = &V[i * n];
            v[j + 1] = 1.0;
            for (int64_t r = j + 2; r < n; ++r) v[r] = col[r];
            if (tj == 0.0 || m == 0) continue;
            // w = tau (A_trailing v - W (V^T v) - V (W^T v)); w -= (tau / 2) (w^T v) v
            symv_lower(A, lda, j + 1, m, v + j + 1, y.data(), part);
            for (int64_t t = 0; t < i; ++t) {
                double sv = 0.0, sw = 0.0;
                const double* vt = &V[t * n];
                const double* wt = &W[t * n];
                for (int64_t r = j + 1; r < n; ++r) {
                    sv += vt[r] * v[r];
                    sw += wt[r] * v[r];
                }
                vw[t] = sv;
                ww[t] = sw;
            }
            double* w = &W[i * n];
            for (int64_t r = j + 1; r < n; ++r) {
                double acc = y[r - j - 1];
                for (int64_t t = 0; t < i; ++t) acc -= W[r + t * n] * vw[t] + V[r + t * n] * ww[t];
                w[r] = tj * acc;
            }
            double wv = 0.0;
            for (int64_t r = j + 1; r < n; ++r) wv += w[r] * v[r];
            const double a2 = -0.5 * tj * wv;
            for (int64_t r = j + 1; r < n; ++r) w[r] += a2 * v[r];
        }
        // trailing matrix (rows and columns j0 + nb ..) -= V W^T + W V^T
        const int64_t s = j0 + nb;
        if (s < n) syr2k_lower(A, lda, s, n - s, nb, V.data(), W.data(), n);
    }
    d[n - 1] = A[(n - 1) + (n - 1) * lda];
}

// Y (n x ncols, ldy) <- Q Y = H_0 H_1 ... H_{n-3} Y, NB reflectors at a time in compact WY
// form (I - Vp Tp Vp^T), the last panel first.
void apply_q(const double* A, int64_t n, const std::vector<double>& tau, double* Y, int64_t ldy, int64_t ncols)
{
    if (n < 3 || ncols == 0) return;
    const int64_t nref = n - 2;
    std::vector<double> Vp, T(NB * NB), Wt, Tw;
    for (int64_t j0 = ((nref - 1) / NB) * NB; j0 >= 0; j0 -= NB) {
        const int64_t nb = imin(NB, nref - j0);
        const int64_t r0 = j0 + 1, rows = n - r0;   // the panel's reflectors touch rows r0..
        Vp.assign(static_cast<size_t>(rows) * nb, 0.0);
        for (int64_t i = 0; i < nb; ++i) {
            const int64_t j = j0 + i;
            double* v = &Vp[i * rows];
            v[j + 1 - r0] = 1.0;
            for (int64_t r = j + 2; r < n; ++r) v[r - r0] = A[r + j * n];
        }
        // T upper triangular: T(i, i) = tau_i, T(0..i, i) = -tau_i T(0..i, 0..i) (Vp^T v_i)
        std::fill(T.begin(), T.end(), 0.0);
        for (int64_t i = 0; i < nb; ++i) {
            const double ti = tau[j0 + i];
            const double* vi = &Vp[i * rows];
            std::vector<double> g(i, 0.0);
            for (int64_t t = 0; t < i; ++t) {
                const double* vt = &Vp[t * rows];
                double acc = 0.0;
                for (int64_t r = 0; r < rows; ++r) acc += vt[r] * vi[r];
                g[t] = acc;
            }
            for (int64_t t = 0; t < i; ++t) {
                double acc = 0.0;
                for (int64_t u = t; u < i; ++u) acc += T[t + u * NB] * g[u];
                T[t + i * NB] = -ti * acc;
            }
            T[i + i * NB] = ti;
        }
        // Wt = Vp^T Y(r0.., :), Tw = T Wt, Y(r0.., :) -= Vp Tw
        Wt.assign(static_cast<size_t>(nb) * ncols, 0.0);
        gemm(true, false, nb, ncols, rows, 1.0, Vp.data(), rows, Y + r0, ldy, Wt.data(), nb);
        Tw.assign(static_cast<size_t>(nb) * ncols, 0.0);
#pragma omp parallel for schedule(static) if (ncols > 64)
        for (int64_t c = 0; c < ncols; ++c)
            for (int64_t i = 0; i < nb; ++i) {
                double acc = 0.0;
                for (int64_t u = i; u < nb; ++u) acc += T[i + u * NB] * Wt[u + c * nb];
                Tw[i + c * nb] = acc;
            }
        gemm(false, false, rows, ncols, nb, -1.0, Vp.data(), rows, Tw.data(), nb, Y + r0, ldy);
    }
}

// ============================================================================ tridiagonal eigenproblem

// Implicit symmetric QR with Wilkinson shifts on (d, e) of order n; the rotations are applied
// to the columns of Z (n x n, ldz, identity on entry). Eigenvalues left in d, unsorted.
bool tridiagonal_qr(int64_t n, double* d, double* e, double* Z, int64_t ldz)
{
    int64_t m = n - 1;
    int64_t iters = 0;
    const int64_t max_iters = 60 * imax(n, 1);
    while (m > 0) {
        for (int64_t i = 0; i < m; ++i)
            if (fabs(e[i]) <= EPS * (fabs(d[i]) + fabs(d[i + 1]))) e[i] = 0.0;
        if (e[m - 1] == 0.0) {
            --m;
            continue;
        }
        int64_t l = m - 1;
        while (l > 0 && e[l - 1] != 0.0) --l;
        if (++iters > max_iters) return false;
        const double dd = 0.5 * (d[m - 1] - d[m]);
        const double em = e[m - 1];
        const double mu = d[m] - em * em / (dd + (dd >= 0.0 ? 1.0 : -1.0) * hypot(dd, em));
        double x = d[l] - mu, z = e[l];
        for (int64_t k = l; k < m; ++k) {
            const double r = hypot(x, z);
            double c = 1.0, s = 0.0;
            if (r != 0.0) {
                c = x / r;
                s = -z / r;
            }
            if (k > l) e[k - 1] = r;
            const double p = d[k], q = d[k + 1], f = e[k];
            d[k] = c * c * p - 2.0 * c * s * f + s * s * q;
            d[k + 1] = s * s * p + 2.0 * c * s * f + c * c * q;
            e[k] = c * s * (p - q) + (c * c - s * s) * f;
            double* zk = Z + k * ldz;
            double* zk1 = Z + (k + 1) * ldz;
            for (int64_t r2 = 0; r2 < n; ++r2) {
                const double a = zk[r2], b = zk1[r2];
                zk[r2] = c * a - s * b;
                zk1[r2] = s * a + c * b;
            }
            if (k + 1 < m) {
                x = e[k];
                z = -s * e[k + 1];
                e[k + 1] = c * e[k + 1];
            }
        }
    }
    return true;
}

// Selects the wanted eigenpairs from the ascending eigenvalues of the whole problem:
// returns indices into that list, in the order the caller wants the vectors.
using Selector = std::function<std::vector<int64_t>(const std::vector<double>&)>;

struct Join {
    int64_t off, n, m;   // block [off, off + n), first half of m rows
    double rho;          // |coupling| >= 0
    double sgn;          // sign of the coupling
};

constexpr int64_t DC_LEAF = 32;      // blocks up to this order: implicit QR
constexpr int64_t DC_SERIAL = 512;   // blocks up to this order: one thread per block

// Tears [off, off + n) recursively: records the joins of blocks above DC_SERIAL (parents
// before children) and the blocks solved serially.
void plan_tears(int64_t off, int64_t n, double* d, const double* e, std::vector<Join>& joins,
                std::vector<std::pair<int64_t, int64_t>>& serial)
{
    if (n <= DC_SERIAL) {
        serial.emplace_back(off, n);
        return;
    }
    const int64_t m = n / 2;
    const double beta = e[off + m - 1];
    Join jn{off, n, m, fabs(beta), beta >= 0.0 ? 1.0 : -1.0};
    d[off + m - 1] -= jn.rho;
    d[off + m] -= jn.rho;
    joins.push_back(jn);
    plan_tears(off, m, d, e, joins, serial);
    plan_tears(off + m, n - m, d, e, joins, serial);
}

bool join_block(int64_t n, int64_t m, double* d, double* Zb, int64_t ldz, double rho, double sgn, bool par,
                const Selector* sel, std::vector<double>* Zsel, std::vector<double>* wsel);

// Solves the tridiagonal block (d, e) of order n (serially): eigenvalues ascending in d,
// eigenvectors in Zb (n x n, ldz; zero on entry).
bool dc_serial(int64_t n, double* d, double* e, double* Zb, int64_t ldz)
{
    if (n <= DC_LEAF) {
        for (int64_t i = 0; i < n; ++i) Zb[i + i * ldz] = 1.0;
        std::vector<double> ec(e, e + (n > 1 ? n - 1 : 0));
        if (!tridiagonal_qr(n, d, ec.data(), Zb, ldz)) return false;
        // ascending order
        std::vector<int64_t> ord(n);
        std::iota(ord.begin(), ord.end(), 0);
        std::stable_sort(ord.begin(), ord.end(), [&](int64_t a, int64_t b) { return d[a] < d[b]; });
        std::vector<double> dz(d, d + n), zz(static_cast<size_t>(n) * n);
        for (int64_t c = 0; c < n; ++c)
            for (int64_t r = 0; r < n; ++r) zz[r + c * n] = Zb[r + c * ldz];
        for (int64_t c = 0; c < n; ++c) {
            d[c] = dz[ord[c]];
            for (int64_t r = 0; r < n; ++r) Zb[r + c * ldz] = zz[r + ord[c] * n];
        }
        return true;
    }
    const int64_t m = n / 2;
    const double beta = e[m - 1];
    const double rho = fabs(beta), sgn = beta >= 0.0 ? 1.0 : -1.0;
    d[m - 1] -= rho;
    d[m] -= rho;
    if (!dc_serial(m, d, e, Zb, ldz)) return false;
    if (!dc_serial(n - m, d + m, e + m, Zb + m + m * ldz, ldz)) return false;
    return join_block(n, m, d, Zb, ldz, rho, sgn, false, nullptr, nullptr, nullptr);
}

// Secular equation 1 + rho sum_j z_j^2 / (dk_j - lambda) = 0 of root i (dk ascending,
// all z_j nonzero): lambda = dk[origin] + tau with origin the nearer end of the root's
// interval, tau found by bisection (the function increases between its poles).
void secular_root(int64_t k, int64_t i, const double* dk, const double* z2, double rho, int64_t* origin, double* tau)
{
    double lo, hi;
    int64_t o;
    if (i < k - 1) {
        const double h = dk[i + 1] - dk[i];
        const double mid = 0.5 * h;
        double f = 1.0;
        for (int64_t j = 0; j < k; ++j) f += rho * z2[j] / ((dk[j] - dk[i]) - mid);
        if (f > 0.0) {
            o = i;
            lo = 0.0;
            hi = mid;
        } else {
            o = i + 1;
            lo = -mid;
            hi = 0.0;
        }
    } else {
        double zs = 0.0;
        for (int64_t j = 0; j < k; ++j) zs += z2[j];
        o = k - 1;
        lo = 0.0;
        hi = rho * zs * (1.0 + 4.0 * EPS) + EPS * fabs(dk[k - 1]);
    }
    const double d0 = dk[o];
    for (int it = 0; it < 2200; ++it) {
        const double t = 0.5 * (lo + hi);
        if (t <= lo || t >= hi) break;
        double g = 1.0;
        for (int64_t j = 0; j < k; ++j) g += rho * z2[j] / ((dk[j] - d0) - t);
        if (g > 0.0)
            hi = t;
        else
            lo = t;
    }
    *origin = o;
    *tau = 0.5 * (lo + hi);
    if (*tau == 0.0) *tau = o == i ? hi : lo;   // strictly inside the interval
}

// Joins the solved halves of a torn block: on entry Zb (n x n, ldz) = diag(Q1, Q2) holds
// the eigenvectors of the halves (eigenvalues d[0..m), d[m..n)), the block is
// diag(T1, T2) + rho u u^T with u = e_{m-1} + sgn e_m. On exit d holds the eigenvalues
// ascending and Zb the eigenvectors; or, with a selector (the last join), Zsel (n x
// count) the selected eigenvectors and wsel their eigenvalues, in the selector's order.
bool join_block(int64_t n, int64_t m, double* d, double* Zb, int64_t ldz, double rho, double sgn, bool par,
                const Selector* sel, std::vector<double>* Zsel, std::vector<double>* wsel)
{
    // z = Qhat^T u: the last row of Q1, sgn times the first row of Q2, normalized
    std::vector<double> z(n);
    for (int64_t i = 0; i < m; ++i) z[i] = Zb[(m - 1) + i * ldz];
    for (int64_t i = m; i < n; ++i) z[i] = sgn * Zb[m + i * ldz];
    double zn2 = 0.0;
    for (int64_t i = 0; i < n; ++i) zn2 += z[i] * z[i];
    const double zn = sqrt(zn2);
    for (int64_t i = 0; i < n; ++i) z[i] /= zn;
    const double r = rho * zn2;

    std::vector<int64_t> perm(n);
    std::iota(perm.begin(), perm.end(), 0);
    std::stable_sort(perm.begin(), perm.end(), [&](int64_t a, int64_t b) { return d[a] < d[b]; });
    double dmax = 0.0;
    for (int64_t i = 0; i < n; ++i) dmax = std::max(dmax, fabs(d[i]));
    const double tol = 8.0 * EPS * std::max(dmax, r);

    // deflation: negligible z entries, and close pairs of d rotated so that one z is zero
    std::vector<int> half(n);   // 1: column has rows in the first half only, 2: second, 3: both
    for (int64_t i = 0; i < n; ++i) half[i] = i < m ? 1 : 2;
    std::vector<int64_t> keep;
    std::vector<int64_t> defl;
    keep.reserve(n);
    for (int64_t t = 0; t < n; ++t) {
        const int64_t j = perm[t];
        if (r * fabs(z[j]) <= tol) {
            defl.push_back(j);
            continue;
        }
        if (!keep.empty()) {
            const int64_t p = keep.back();
            const double rr = hypot(z[p], z[j]);
            const double c = z[j] / rr, s = z[p] / rr;
            if (fabs(c * s * (d[j] - d[p])) <= tol) {
                double* cp = Zb + p * ldz;
                double* cj = Zb + j * ldz;
                for (int64_t q = 0; q < n; ++q) {
                    const double a = cp[q], b = cj[q];
                    cp[q] = c * a - s * b;
                    cj[q] = s * a + c * b;
                }
                const double dp = c * c * d[p] + s * s * d[j];
                const double dj = s * s * d[p] + c * c * d[j];
                d[p] = dp;
                d[j] = dj;
                z[p] = 0.0;
                z[j] = rr;
                half[p] |= half[j];
                half[j] |= half[p];
                keep.pop_back();
                defl.push_back(p);
            }
        }
        keep.push_back(j);
    }
    const int64_t k = static_cast<int64_t>(keep.size());
    std::vector<double> dk(k), zk(k), z2(k);
    for (int64_t i = 0; i < k; ++i) {
        dk[i] = d[keep[i]];
        zk[i] = z[keep[i]];
        z2[i] = zk[i] * zk[i];
    }
    // roots, then the recomputed z (Gu & Eisenstat) and the eigenvectors U (k x k) of D + r z z^T
    std::vector<int64_t> org(k);
    std::vector<double> tau(k), zh(k), U(static_cast<size_t>(k) * k);
#pragma omp parallel for schedule(dynamic, 16) if (par && k > 64)
    for (int64_t i = 0; i < k; ++i) secular_root(k, i, dk.data(), z2.data(), r, &org[i], &tau[i]);
    auto lam_minus_d = [&](int64_t i, int64_t j) { return (dk[org[i]] - dk[j]) + tau[i]; };
#pragma omp parallel for schedule(static) if (par && k > 64)
    for (int64_t j = 0; j < k; ++j) {
        double prod = lam_minus_d(k - 1, j) / r;
        for (int64_t i = 0; i < j; ++i) prod *= lam_minus_d(i, j) / (dk[i] - dk[j]);
        for (int64_t i = j; i < k - 1; ++i) prod *= lam_minus_d(i, j) / (dk[i + 1] - dk[j]);
        zh[j] = copysign(sqrt(fabs(prod)), zk[j]);
    }
#pragma omp parallel for schedule(static) if (par && k > 64)
    for (int64_t i = 0; i < k; ++i) {
        double* u = &U[i * k];
        double nrm = 0.0;
        for (int64_t j = 0; j < k; ++j) {
            u[j] = zh[j] / ((dk[j] - dk[org[i]]) - tau[i]);
            nrm += u[j] * u[j];
        }
        nrm = 1.0 / sqrt(nrm);
        for (int64_t j = 0; j < k; ++j) u[j] *= nrm;
    }

    // all n eigenvalues, ascending; source >= 0: root index, < 0: deflated column -1 - j
    std::vector<std::pair<double, int64_t>> all;
    all.reserve(n);
    for (int64_t i = 0; i < k; ++i) all.emplace_back(dk[org[i]] + tau[i], i);
    for (int64_t j : defl) all.emplace_back(d[j], -1 - j);
    std::stable_sort(all.begin(), all.end(),
                     [](const std::pair<double, int64_t>& a, const std::pair<double, int64_t>& b) {
                         return a.first < b.first;
                     });
    std::vector<int64_t> want;
    if (sel != nullptr) {
        std::vector<double> lam(n);
        for (int64_t i = 0; i < n; ++i) lam[i] = all[i].first;
        want = (*sel)(lam);
    } else {
        want.resize(n);
        std::iota(want.begin(), want.end(), 0);
    }
    const int64_t nw = static_cast<int64_t>(want.size());
    // destination: a fresh n x nw matrix (the join reads Zb while it writes)
    std::vector<double> out(static_cast<size_t>(n) * nw, 0.0);
    // wanted roots: out(:, c) = Zb(:, keep) U(:, i), the first-half rows from the columns
    // with first-half rows only, the second-half rows likewise
    std::vector<int64_t> wc, wr;   // output column, root index
    for (int64_t c = 0; c < nw; ++c) {
        const int64_t src = all[want[c]].second;
        if (src >= 0) {
            wc.push_back(c);
            wr.push_back(src);
        } else {
            const double* col = Zb + (-1 - src) * ldz;
            std::copy(col, col + n, out.begin() + c * n);
        }
    }
    const int64_t nr = static_cast<int64_t>(wc.size());
    if (nr > 0) {
        std::vector<double> Us;   // rows of U for the contributing columns, nr columns
        std::vector<double> Ag, R;
        for (int part = 1; part <= 2; ++part) {
            const int64_t r0 = part == 1 ? 0 : m, rows = part == 1 ? m : n - m;
            std::vector<int64_t> cols;
            for (int64_t t = 0; t < k; ++t)
                if (half[keep[t]] & part) cols.push_back(t);
            const int64_t kc = static_cast<int64_t>(cols.size());
            if (kc == 0 || rows == 0) continue;
            Ag.assign(static_cast<size_t>(rows) * kc, 0.0);
            for (int64_t c = 0; c < kc; ++c) {
                const double* col = Zb + keep[cols[c]] * ldz + r0;
                std::copy(col, col + rows, Ag.begin() + c * rows);
            }
            Us.assign(static_cast<size_t>(kc) * nr, 0.0);
            for (int64_t q = 0; q < nr; ++q)
                for (int64_t c = 0; c < kc; ++c) Us[c + q * kc] = U[cols[c] + wr[q] * k];
            R.assign(static_cast<size_t>(rows) * nr, 0.0);
            gemm(false, false, rows, nr, kc, 1.0, Ag.data(), rows, Us.data(), kc, R.data(), rows);
            for (int64_t q = 0; q < nr; ++q)
                std::copy(R.begin() + q * rows, R.begin() + (q + 1) * rows, out.begin() + wc[q] * n + r0);
        }
    }
    if (sel != nullptr) {
        wsel->resize(nw);
        for (int64_t c = 0; c < nw; ++c) (*wsel)[c] = all[want[c]].first;
        Zsel->swap(out);
    } else {
        for (int64_t c = 0; c < n; ++c) {
            d[c] = all[c].first;
            std::copy(out.begin() + c * n, out.begin() + (c + 1) * n, Zb + c * ldz);
        }
    }
    return true;
}

// Eigen-decomposition of the tridiagonal (d, e) of order n. Without a selector: d gets the
// eigenvalues ascending and Z (n x n) the eigenvectors. With one: wsel / Zsel (n x count)
// get the selected pairs in the selector's order (d and Z are then scratch).
bool tridiagonal_eigen(int64_t n, double* d, double* e, double* Z, const Selector* sel, std::vector<double>* wsel,
                       std::vector<double>* Zsel)
{
    std::fill(Z, Z + n * n, 0.0);
    std::vector<Join> joins;
    std::vector<std::pair<int64_t, int64_t>> serial;
    plan_tears(0, n, d, e, joins, serial);
    bool ok = true;
    const int64_t ns = static_cast<int64_t>(serial.size());
#pragma omp parallel for schedule(dynamic) reduction(&& : ok)
    for (int64_t b = 0; b < ns; ++b) {
        const int64_t off = serial[b].first, bn = serial[b].second;
        ok = dc_serial(bn, d + off, e + off, Z + off + off * n, n) && ok;
    }
    if (!ok) return false;
    for (int64_t q = static_cast<int64_t>(joins.size()) - 1; q >= 0; --q) {
        const Join& jn = joins[q];
        const bool last = q == 0 && sel != nullptr;
        if (!join_block(jn.n, jn.m, d + jn.off, Z + jn.off + jn.off * n, n, jn.rho, jn.sgn, true, last ? sel : nullptr,
                        last ? Zsel : nullptr, last ? wsel : nullptr))
            return false;
    }
    if (sel != nullptr && joins.empty()) {
        // one serial block: select from its full solution
        std::vector<double> lam(d, d + n);
        const std::vector<int64_t> want = (*sel)(lam);
        Zsel->assign(static_cast<size_t>(n) * want.size(), 0.0);
        wsel->resize(want.size());
        for (size_t c = 0; c < want.size(); ++c) {
            (*wsel)[c] = lam[want[c]];
            std::copy(Z + want[c] * n, Z + (want[c] + 1) * n, Zsel->begin() + c * n);
        }
    }
    return true;
}

// Sign convention: each eigenvector's largest-magnitude entry positive (lowest index on ties).
void normalize_sign(double* v, int64_t n)
{
    int64_t best = 0;
    double bestv = -1.0;
    for (int64_t i = 0; i < n; ++i) {
        const double a = fabs(v[i]);
        if (a > bestv) {
            bestv = a;
            best = i;
        }
    }
    if (v[best] < 0.0)
        for (int64_t i = 0; i < n; ++i) v[i] = -v[i];
}

}  // namespace

// Eigenvalues of the symmetric A (n x n, row-major, only read) in decreasing order into w
// (n values), and the eigenvectors that `order_sel` picks: given the eigenvalues in
// decreasing order it returns the positions (into that list) of the eigenvectors wanted,
// written as the columns of V (n x count, row-major) in the returned order, each with its
// largest-magnitude entry positive. Returns ESPACE_OK or ESPACE_ERR_NUMERIC.
int host_eigh_select(const double* A_in, int64_t n, double* w,
                     const std::function<std::vector<int64_t>(const std::vector<double>&)>& order_sel,
                     std::vector<double>& V, int threads)
{
    if (threads > 0) omp_set_num_threads(threads);
    if (n == 1) {
        w[0] = A_in[0];
        const std::vector<int64_t> want = order_sel(std::vector<double>(1, w[0]));
        V.assign(want.size(), 1.0);
        return ESPACE_OK;
    }
    // symmetric: the row-major array read as column-major is the same matrix
    std::vector<double> A(A_in, A_in + n * n);
    std::vector<double> d, e, tau;
    tridiagonalize(A.data(), n, d, e, tau);
    std::vector<double> dd = d;
    std::vector<double> ee = e;
    std::vector<double> Z(static_cast<size_t>(n) * n);
    // the selector of the tridiagonal solver sees ascending eigenvalues
    std::vector<double> desc;
    std::vector<int64_t> want_desc;
    const Selector sel = [&](const std::vector<double>& asc) {
        const int64_t m = static_cast<int64_t>(asc.size());
        desc.assign(asc.rbegin(), asc.rend());
        want_desc = order_sel(desc);
        std::vector<int64_t> want(want_desc.size());
        for (size_t c = 0; c < want.size(); ++c) want[c] = m - 1 - want_desc[c];
        return want;
    };
    std::vector<double> wsel, Zsel;
    if (!tridiagonal_eigen(n, dd.data(), ee.data(), Z.data(), &sel, &wsel, &Zsel)) return ESPACE_ERR_NUMERIC;
    for (int64_t i = 0; i < n; ++i) w[i] = desc[i];
    const int64_t cnt = static_cast<int64_t>(wsel.size());
    Z.clear();
    Z.shrink_to_fit();
    apply_q(A.data(), n, tau, Zsel.data(), n, cnt);
    V.assign(static_cast<size_t>(n) * cnt, 0.0);
#pragma omp parallel for schedule(static)
    for (int64_t c = 0; c < cnt; ++c) {
        double* v = Zsel.data() + c * n;
        normalize_sign(v, n);
        for (int64_t i = 0; i < n; ++i) V[i * cnt + c] = v[i];
    }
    return ESPACE_OK;
}

// All eigenvalues (decreasing) into w and, if V is not null, all eigenvectors as the columns
// of V (n x n, row-major), each with its largest-magnitude entry positive.
int host_eigh(const double* A_in, int64_t n, double* w, double* V, int threads)
{
    std::vector<double> Vs;
    const int64_t cnt = V != nullptr ? n : 0;
    const int rc = host_eigh_select(
        A_in, n, w,
        [cnt](const std::vector<double>&) {
            std::vector<int64_t> idx(cnt);
            std::iota(idx.begin(), idx.end(), 0);
            return idx;
        },
        Vs, threads);
    if (rc != ESPACE_OK) return rc;
    if (V != nullptr) std::copy(Vs.begin(), Vs.end(), V);
    return ESPACE_OK;
}

}  // namespace espace
