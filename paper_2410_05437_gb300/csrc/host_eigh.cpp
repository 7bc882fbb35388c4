// host_eigh.cpp -- fp64 symmetric eigen-decomposition on the host for
// espace_build_projection (Thm. 1 needs the principal eigenvectors of the K x K
// autocorrelation; the paper runs this step off the hot path, App. B.1).
//
// Method (Golub & Van Loan, "Matrix Computations", Sec. 8.3):
//   1. Householder tridiagonalization A = Q T Q^T, one reflector per column;
//   2. Q formed explicitly by backward accumulation of the reflectors;
//   3. implicit symmetric QR steps with the Wilkinson shift on T, chasing the bulge with
//      Givens rotations that are also applied to the columns of Q;
//   4. eigenvalues sorted decreasing, eigenvectors permuted alongside, each column's
//      largest-magnitude entry made positive (lowest index on ties).
// The O(K^3) loops run over rows (or columns) in parallel with OpenMP.
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <numeric>
#include <vector>

#include "../../include/espace.h"

namespace espace {

namespace {

struct Rot {
    int k;
    double c, s;
};

// Reduces the symmetric n x n row-major A (overwritten) to tridiagonal form: d = diagonal,
// e = superdiagonal (n-1), and Q (row-major n x n) with A_in = Q T Q^T.
void tridiagonalize(std::vector<double>& A, int64_t n, std::vector<double>& d,
                    std::vector<double>& e, std::vector<double>& Q)
{
    std::vector<std::vector<double>> us;
    std::vector<double> betas;
    us.reserve(n > 2 ? n - 2 : 0);
    std::vector<double> p(n), w(n);
    for (int64_t k = 0; k + 2 < n; ++k) {
        const int64_t m = n - k - 1;           // length of the column below the diagonal
        const int64_t o = k + 1;               // offset of the trailing block
        std::vector<double> u(m);
        double norm2 = 0.0;
        for (int64_t i = 0; i < m; ++i) {
            u[i] = A[(o + i) * n + k];
            norm2 += u[i] * u[i];
        }
        const double x0 = u[0];
        const double alpha = -(x0 >= 0.0 ? 1.0 : -1.0) * sqrt(norm2);
        double beta = 0.0;
        if (norm2 > 0.0) {
            u[0] = x0 - alpha;
            const double uu = norm2 - x0 * x0 + u[0] * u[0];
            beta = uu > 0.0 ? 2.0 / uu : 0.0;
        }
        if (beta != 0.0) {
            // p = beta * A' u
#pragma omp parallel for schedule(static)
            for (int64_t i = 0; i < m; ++i) {
                const double* row = &A[(o + i) * n + o];
                double acc = 0.0;
                for (int64_t j = 0; j < m; ++j) acc += row[j] * u[j];
                p[i] = beta * acc;
            }
            double pu = 0.0;
            for (int64_t i = 0; i < m; ++i) pu += p[i] * u[i];
            const double kk = 0.5 * beta * pu;
            for (int64_t i = 0; i < m; ++i) w[i] = p[i] - kk * u[i];
            // A' -= u w^T + w u^T
#pragma omp parallel for schedule(static)
            for (int64_t i = 0; i < m; ++i) {
                double* row = &A[(o + i) * n + o];
                const double ui = u[i], wi = w[i];
                for (int64_t j = 0; j < m; ++j) row[j] -= ui * w[j] + wi * u[j];
            }
            A[o * n + k] = alpha;
            A[k * n + o] = alpha;
            for (int64_t i = 1; i < m; ++i) {
                A[(o + i) * n + k] = 0.0;
                A[k * n + o + i] = 0.0;
            }
        }
        us.push_back(std::move(u));
        betas.push_back(beta);
    }
    d.assign(n, 0.0);
    e.assign(n > 1 ? n - 1 : 0, 0.0);
    for (int64_t i = 0; i < n; ++i) d[i] = A[i * n + i];
    for (int64_t i = 0; i + 1 < n; ++i) e[i] = A[i * n + i + 1];

    // Q = H_0 H_1 ... H_{n-3}, accumulated from the last reflector backwards
    Q.assign(static_cast<size_t>(n * n), 0.0);
    for (int64_t i = 0; i < n; ++i) Q[i * n + i] = 1.0;
    for (int64_t k = static_cast<int64_t>(us.size()) - 1; k >= 0; --k) {
        const double beta = betas[k];
        if (beta == 0.0) continue;
        const std::vector<double>& u = us[k];
        const int64_t m = n - k - 1, o = k + 1;
        // Q' <- Q' - beta u (u^T Q') on the trailing block (columns o.. of rows o..)
#pragma omp parallel
        {
            std::vector<double> t;
#pragma omp for schedule(static)
            for (int64_t jb = o; jb < n; jb += 64) {
                const int64_t je = std::min<int64_t>(jb + 64, n);
                t.assign(je - jb, 0.0);
                for (int64_t i = 0; i < m; ++i) {
                    const double ui = u[i];
                    const double* row = &Q[(o + i) * n];
                    for (int64_t j = jb; j < je; ++j) t[j - jb] += ui * row[j];
                }
                for (int64_t i = 0; i < m; ++i) {
                    const double f = beta * u[i];
                    double* row = &Q[(o + i) * n];
                    for (int64_t j = jb; j < je; ++j) row[j] -= f * t[j - jb];
                }
            }
        }
    }
}

// Applies the Givens rotations of one QR sweep (in order) to the columns of Q.
void apply_rotations(std::vector<double>& Q, int64_t n, const std::vector<Rot>& rots)
{
    if (rots.empty()) return;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < n; ++r) {
        double* row = &Q[r * n];
        for (const Rot& g : rots) {
            const double a = row[g.k], b = row[g.k + 1];
            row[g.k] = g.c * a - g.s * b;
            row[g.k + 1] = g.s * a + g.c * b;
        }
    }
}

// Implicit symmetric QR with Wilkinson shifts on (d, e); rotations accumulate into Q.
bool tridiagonal_qr(std::vector<double>& d, std::vector<double>& e, std::vector<double>& Q,
                    int64_t n)
{
    const double eps = 2.220446049250313e-16;
    int64_t m = n - 1;
    int64_t iters = 0;
    const int64_t max_iters = 60 * std::max<int64_t>(n, 1);
    std::vector<Rot> rots;
    rots.reserve(n);
    while (m > 0) {
        for (int64_t i = 0; i < m; ++i)
            if (fabs(e[i]) <= eps * (fabs(d[i]) + fabs(d[i + 1]))) e[i] = 0.0;
        if (e[m - 1] == 0.0) {
            --m;
            continue;
        }
        int64_t l = m - 1;
        while (l > 0 && e[l - 1] != 0.0) --l;
        if (++iters > max_iters) return false;
        // Wilkinson shift from the trailing 2 x 2 block
        const double dd = 0.5 * (d[m - 1] - d[m]);
        const double em = e[m - 1];
        const double mu = d[m] - em * em / (dd + (dd >= 0.0 ? 1.0 : -1.0) * hypot(dd, em));
        double x = d[l] - mu, z = e[l];
        rots.clear();
        for (int64_t k = l; k < m; ++k) {
            const double r = hypot(x, z);
            double c = 1.0, s = 0.0;
            if (r != 0.0) {
                c = x / r;
                s = -z / r;
            }
            if (k > l) e[k - 1] = r;   // the bulge is folded into the superdiagonal
            const double p = d[k], q = d[k + 1], f = e[k];
            d[k] = c * c * p - 2.0 * c * s * f + s * s * q;
            d[k + 1] = s * s * p + 2.0 * c * s * f + c * c * q;
            e[k] = c * s * (p - q) + (c * c - s * s) * f;
            rots.push_back(Rot{static_cast<int>(k), c, s});
            if (k + 1 < m) {
                x = e[k];
                z = -s * e[k + 1];
                e[k + 1] = c * e[k + 1];
            }
        }
        apply_rotations(Q, n, rots);
    }
    return true;
}

}  // namespace

int host_eigh(const double* A_in, int64_t n, double* w, double* V, int threads)
{
    if (threads > 0) omp_set_num_threads(threads);
    std::vector<double> A(A_in, A_in + n * n);
    std::vector<double> d, e, Q;
    if (n == 1) {
        w[0] = A[0];
        if (V) V[0] = 1.0;
        return ESPACE_OK;
    }
    tridiagonalize(A, n, d, e, Q);
    if (!tridiagonal_qr(d, e, Q, n)) return ESPACE_ERR_NUMERIC;
    std::vector<int64_t> order(n);
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [&](int64_t a, int64_t b) { return d[a] > d[b]; });
    for (int64_t i = 0; i < n; ++i) w[i] = d[order[i]];
    if (V) {
#pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < n; ++j) {
            const int64_t src = order[j];
            int64_t best = 0;
            double bestv = -1.0;
            for (int64_t i = 0; i < n; ++i) {
                const double a = fabs(Q[i * n + src]);
                if (a > bestv) {
                    bestv = a;
                    best = i;
                }
            }
            const double sign = Q[best * n + src] < 0.0 ? -1.0 : 1.0;
            for (int64_t i = 0; i < n; ++i) V[i * n + j] = sign * Q[i * n + src];
        }
    }
    return ESPACE_OK;
}

}  // namespace espace
