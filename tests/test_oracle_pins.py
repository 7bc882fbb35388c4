"""Pins the fp64 oracle to facts the paper and plain mathematics fix (no GPU needed).

The oracle is trusted only through these checks: closed forms, brute force on tiny inputs
(pure-Python loops), identities the paper proves (Thm. 1's MSE formula, Eq. 3's
associativity, Prop. 1's bounds, L = K being exact), and library routines (numpy's LAPACK
eigh, torch's bf16 cast) used as independent witnesses.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth


def rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- bf16 round-to-nearest-even

def _all_bf16_values():
    bits = torch.arange(0, 1 << 16, dtype=torch.int32).to(torch.int16)
    vals = bits.view(torch.bfloat16).to(torch.float64).numpy()
    pat = np.arange(1 << 16)
    ok = np.isfinite(vals) & (vals >= 0) & (pat < 0x8000)
    return vals[ok], pat[ok]


def test_bf16_round_matches_torch_on_fp32_inputs():
    r = rng(1)
    u = r.integers(0, 1 << 32, size=1_000_000, dtype=np.uint64).astype(np.uint32)
    x = u.view(np.float32)
    x = x[np.isfinite(x)]
    # exact ties: a bf16 value plus half of its spacing (representable in fp32)
    base = (r.integers(0, 1 << 16, size=20000, dtype=np.uint32) << 16).view(np.float32)
    base = base[np.isfinite(base) & (np.abs(base) < 1e38)]
    tie = (base.view(np.uint32) | np.uint32(0x8000)).view(np.float32)
    x = np.concatenate([x, tie, np.array([0.0, -0.0, 1e-40, -1e-40, 3.4e38, -3.4e38,
                                          np.inf, -np.inf], dtype=np.float32)])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = oracle.bf16_round(x.astype(np.float64))
    assert np.array_equal(got, want)


def test_bf16_round_matches_nearest_in_table_of_all_bf16_values():
    vals, pat = _all_bf16_values()
    order = np.argsort(vals, kind="stable")
    vals, pat = vals[order], pat[order]
    keep = np.concatenate([[True], np.diff(vals) > 0])     # +0 and -0 collapse
    vals, pat = vals[keep], pat[keep]
    r = rng(2)
    x = np.concatenate([
        np.exp(r.uniform(-300, 88, size=200000)),          # wide dynamic range, fp64 values
        r.uniform(0, 1e-38, size=20000),                   # subnormal range of bf16
        (vals[1:2000] + vals[:1999]) / 2.0,                # exact midpoints -> ties to even
    ])
    got = oracle.bf16_round(x)
    idx = np.clip(np.searchsorted(vals, x), 1, len(vals) - 1)
    lo, hi = vals[idx - 1], vals[idx]
    dlo, dhi = x - lo, hi - x
    pick_hi = (dhi < dlo) | ((dhi == dlo) & (pat[idx] % 2 == 0))
    want = np.where(pick_hi, hi, lo)
    assert np.array_equal(got, want)
    assert np.array_equal(oracle.bf16_round(-x), -want)


# ---------------------------------------------------------------- autocorrelation (Eq. 4)

def test_autocorr_brute_force():
    r = rng(3)
    X = r.standard_normal((7, 5))
    S = oracle.autocorr_sum(X)
    for i in range(5):
        for j in range(5):
            acc = 0.0
            for t in range(7):
                acc += X[t][i] * X[t][j]
            assert abs(S[i, j] - acc) <= 1e-14 * (1 + abs(acc))


def test_autocorr_invariants():
    r = rng(4)
    X = r.standard_normal((300, 12)) * np.linspace(0.1, 3.0, 12)
    S = oracle.autocorr_sum(X)
    assert np.array_equal(S, S.T)
    # trace(C) = mean ||x||^2
    assert math.isclose(np.trace(S) / 300, np.mean(np.sum(X * X, axis=1)), rel_tol=1e-12)
    # shard invariance: accumulating two shards equals accumulating the whole
    S2 = oracle.autocorr_sum(X[170:], oracle.autocorr_sum(X[:170]))
    assert np.allclose(S, S2, rtol=1e-13, atol=1e-12)
    # positive semi-definite
    w = np.linalg.eigvalsh(S)
    assert w.min() >= -1e-12 * w.max()


def test_autocorr_rows_are_rows_of_the_full_sum():
    r = rng(17)
    X = r.standard_normal((40, 11))
    rows = [0, 7, 3, 10]
    assert np.allclose(oracle.autocorr_rows(X, rows), oracle.autocorr_sum(X)[rows], rtol=1e-13, atol=1e-13)


def test_structured_projection_is_orthonormal():
    P = synth.structured_projection(300, 120, seed=4)
    assert np.allclose(P.T @ P, np.eye(120), atol=1e-12)


def test_normalized_autocorr_is_autocorr_of_unit_vectors():
    r = rng(5)
    X = r.standard_normal((50, 9)) * 7.0
    X[3] = 0.0                                   # a zero token contributes nothing
    U = X.copy()
    nz = np.linalg.norm(U, axis=1) > 0
    U[nz] /= np.linalg.norm(U[nz], axis=1, keepdims=True)
    Shat = oracle.autocorr_normalized_sum(X)
    assert np.allclose(Shat, oracle.autocorr_sum(U), rtol=1e-13, atol=1e-13)
    assert math.isclose(np.trace(Shat), 49.0, rel_tol=1e-13)


# ---------------------------------------------------------------- Jacobi EVD

def test_eigh_2x2_closed_form():
    a, b, c = 2.5, -1.25, 0.75
    w, V, _ = oracle.eigh(np.array([[a, b], [b, c]]))
    mid, rad = (a + c) / 2, math.hypot((a - c) / 2, b)
    assert np.allclose(w, [mid + rad, mid - rad], rtol=0, atol=1e-15)
    # first eigenvector solves (A - l1 I) v = 0
    v = V[:, 0]
    assert abs((a - w[0]) * v[0] + b * v[1]) < 1e-14


def test_eigh_diagonal_and_sorting():
    d = np.array([0.5, 3.0, -1.0, 2.0])
    w, V, sweeps = oracle.eigh(np.diag(d))
    assert sweeps == 0
    assert np.array_equal(w, np.sort(d)[::-1])
    assert np.array_equal(np.abs(V), np.abs(np.eye(4)[:, np.argsort(-d)]))


@pytest.mark.parametrize("K", [17, 64, 150])
def test_eigh_reconstruction_and_lapack(K):
    r = rng(K)
    B = r.standard_normal((K, K))
    C = B @ B.T / K + np.diag(np.linspace(0, 1, K))
    w, V, sweeps = oracle.eigh(C)
    assert sweeps < 60
    assert np.all(np.diff(w) <= 0)
    assert np.allclose(V.T @ V, np.eye(K), atol=1e-12)
    assert np.allclose(V @ np.diag(w) @ V.T, C, atol=1e-12 * np.abs(C).max())
    ref = np.linalg.eigh(C)[0][::-1]
    assert np.allclose(w, ref, rtol=0, atol=1e-12 * ref[0])
    # well-separated spectrum: eigenvectors agree with LAPACK up to sign
    wl, Vl = np.linalg.eigh(C)
    Vl = Vl[:, ::-1]
    gaps = np.minimum(np.abs(np.diff(ref, prepend=np.inf)), np.abs(np.diff(ref, append=-np.inf)))
    sep = gaps > 1e-6 * ref[0]
    dots = np.abs(np.sum(V * Vl, axis=0))
    assert np.all(dots[sep] > 1 - 1e-9)


def test_population_spectrum_power_law():
    """With unit channel scales, no outliers and n >> K, the eigenvalues of C approach the
    generator's s_i^2 = i^-1.6."""
    K, n = 16, 200000
    model = synth.ActivationModel(K, seed=11, outliers=0, lognormal_sigma=0.0)
    X = model.sample_f32(n).astype(np.float64)
    w, _, _ = oracle.eigh(oracle.autocorr_sum(X) / n)
    target = np.arange(1, K + 1) ** -1.6
    assert np.allclose(w, target, rtol=0.03)


# ---------------------------------------------------------------- Thm. 1 and Eq. 5-6

def _calib(K=24, n=4000, seed=6):
    model = synth.ActivationModel(K, seed=seed, outliers=2, lognormal_sigma=0.5)
    return model.sample_f32(n).astype(np.float64)


def test_theorem1_mse_equals_discarded_eigenvalues():
    X = _calib()
    n, K = X.shape
    for L in (1, 5, 12, 23, 24):
        P, _, w, _ = oracle.build_projection(oracle.autocorr_sum(X), n, L)
        mse = oracle.projection_mse(X, P)
        tail = float(np.sum(w[L:]))
        assert abs(mse - tail) <= 1e-10 * float(np.sum(w)) + 1e-10 * tail


def test_theorem1_top_eigenvectors_minimize_mse():
    X = _calib(seed=7)
    n, K = X.shape
    L = 6
    S = oracle.autocorr_sum(X)
    P, _, w, _ = oracle.build_projection(S, n, L)
    best = oracle.projection_mse(X, P)
    r = rng(8)
    for _ in range(100):
        Q = synth.haar_orthonormal(r, K, L)
        assert best <= oracle.projection_mse(X, Q) * (1 + 1e-12)
    _, V, _ = oracle.eigh(S / n)
    for _ in range(20):
        idx = np.sort(r.choice(K, size=L, replace=False))
        if np.array_equal(idx, np.arange(L)):
            continue
        assert best <= oracle.projection_mse(X, V[:, idx]) * (1 + 1e-12)


def test_projection_columns_orthonormal_and_signs_normalized():
    X = _calib(seed=9)
    P, P_b, _, _ = oracle.build_projection(oracle.autocorr_sum(X), X.shape[0], 10)
    assert np.allclose(P.T @ P, np.eye(10), atol=1e-12)
    for j in range(10):
        i = int(np.argmax(np.abs(P[:, j])))
        assert P[i, j] > 0
    assert np.array_equal(P_b, oracle.bf16_round(P))


def test_normalize_signs_rules():
    """Eigenvectors are fixed only up to sign: every output column is its input column or
    its negation, with the entry of largest magnitude positive and, on a tie of magnitudes,
    the lowest such index deciding; flipping input columns changes nothing and a second
    pass is the identity."""
    r = np.random.default_rng(12)
    P = r.standard_normal((7, 5))
    P[:, 3] = [0.5, -0.5, 0.1, 0.2, -0.3, 0.0, 0.25]       # tie: index 0 decides, kept
    P[:, 4] = [-0.5, 0.5, 0.1, 0.2, -0.3, 0.0, 0.25]       # tie: index 0 decides, flipped
    Q = oracle.normalize_signs(P)
    for j in range(5):
        assert np.array_equal(Q[:, j], P[:, j]) or np.array_equal(Q[:, j], -P[:, j])
        m = np.max(np.abs(Q[:, j]))
        i = int(np.flatnonzero(np.abs(Q[:, j]) == m)[0])
        assert Q[i, j] > 0
    assert np.array_equal(Q[:, 3], P[:, 3])
    assert np.array_equal(Q[:, 4], -P[:, 4])
    flips = np.array([1.0, -1.0, -1.0, 1.0, -1.0])
    assert np.array_equal(oracle.normalize_signs(P * flips), Q)
    assert np.array_equal(oracle.normalize_signs(Q), Q)


def test_weight_autocorr_brute_force_and_orthogonal_rows():
    """C_W = W^T W / M (Thm. 2): plain loops over the M weight vectors on a tiny W, and the
    closed form sqrt(M) Q with orthonormal columns, whose C_W is the identity."""
    r = np.random.default_rng(13)
    M, K = 5, 3
    W = r.standard_normal((M, K))
    E = [[sum(W[m][i] * W[m][j] for m in range(M)) / M for j in range(K)] for i in range(K)]
    assert np.allclose(oracle.weight_autocorr(W), np.array(E), rtol=0, atol=1e-14)
    Q, _ = np.linalg.qr(r.standard_normal((40, 6)))
    assert np.allclose(oracle.weight_autocorr(math.sqrt(40) * Q), np.eye(6), rtol=0, atol=1e-12)


def test_prop1_bounds_hold_per_sample():
    X = _calib(K=20, n=500, seed=10)
    P, _, _, _ = oracle.build_projection(oracle.autocorr_sum(X), X.shape[0], 7)
    Xt = oracle.reconstruct(X, P)
    assert np.all(np.sum(Xt * Xt, 1) <= np.sum(X * X, 1) * (1 + 1e-12))
    w = rng(11).standard_normal(20)
    y, yt = X @ w, Xt @ w
    bound = 2 * (w @ w) * np.sum(X * X, 1) - 2 * y * yt
    assert np.all((y - yt) ** 2 <= bound + 1e-9 * np.abs(bound).max())


# ---------------------------------------------------------------- Eq. 1 and Eq. 3

def test_fold_project_contract_dense_brute_force():
    r = rng(12)
    N, K, M, L = 4, 6, 5, 3
    X, W, P = r.standard_normal((N, K)), r.standard_normal((M, K)), r.standard_normal((K, L))
    Wf = oracle.fold(P, W, round_bf16=False)
    Z = oracle.project(X, P, round_bf16=False)
    Y = oracle.contract(Z, Wf)
    Yd = oracle.dense(X, W)
    for l in range(L):
        for m in range(M):
            assert abs(Wf[l, m] - sum(P[k][l] * W[m][k] for k in range(K))) < 1e-13
    for t in range(N):
        for l in range(L):
            assert abs(Z[t, l] - sum(X[t][k] * P[k][l] for k in range(K))) < 1e-13
        for m in range(M):
            assert abs(Y[t, m] - sum(Z[t][l] * Wf[l][m] for l in range(L))) < 1e-12
            assert abs(Yd[t, m] - sum(W[m][k] * X[t][k] for k in range(K))) < 1e-13


def test_fold_matmul_matches_the_loop_fold():
    """The matrix-product fold used at full sizes: brute force on a tiny shape, and the
    loop fold's bf16 values on a moderate one (same fp64 definition, another summation
    order: a rounding can differ only where the fp64 sums straddle a tie)."""
    r = rng(14)
    K, M, L = 6, 5, 3
    P, W = r.standard_normal((K, L)), r.standard_normal((M, K))
    Wf = oracle.fold_matmul(P, W, round_bf16=False)
    for l in range(L):
        for m in range(M):
            assert abs(Wf[l, m] - sum(P[k][l] * W[m][k] for k in range(K))) < 1e-13
    K, M, L = 384, 200, 96
    P = oracle.bf16_round(r.standard_normal((K, L)) * K ** -0.5)
    W = oracle.bf16_round(r.standard_normal((M, K)) * K ** -0.5)
    a, b = oracle.fold_matmul(P, W), oracle.fold(P, W)
    assert a.shape == (L, M)
    assert np.mean(a == b) > 0.9999
    assert np.all(np.abs(a - b) <= 2.0 ** -7 * np.abs(b))      # at most one bf16 ulp apart
    assert np.array_equal(oracle.bf16_round(a), a)


def test_eq3_associativity():
    """(P^T W)^T (P^T X) = W^T (P P^T X) for non-square shapes."""
    r = rng(13)
    N, K, M, L = 9, 14, 11, 5
    X, W = r.standard_normal((N, K)), r.standard_normal((M, K))
    P = synth.haar_orthonormal(r, K, L)
    Y, _, _ = oracle.forward(X, P, W, round_bf16=False)
    assert np.allclose(Y, oracle.dense(oracle.reconstruct(X, P), W), rtol=1e-12, atol=1e-12)


def test_full_rank_projection_is_exact():
    """L = K gives P P^T = I, so the projected layer equals the dense one."""
    X = _calib(K=16, n=40, seed=14)
    W = rng(15).standard_normal((21, 16))
    P, P_b, _, _ = oracle.build_projection(oracle.autocorr_sum(X), X.shape[0], 16)
    Y, _, _ = oracle.forward(X, P, W, round_bf16=False)
    Yd = oracle.dense(X, W)
    assert np.allclose(Y, Yd, rtol=1e-12, atol=1e-12 * np.abs(Yd).max())
    # with the bf16 projection and bf16 intermediates it still holds to bf16 accuracy
    Yb, _, _ = oracle.forward(X, P_b, W)
    assert np.linalg.norm(Yb - Yd) / np.linalg.norm(Yd) < 2e-2


def test_rounded_intermediates_are_bf16_values():
    r = rng(16)
    X, W, P = r.standard_normal((8, 32)), r.standard_normal((24, 32)), r.standard_normal((32, 16))
    Y, Z, Wf = oracle.forward(X, P, W)
    assert np.array_equal(Z, oracle.bf16_round(Z))
    assert np.array_equal(Wf, oracle.bf16_round(Wf))
    assert np.array_equal(Z, oracle.bf16_round(oracle.project(X, P, round_bf16=False)))


# ------------------------------------------------------------------------------ Thm. 2 (GO-MSE)

def test_go_matrix_equals_the_pairwise_expectation():
    """Thm. 2: E[x x^T w w^T + w w^T x x^T] over independent x (tokens) and w (weight
    vectors), written out over every (token, weight) pair with plain loops, is
    C_X C_W + C_W C_X."""
    r = np.random.default_rng(21)
    n, M, K = 5, 3, 4
    X = r.standard_normal((n, K))
    W = r.standard_normal((M, K))
    E = [[0.0] * K for _ in range(K)]
    for t in range(n):
        for m in range(M):
            x, w = X[t], W[m]
            xw = sum(x[k] * w[k] for k in range(K))
            for i in range(K):
                for j in range(K):
                    E[i][j] += x[i] * xw * w[j] + w[i] * xw * x[j]
    E = np.array(E) / (n * M)
    C = oracle.go_mse_matrix(oracle.autocorr_sum(X) / n, W)
    assert np.allclose(C, E, rtol=0, atol=1e-12)
    assert np.array_equal(C, C.T)


def test_go_bound_term_is_half_the_quadratic_form():
    """The P-dependent term of Prop. 1's GO-MSE bound, E[<w,x> <w,x~>] over all (token,
    weight) pairs, equals 1/2 sum_i p_i^T C p_i for any orthonormal P -- the identity the
    proof of Thm. 2 rests on."""
    r = np.random.default_rng(22)
    n, M, K, L = 20, 9, 6, 3
    X = r.standard_normal((n, K)) * np.linspace(2.0, 0.5, K)
    W = r.standard_normal((M, K))
    P, _ = np.linalg.qr(r.standard_normal((K, L)))
    Xt = oracle.reconstruct(X, P)
    lhs = np.mean([(W[m] @ X[t]) * (W[m] @ Xt[t]) for t in range(n) for m in range(M)])
    C = oracle.go_mse_matrix(oracle.autocorr_sum(X) / n, W)
    rhs = 0.5 * np.trace(P.T @ C @ P)
    assert abs(lhs - rhs) <= 1e-12 * max(1.0, abs(rhs))


def test_go_reduces_to_mse_for_isotropic_weights():
    """Orthogonal weight rows give C_W = I / K, so C = (2/K) C_X: GO-MSE picks Thm. 1's P
    with eigenvalues scaled by 2/K."""
    r = np.random.default_rng(23)
    n, K, L = 60, 8, 3
    X = r.standard_normal((n, K)) * np.linspace(3.0, 0.2, K)
    Q, _ = np.linalg.qr(r.standard_normal((K, K)))
    S = oracle.autocorr_sum(X)
    P_go, _, w_go, _ = oracle.build_projection_go(S, n, Q, L)
    P_mse, _, w_mse, _ = oracle.build_projection(S, n, L)
    assert np.allclose(P_go, P_mse, rtol=0, atol=1e-9)
    assert np.allclose(w_go, (2.0 / K) * w_mse, rtol=1e-10, atol=1e-14)


def test_go_eigenvalues_ordered_by_magnitude():
    """An indefinite C (this seed has a negative eigenvalue): the order is by |eigenvalue|,
    as the paper does when C is not positive definite, and C = V diag(w) V^T still holds."""
    r = np.random.default_rng(0)
    X = r.standard_normal((50, 6))
    W = r.standard_normal((7, 6))
    S = oracle.autocorr_sum(X)
    C = oracle.go_mse_matrix(S / 50, W)
    P, _, w, _ = oracle.build_projection_go(S, 50, W, 6)
    assert (w < 0).any()
    assert np.all(np.diff(np.abs(w)) <= 1e-15)
    assert np.allclose(P.T @ P, np.eye(6), atol=1e-12)
    assert np.allclose(P @ np.diag(w) @ P.T, C, atol=1e-12 * np.abs(w).max())


# ---------------------------------------------------------------- tensor-parallel ranks (App. B.2)

def test_tp_row_brute_force():
    """Row-parallel ranks, straight from the definition with pure-Python loops: rank r owns
    the inputs r Kr .. (r+1) Kr - 1, projects them with its own P_r, folds its columns of W
    with P_r, and the ranks' outputs add up."""
    r = rng(21)
    N, K, M, L, tp = 3, 6, 4, 2, 3
    Kr = K // tp
    X, W = r.standard_normal((N, K)), r.standard_normal((M, K))
    P = r.standard_normal((tp, Kr, L))
    Y = oracle.forward_tp(X, P, W, "row", round_bf16=False)
    for t in range(N):
        for m in range(M):
            ref = 0.0
            for q in range(tp):
                for l in range(L):
                    z = sum(X[t][q * Kr + k] * P[q][k][l] for k in range(Kr))
                    wf = sum(P[q][k][l] * W[m][q * Kr + k] for k in range(Kr))
                    ref += z * wf
            assert abs(Y[t, m] - ref) < 1e-12


def test_tp_column_brute_force():
    """Column-parallel ranks: rank r owns the output rows r Mr .. (r+1) Mr - 1 and projects
    all K inputs with its own P_r."""
    r = rng(22)
    N, K, M, L, tp = 3, 5, 6, 2, 3
    Mr = M // tp
    X, W = r.standard_normal((N, K)), r.standard_normal((M, K))
    P = r.standard_normal((tp, K, L))
    Y = oracle.forward_tp(X, P, W, "column", round_bf16=False)
    for t in range(N):
        for m in range(M):
            q = m // Mr
            ref = 0.0
            for l in range(L):
                z = sum(X[t][k] * P[q][k][l] for k in range(K))
                wf = sum(P[q][k][l] * W[m][k] for k in range(K))
                ref += z * wf
            assert abs(Y[t, m] - ref) < 1e-12


@pytest.mark.parametrize("kind", ["row", "column"])
def test_tp_identity_projections_reproduce_the_dense_layer(kind):
    """Full-rank identity projections (L = Kr): every rank passes its inputs through, so the
    folded layer equals Eq. 1 exactly, bf16 roundings included (they act on bf16 values)."""
    r = rng(23)
    N, K, M, tp = 7, 32, 24, 4
    X = oracle.bf16_round(r.standard_normal((N, K)))
    W = oracle.bf16_round(r.standard_normal((M, K)) / np.sqrt(K))
    Kr = K // tp if kind == "row" else K
    P = np.stack([np.eye(Kr)] * tp)
    assert np.array_equal(oracle.forward_tp(X, P, W, kind), oracle.dense(X, W))


def test_tp_column_with_one_shared_projection_is_the_plain_layer():
    r = rng(24)
    N, K, M, L, tp = 5, 16, 12, 6, 4
    X, W = r.standard_normal((N, K)), r.standard_normal((M, K))
    P = synth.haar_orthonormal(r, K, L)
    Y = oracle.forward_tp(X, np.stack([P] * tp), W, "column", round_bf16=False)
    assert np.allclose(Y, oracle.forward(X, P, W, round_bf16=False)[0], rtol=1e-13, atol=1e-13)


def test_tp_row_projections_are_optimal_per_rank():
    """Thm. 1 applied to each rank's own inputs: rank r's projection MSE on its input slice
    equals the sum of the discarded eigenvalues of C's r-th diagonal block, which no other
    L-dimensional projection of that slice beats; the column kind solves the whole C."""
    r = rng(25)
    n, K, L, tp = 400, 12, 2, 3
    Kr = K // tp
    X = r.standard_normal((n, K)) @ np.diag(np.linspace(2.0, 0.2, K)) @ synth.haar_orthonormal(r, K, K).T
    S = oracle.autocorr_sum(X)
    P, _, w = oracle.build_projection_tp(S, n, L, "row", tp)
    for q in range(tp):
        Xq = X[:, q * Kr:(q + 1) * Kr]
        mse = oracle.projection_mse(Xq, P[q])
        assert abs(mse - np.sum(w[q][L:])) < 1e-10 * np.sum(w[q])
        for trial in range(20):
            Q = synth.haar_orthonormal(r, Kr, L)
            assert oracle.projection_mse(Xq, Q) >= mse - 1e-12
        assert np.allclose(np.sort(w[q])[::-1], np.linalg.eigvalsh(S[q * Kr:(q + 1) * Kr, q * Kr:(q + 1) * Kr] / n)[::-1])
    Pc, _, wc = oracle.build_projection_tp(S, n, L, "column", tp)
    P1, _, w1, _ = oracle.build_projection(S, n, L)
    assert all(np.array_equal(Pc[q], P1) for q in range(tp)) and np.allclose(wc[0], w1)


# ---------------------------------------------------------------- NL-MSE (Thm. 2, App. A.4)

def test_nl_mse_term_brute_force():
    """C_i = (X^T X G^T G + G^T G X^T X) / T^2 from the definition, pure-Python loops."""
    r = rng(31)
    T, K = 3, 4
    X, G = r.standard_normal((T, K)), r.standard_normal((T, K))
    C = oracle.nl_mse_term(X, G)
    A = [[sum(X[t][p] * X[t][q] for t in range(T)) for q in range(K)] for p in range(K)]
    B = [[sum(G[t][p] * G[t][q] for t in range(T)) for q in range(K)] for p in range(K)]
    for p in range(K):
        for q in range(K):
            ref = sum(A[p][s] * B[s][q] + B[p][s] * A[s][q] for s in range(K)) / T ** 2
            assert abs(C[p, q] - ref) < 1e-12


def test_nl_mse_single_token_quadratic_form():
    """One token (T = 1): p^T C p = 2 (x.g)(p.x)(p.g), and over an orthonormal set the sum is
    2 <g, x> <g, P P^T x>, the term App. A.4 maximizes (the NL-MSE bound of Prop. 1)."""
    r = rng(32)
    K, L = 7, 3
    x, g = r.standard_normal(K), r.standard_normal(K)
    C = oracle.nl_mse_term(x[None, :], g[None, :])
    for _ in range(5):
        p = r.standard_normal(K)
        assert abs(p @ C @ p - 2 * (x @ g) * (p @ x) * (p @ g)) < 1e-10 * (1 + abs(p @ C @ p))
    P = synth.haar_orthonormal(r, K, L)
    lhs = sum(P[:, l] @ C @ P[:, l] for l in range(L))
    assert abs(lhs - 2 * (g @ x) * (g @ (P @ (P.T @ x)))) < 1e-10


def test_nl_mse_trace_is_twice_the_cross_gram_norm():
    """tr((A B + B A) / T^2) = 2 ||G X^T||_F^2 / T^2 (token-pair dot products)."""
    r = rng(33)
    T, K = 9, 6
    X, G = r.standard_normal((T, K)), r.standard_normal((T, K))
    C = oracle.nl_mse_term(X, G)
    cross = sum((G[s] @ X[t]) ** 2 for s in range(T) for t in range(T))
    assert abs(np.trace(C) - 2 * cross / T ** 2) < 1e-10 * cross


def test_nl_mse_with_gradients_equal_to_activations_is_mse_squared():
    """G = X: C = 2 C_X^2 with C_X = X^T X / T, so its eigenvectors are Thm. 1's and its
    eigenvalues 2 lambda^2 (the order of C_X's eigenvalues is kept: all are positive)."""
    r = rng(34)
    T, K, L = 40, 6, 3
    X = r.standard_normal((T, K)) @ np.diag(np.linspace(2.0, 0.3, K))
    C = oracle.nl_mse_term(X, X)
    w, V, _ = oracle.eigh(C)
    P1, _, w1, _ = oracle.build_projection(oracle.autocorr_sum(X), T, L)
    assert np.allclose(w, 2 * w1 ** 2, rtol=1e-10)
    assert np.allclose(V[:, :L] @ V[:, :L].T, P1 @ P1.T, atol=1e-9)


def test_nl_mse_normalized_is_scale_invariant_per_row():
    r = rng(35)
    T, K = 8, 5
    X, G = r.standard_normal((T, K)), r.standard_normal((T, K))
    sx, sg = np.exp(r.standard_normal((T, 1))), np.exp(r.standard_normal((T, 1)))
    C = oracle.nl_mse_term(X, G, normalized=True)
    assert np.allclose(oracle.nl_mse_term(X * sx, G * sg, normalized=True), C, atol=1e-12)
    Xz = X.copy()
    Xz[2] = 0.0
    Cz = oracle.nl_mse_term(Xz, G, normalized=True)
    Xd = np.delete(X, 2, axis=0)
    Xd = Xd / np.linalg.norm(Xd, axis=1, keepdims=True)
    Gn = G / np.linalg.norm(G, axis=1, keepdims=True)
    A = Xd.T @ Xd
    B = Gn.T @ Gn
    assert np.allclose(Cz, (A @ B + B @ A) / T ** 2, atol=1e-12)


def test_eigenpair_order_by_magnitude_only_when_indefinite():
    """Activations and gradients with opposite anisotropy (G's strong directions rotated
    onto X's weak ones) give an indefinite C: magnitude order, C = V diag(w) V^T kept. A
    positive semidefinite C keeps the decreasing order."""
    r = rng(36)
    X = r.standard_normal((30, 6)) @ np.diag([4, 2, 1, 0.5, 0.2, 0.1])
    G = r.standard_normal((30, 6)) @ np.diag([0.1, 0.2, 0.5, 1, 2, 4]) @ synth.haar_orthonormal(r, 6, 6).T
    C = oracle.nl_mse_term(X, G)
    w, V, _ = oracle.eigh(C)
    assert w[-1] < -1e-3 * np.abs(w).max()          # indefinite
    wo, Vo = oracle.order_eigenpairs(w, V)
    assert np.all(np.diff(np.abs(wo)) <= 1e-15 * np.abs(wo).max())
    assert np.allclose(Vo @ np.diag(wo) @ Vo.T, C, atol=1e-12 * np.abs(w).max())
    Cp = oracle.nl_mse_term(X, X)                    # positive semidefinite
    wp, Vp, _ = oracle.eigh(Cp)
    wq, Vq = oracle.order_eigenpairs(wp, Vp)
    assert np.array_equal(wq, wp) and np.array_equal(Vq, Vp)


# ---------------------------------------------------------------- training view (Sec. 2.2)

def _train_loss(X, W, P, R):
    """sum(R * Y) for Y = W^T (P P^T X), token-major: Y = X P P^T W^T."""
    return float(np.sum(R * (X @ P @ P.T @ W.T)))


def test_train_backward_matches_finite_differences():
    """Unrounded gradients of sum(R * Y) against central differences of the forward."""
    r = rng(41)
    N, K, M, L = 4, 6, 5, 3
    X, W, R = r.standard_normal((N, K)), r.standard_normal((M, K)), r.standard_normal((N, M))
    P = synth.haar_orthonormal(r, K, L)
    Z = oracle.project(X, P, round_bf16=False)
    dX, dW = oracle.train_backward(R, Z, P, oracle.fold(P, W, round_bf16=False), round_bf16=False)
    h = 1e-6
    for (i, j) in ((0, 0), (1, 3), (3, 5), (2, 2)):
        Xp, Xm = X.copy(), X.copy()
        Xp[i, j] += h
        Xm[i, j] -= h
        fd = (_train_loss(Xp, W, P, R) - _train_loss(Xm, W, P, R)) / (2 * h)
        assert abs(dX[i, j] - fd) < 1e-7 * (1 + abs(fd))
    for (m, k) in ((0, 0), (4, 5), (2, 3)):
        Wp, Wm = W.copy(), W.copy()
        Wp[m, k] += h
        Wm[m, k] -= h
        fd = (_train_loss(X, Wp, P, R) - _train_loss(X, Wm, P, R)) / (2 * h)
        assert abs(dW[m, k] - fd) < 1e-7 * (1 + abs(fd))


def test_train_backward_full_rank_is_the_dense_backward():
    """P = I (L = K): the training view is the dense layer, and so are its gradients."""
    r = rng(42)
    N, K, M = 5, 7, 6
    X, W, dY = r.standard_normal((N, K)), r.standard_normal((M, K)), r.standard_normal((N, M))
    P = np.eye(K)
    dX, dW = oracle.train_backward(dY, X, P, oracle.fold(P, W, round_bf16=False), round_bf16=False)
    dXd, dWd = oracle.dense_backward(dY, X, W)
    for t in range(N):
        for k in range(K):
            assert abs(dXd[t, k] - sum(dY[t][m] * W[m][k] for m in range(M))) < 1e-12
    for m in range(M):
        for k in range(K):
            assert abs(dWd[m, k] - sum(dY[t][m] * X[t][k] for t in range(N))) < 1e-12
    assert np.allclose(dX, dXd, atol=1e-12) and np.allclose(dW, dWd, atol=1e-12)


def test_train_input_gradient_is_the_adjoint():
    """<dY, J V> = <J^T dY, V> for the map X -> X P P^T W^T (linear in X)."""
    r = rng(43)
    N, K, M, L = 6, 9, 4, 4
    W, dY, V = r.standard_normal((M, K)), r.standard_normal((N, M)), r.standard_normal((N, K))
    P = synth.haar_orthonormal(r, K, L)
    Wf = oracle.fold(P, W, round_bf16=False)
    JV = oracle.forward(V, P, W, Wf=Wf, round_bf16=False)[0]
    dX, _ = oracle.train_backward(dY, oracle.project(V, P, round_bf16=False), P, Wf, round_bf16=False)
    assert abs(np.sum(dY * JV) - np.sum(dX * V)) < 1e-10 * (1 + abs(np.sum(dY * JV)))
