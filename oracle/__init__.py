"""fp64 CPU oracle of ESPACE's projected linear layer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's ``cpu_baseline`` /
``--impl reference`` legs may import this package. The product library never does, and the
oracle never imports the product: the two share no code. The arithmetic lives in the plain
C file ``espace_oracle.c`` (built by ``oracle.build``); this module only marshals numpy
arrays and chains the steps in the order the paper states them:

* ``autocorr_sum``      Eq. 4, the sum of x x^T over calibration tokens (no centering);
* ``autocorr_rows``     the same for selected rows (large K);
* ``eigh``              the EVD of Sec. 3.1 by cyclic Jacobi, eigenvalues decreasing;
* ``build_projection``  Thm. 1: P = the L principal eigenvectors of C = S / n, then bf16;
* ``fold``              W' = P^T W (Sec. 2.2), bf16 (``fold_matmul``: the same with
  numpy's matrix product as the product step, for full-size layers);
* ``project``           Z = P^T X, rounded to bf16 (the rank-L intermediate of Eq. 3);
* ``contract``          Y = W'^T Z (Eq. 3), fp64;
* ``forward``           project then contract: the projected linear layer of Eq. 3;
* ``dense``             Y = W^T X (Eq. 1);
* ``reconstruct`` / ``projection_mse``  Eq. 5 and Eq. 6;
* ``autocorr_normalized_sum``           Cor. 1's input-normalized autocorrelation;
* ``go_mse_matrix`` / ``build_projection_go``  Thm. 2: C = C_X C_W + C_W C_X, P its L
  principal eigenvectors (ordered by |eigenvalue|, as the paper does when C is indefinite);
* ``forward_tp`` / ``build_projection_tp``  ESPACE applied per tensor-parallel rank
  (App. B.2, Table 2), the ranks folded onto one device (App. B.4);
* ``train_backward`` / ``dense_backward``  the training view of Sec. 2.2, Y = W^T (P P^T X)
  with P static: gradients with respect to X and W, in the order that keeps Z;
* ``nl_mse_term`` / ``order_eigenpairs``  Thm. 2's NL-MSE matrix for one calibration
  sequence (App. A.4's per-sequence form) and the eigenvalue order the paper uses when a
  calibrated C is not positive definite.

Layout: tokens are rows (``X`` is ``[N, K]``), ``W`` is ``[M, K]`` as in ``nn.Linear``,
``P`` is ``[K, L]``, ``W'`` is ``[L, M]``, ``Z`` is ``[N, L]`` and ``Y`` is ``[N, M]``.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build import build, library_path

_lib = None
_dp = ctypes.POINTER(ctypes.c_double)
_i64 = ctypes.c_int64


def _load():
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            build()
        lib = ctypes.CDLL(path)
        lib.oracle_bf16_round.restype = ctypes.c_double
        lib.oracle_bf16_round.argtypes = [ctypes.c_double]
        lib.oracle_bf16_round_array.argtypes = [_dp, _i64]
        lib.oracle_autocorr_sum.argtypes = [_dp, _i64, _i64, _dp]
        lib.oracle_autocorr_normalized_sum.argtypes = [_dp, _i64, _i64, _dp]
        lib.oracle_autocorr_rows.argtypes = [_dp, _i64, _i64, ctypes.POINTER(ctypes.c_int64), _i64, _dp]
        lib.oracle_jacobi_eigh.restype = ctypes.c_int
        lib.oracle_jacobi_eigh.argtypes = [_dp, _i64, _dp, _dp, ctypes.c_int, ctypes.c_double]
        lib.oracle_fold.argtypes = [_dp, _dp, _i64, _i64, _i64, _dp, ctypes.c_int]
        lib.oracle_project.argtypes = [_dp, _dp, _i64, _i64, _i64, _dp, ctypes.c_int]
        lib.oracle_contract.argtypes = [_dp, _dp, _i64, _i64, _i64, _dp]
        lib.oracle_dense.argtypes = [_dp, _dp, _i64, _i64, _i64, _dp]
        lib.oracle_reconstruct.argtypes = [_dp, _dp, _i64, _i64, _i64, _dp]
        lib.oracle_go_combine.argtypes = [_dp, _dp, _i64, _dp]
        lib.oracle_projection_mse.restype = ctypes.c_double
        lib.oracle_projection_mse.argtypes = [_dp, _dp, _i64, _i64, _i64]
        _lib = lib
    return _lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(_dp)


def bf16_round(a) -> np.ndarray:
    """Round every entry to the nearest bf16 value (ties to even), returned as fp64."""
    out = _f64(a).copy()
    _load().oracle_bf16_round_array(_ptr(out), out.size)
    return out


def autocorr_sum(X, S: np.ndarray | None = None) -> np.ndarray:
    """Eq. 4: ``S + sum_t x_t x_t^T`` over the token rows of ``X`` ([n, K])."""
    X = _f64(X)
    n, K = X.shape
    S = np.zeros((K, K)) if S is None else _f64(S).copy()
    _load().oracle_autocorr_sum(_ptr(X), n, K, _ptr(S))
    return S


def autocorr_rows(X, rows) -> np.ndarray:
    """Eq. 4 for the listed rows only: ``sum_t x_t[rows] x_t^T`` as ``[len(rows), K]``."""
    X = _f64(X)
    n, K = X.shape
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
    S = np.zeros((len(r), K))
    _load().oracle_autocorr_rows(_ptr(X), n, K, r.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), len(r), _ptr(S))
    return S


def autocorr_normalized_sum(X, S: np.ndarray | None = None) -> np.ndarray:
    """Cor. 1: ``S + sum_t (x_t/|x_t|)(x_t/|x_t|)^T``."""
    X = _f64(X)
    n, K = X.shape
    S = np.zeros((K, K)) if S is None else _f64(S).copy()
    _load().oracle_autocorr_normalized_sum(_ptr(X), n, K, _ptr(S))
    return S


def eigh(C, max_sweeps: int = 60, tol: float = 1e-15):
    """Symmetric EVD by cyclic Jacobi: ``(w, V, sweeps)`` with ``w`` decreasing and
    ``C = V diag(w) V^T``."""
    A = _f64(C).copy()
    K = A.shape[0]
    w = np.zeros(K)
    V = np.zeros((K, K))
    sweeps = _load().oracle_jacobi_eigh(_ptr(A), K, _ptr(w), _ptr(V), max_sweeps, tol)
    return w, V, sweeps


def normalize_signs(P: np.ndarray) -> np.ndarray:
    """Flip each column so that its entry of largest magnitude (lowest index on ties) is
    positive. Eigenvectors are defined up to sign; Y does not depend on the choice."""
    P = _f64(P).copy()
    for j in range(P.shape[1]):
        i = int(np.argmax(np.abs(P[:, j])))
        if P[i, j] < 0:
            P[:, j] = -P[:, j]
    return P


def build_projection(S, n: int, L: int):
    """Thm. 1: ``C = S / n``; ``P`` = its ``L`` principal eigenvectors (fp64, signs
    normalized) and ``P_b`` = ``P`` rounded to bf16. Returns ``(P, P_b, w, sweeps)``."""
    C = _f64(S) / float(n)
    w, V, sweeps = eigh(C)
    P = normalize_signs(V[:, :L])
    return P, bf16_round(P), w, sweeps


def fold(P, W, round_bf16: bool = True) -> np.ndarray:
    """``W' = P^T W`` as ``[L, M]`` from ``P`` ([K, L]) and ``W`` ([M, K])."""
    P, W = _f64(P), _f64(W)
    K, L = P.shape
    M = W.shape[0]
    assert W.shape[1] == K
    Wf = np.zeros((L, M))
    _load().oracle_fold(_ptr(P), _ptr(W), K, M, L, _ptr(Wf), int(round_bf16))
    return Wf


def fold_matmul(P, W, round_bf16: bool = True) -> np.ndarray:
    """``W' = P^T W`` by the same definition as ``fold``, with numpy's fp64 matrix product
    (a library primitive) as the product step: the full-size parity tests fold layers of
    up to 12288 x 24576 x 6144, where the plain loops take many minutes. Only the
    summation order differs from ``fold`` (fp64 either way); each entry is then rounded to
    bf16 by the oracle's own rounding."""
    P, W = _f64(P), _f64(W)
    assert W.shape[1] == P.shape[0]
    Wf = np.ascontiguousarray(P.T @ W.T)
    return bf16_round(Wf) if round_bf16 else Wf


def project(X, P, round_bf16: bool = True) -> np.ndarray:
    """``Z = P^T X`` stored token-major as ``[N, L]``."""
    X, P = _f64(X), _f64(P)
    N, K = X.shape
    L = P.shape[1]
    assert P.shape[0] == K
    Z = np.zeros((N, L))
    _load().oracle_project(_ptr(X), _ptr(P), N, K, L, _ptr(Z), int(round_bf16))
    return Z


def contract(Z, Wf) -> np.ndarray:
    """``Y = W'^T Z`` as ``[N, M]`` in fp64."""
    Z, Wf = _f64(Z), _f64(Wf)
    N, L = Z.shape
    M = Wf.shape[1]
    assert Wf.shape[0] == L
    Y = np.zeros((N, M))
    _load().oracle_contract(_ptr(Z), _ptr(Wf), N, L, M, _ptr(Y))
    return Y


def forward(X, P_b, W, Wf=None, round_bf16: bool = True):
    """The projected linear layer of Eq. 3: ``(Y, Z, W')``."""
    if Wf is None:
        Wf = fold(P_b, W, round_bf16)
    Z = project(X, P_b, round_bf16)
    return contract(Z, Wf), Z, Wf


def dense(X, W) -> np.ndarray:
    """Eq. 1: ``Y = W^T X`` as ``[N, M]``."""
    X, W = _f64(X), _f64(W)
    N, K = X.shape
    M = W.shape[0]
    assert W.shape[1] == K
    Y = np.zeros((N, M))
    _load().oracle_dense(_ptr(X), _ptr(W), N, K, M, _ptr(Y))
    return Y


def reconstruct(X, P) -> np.ndarray:
    """Eq. 5: ``x~ = sum_i <p_i, x> p_i`` for each token row."""
    X, P = _f64(X), _f64(P)
    N, K = X.shape
    L = P.shape[1]
    Xt = np.zeros((N, K))
    _load().oracle_reconstruct(_ptr(X), _ptr(P), N, K, L, _ptr(Xt))
    return Xt


def projection_mse(X, P) -> float:
    """Eq. 6: sample mean of ``||x - x~||^2``."""
    X, P = _f64(X), _f64(P)
    N, K = X.shape
    return float(_load().oracle_projection_mse(_ptr(X), _ptr(P), N, K, P.shape[1]))


def weight_autocorr(W) -> np.ndarray:
    """``C_W = E[w w^T] = W^T W / M`` over the M rows (weight vectors) of ``W`` ([M, K])."""
    W = _f64(W)
    return autocorr_sum(W) / W.shape[0]


def go_mse_matrix(CX, W) -> np.ndarray:
    """Thm. 2: ``C = C_X C_W + C_W C_X`` with ``C_W = W^T W / M`` (weights and activations
    taken as independent, as the paper does)."""
    CX = _f64(CX)
    K = CX.shape[0]
    CW = weight_autocorr(W)
    assert CW.shape == (K, K)
    C = np.zeros((K, K))
    _load().oracle_go_combine(_ptr(CX), _ptr(_f64(CW)), K, _ptr(C))
    return C


def build_projection_go(S, n: int, W, L: int):
    """Thm. 2 calibration: ``C = C_X C_W + C_W C_X`` from ``C_X = S / n``; eigenvalues
    ordered by magnitude (largest first; the paper sorts absolute values when C is not
    positive definite); ``P`` = the first L eigenvectors (signs normalized), ``P_b`` its
    bf16 rounding. Returns ``(P, P_b, w, sweeps)`` with ``w`` in that order."""
    C = go_mse_matrix(_f64(S) / float(n), W)
    w, V, sweeps = eigh(C)
    order = np.argsort(-np.abs(w), kind="stable")
    w, V = w[order], V[:, order]
    P = normalize_signs(V[:, :L])
    return P, bf16_round(P), w, sweeps


def forward_tp(X, P_blocks, W, kind: str, round_bf16: bool = True) -> np.ndarray:
    """ESPACE applied per tensor-parallel rank (App. B.2, Table 2), the tp ranks' outputs
    combined on one device (App. B.4). ``P_blocks`` is ``[tp, Kr, L]``: rank r's projection.

    ``kind == "column"`` (QKV, FC1): rank r holds all K inputs and the output rows
    ``W_r = W[r M/tp : (r+1) M/tp]``; its outputs are the layer of Eq. 3 with ``P_r``
    (``Kr = K``): ``Y[:, r M/tp ..] = forward(X, P_r, W_r)``.
    ``kind == "row"`` (attention projection, FC2): rank r holds the inputs
    ``X_r = X[:, r K/tp : (r+1) K/tp]`` and the matching columns of W (``Kr = K / tp``); the
    ranks' outputs are summed: ``Y = sum_r forward(X_r, P_r, W[:, r K/tp ..])``.
    Returns ``Y`` ([N, M], fp64)."""
    X, W, P_blocks = _f64(X), _f64(W), _f64(P_blocks)
    N, K = X.shape
    M = W.shape[0]
    tp = P_blocks.shape[0]
    Y = np.zeros((N, M))
    if kind == "column":
        assert M % tp == 0 and P_blocks.shape[1] == K
        Mr = M // tp
        for r in range(tp):
            Y[:, r * Mr:(r + 1) * Mr] = forward(X, P_blocks[r], W[r * Mr:(r + 1) * Mr], round_bf16=round_bf16)[0]
    elif kind == "row":
        assert K % tp == 0 and P_blocks.shape[1] == K // tp
        Kr = K // tp
        for r in range(tp):
            Y += forward(X[:, r * Kr:(r + 1) * Kr], P_blocks[r], W[:, r * Kr:(r + 1) * Kr], round_bf16=round_bf16)[0]
    else:
        raise ValueError(kind)
    return Y


def build_projection_tp(S, n: int, L: int, kind: str, tp: int):
    """Thm. 1 per tensor-parallel rank: rank r's autocorrelation is that of its own inputs,
    all of ``C = S / n`` for ``"column"`` (every rank sees all K inputs) and the r-th
    diagonal ``K/tp x K/tp`` block of C for ``"row"``. Returns ``(P, P_b, w)``: ``[tp, Kr,
    L]`` fp64 projections, their bf16 rounding, and ``[tp, Kr]`` eigenvalues (decreasing)."""
    S = _f64(S)
    K = S.shape[0]
    Kr = K if kind == "column" else K // tp
    P = np.zeros((tp, Kr, L))
    w = np.zeros((tp, Kr))
    for r in range(tp):
        Sr = S if kind == "column" else S[r * Kr:(r + 1) * Kr, r * Kr:(r + 1) * Kr]
        P[r], _, w[r], _ = build_projection(Sr, n, L)
    return P, bf16_round(P), w


def nl_mse_term(X, G, normalized: bool = False) -> np.ndarray:
    """Thm. 2, NL-MSE, in App. A.4's per-sequence form: for one calibration sequence of T
    tokens (rows of ``X``) and the loss gradients with respect to them (rows of ``G``),
    ``C_i = (X^T X G^T G + G^T G X^T X) / T^2``; C is the mean of C_i over sequences. With
    ``normalized`` the L2-normalized variant of Sec. 3.3: every row of X and of G is
    divided by its norm first (a zero row stays zero)."""
    X, G = _f64(X), _f64(G)
    T = X.shape[0]
    assert G.shape == X.shape
    if normalized:
        nx = np.linalg.norm(X, axis=1, keepdims=True)
        ng = np.linalg.norm(G, axis=1, keepdims=True)
        X = np.where(nx > 0, X / np.where(nx > 0, nx, 1.0), 0.0)
        G = np.where(ng > 0, G / np.where(ng > 0, ng, 1.0), 0.0)
    A = autocorr_sum(X)
    B = autocorr_sum(G)
    return (A @ B + B @ A) / float(T) ** 2


def order_eigenpairs(w, V, tol: float = 1e-6):
    """Eigenvalues decreasing (Sec. 3.1); when C is not positive semidefinite -- its smallest
    eigenvalue below ``-tol`` times the largest magnitude, a margin for rounding -- by
    decreasing magnitude instead, as the paper does (ties keep the decreasing order).
    ``w`` decreasing as ``eigh`` returns it; returns the reordered ``(w, V)``."""
    w, V = np.asarray(w), np.asarray(V)
    if w[-1] < -tol * np.abs(w).max():
        order = np.argsort(-np.abs(w), kind="stable")
        return w[order], V[:, order]
    return w, V


def train_backward(dY, Z, P_b, Wf, round_bf16: bool = True):
    """Backward pass of the training view (Sec. 2.2): the layer is ``Y = W^T (P P^T X)``,
    computed as ``Z = P^T X`` and ``Y = W'^T Z`` with ``W' = P^T W`` (Eq. 3's associativity),
    P static. For the output gradient ``dY`` ([N, M]), the saved ``Z`` ([N, L]), ``P_b``
    ([K, L]) and ``Wf`` = W' ([L, M]):
    ``dZ = dY W'^T`` (bf16), ``dX = dZ P^T`` (bf16) -- the input gradient passes through the
    projection P P^T -- and ``dW = (dY^T Z) P^T`` with ``dY^T Z`` rounded to bf16 (fp64 result).
    Returns ``(dX [N, K], dW [M, K])``."""
    dY, Z, P_b, Wf = _f64(dY), _f64(Z), _f64(P_b), _f64(Wf)
    rnd = bf16_round if round_bf16 else (lambda a: a)
    dZ = rnd(dY @ Wf.T)
    dX = rnd(dZ @ P_b.T)
    dWP = rnd(dY.T @ Z)
    return dX, dWP @ P_b.T


def dense_backward(dY, X, W):
    """Backward pass of Eq. 1, ``Y = W^T X`` stored as ``Y = X W^T``: ``dX = dY W`` and
    ``dW = dY^T X`` (fp64). Returns ``(dX [N, K], dW [M, K])``."""
    dY, X, W = _f64(dY), _f64(X), _f64(W)
    return dY @ W, dY.T @ X
