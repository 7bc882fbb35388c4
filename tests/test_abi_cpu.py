"""Host-side checks of the C-ABI library that need no GPU: it loads, it exports every entry
point include/espace.h declares, and its fp64 host eigen-solver (the non-hot step of
espace_build_projection) agrees with the oracle's Jacobi solver."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "espace.h")).read()
    return sorted(set(re.findall(r"^\s*(?:int|void|const char\*)\s+(espace_\w+)\s*\(", text, re.M)))


def test_library_loads_and_exports_every_declared_symbol():
    import paper_2410_05437_gb300 as esp
    names = _declared_functions()
    assert len(names) >= 25
    lib = ctypes.CDLL(esp.LIBRARY_PATH)
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    assert sorted(esp.EXPORTED_SYMBOLS) == names
    assert esp.espace_version() == 100


def test_error_codes_without_gpu():
    import paper_2410_05437_gb300 as esp
    # shape errors are rejected before any CUDA call
    with pytest.raises(esp.EspaceError) as e:
        esp.espace_calib_create(12)
    assert e.value.code == 2
    assert esp.lib.espace_host_eigh(None, 3, None, None, 0) == 1      # ESPACE_ERR_ARG
    assert "null" in esp.lib.espace_last_error().decode()
    out = ctypes.c_void_p()
    assert esp.lib.espace_proj_from_device(512, 512, 256, None, None, None, ctypes.byref(out)) == 1
    assert out.value is None
    # tensor-parallel layers: null pointers, then shapes, are refused before any CUDA call
    P = np.zeros(4, dtype=np.float64)
    Pp = P.ctypes.data_as(ctypes.POINTER(ctypes.c_double))
    fake_w = ctypes.c_void_p(16)
    assert esp.lib.espace_proj_tp_from_host(esp.TP_ROW, 4, 1024, 512, 64, None, fake_w, None, ctypes.byref(out)) == 1
    assert esp.lib.espace_proj_tp_from_host(3, 4, 1024, 512, 64, Pp, fake_w, None, ctypes.byref(out)) == 1   # kind
    assert esp.lib.espace_proj_tp_from_host(esp.TP_ROW, 9, 1152, 512, 64, Pp, fake_w, None, ctypes.byref(out)) == 2
    assert esp.lib.espace_proj_tp_from_host(esp.TP_ROW, 3, 1008, 512, 64, Pp, fake_w, None, ctypes.byref(out)) == 2
    assert esp.lib.espace_proj_tp_from_host(esp.TP_ROW, 4, 1024, 512, 320, Pp, fake_w, None, ctypes.byref(out)) == 2
    assert esp.lib.espace_proj_tp_from_host(esp.TP_COLUMN, 4, 1024, 1000, 64, Pp, fake_w, None, ctypes.byref(out)) == 2
    assert esp.lib.espace_proj_tp_from_host(esp.TP_COLUMN, 4, 1024, 1024, 96, Pp, fake_w, None, ctypes.byref(out)) == 2
    assert out.value is None


def test_null_handles_and_pointers_are_refused_without_gpu():
    """Every entry point that takes a handle refuses a null one with ESPACE_ERR_ARG, and the
    dense entry points refuse null pointers and bad shapes, before any CUDA call."""
    import paper_2410_05437_gb300 as esp
    L = esp.lib
    x = ctypes.c_void_p(256)          # never dereferenced: the calls fail on their first check
    out = ctypes.c_void_p()
    i = ctypes.c_int()
    i64 = ctypes.c_int64()
    calls = {
        "espace_calib_accumulate": lambda: L.espace_calib_accumulate(None, x, 8, None),
        "espace_calib_accumulate_normalized": lambda: L.espace_calib_accumulate_normalized(None, x, 8, None),
        "espace_calib_accumulate_nl": lambda: L.espace_calib_accumulate_nl(None, x, x, 8, 0, None),
        "espace_calib_read": lambda: L.espace_calib_read(None, None, None, None),
        "espace_calib_export": lambda: L.espace_calib_export(None, None, None, None),
        "espace_calib_import": lambda: L.espace_calib_import(None, None, 0, None),
        "espace_calib_reset": lambda: L.espace_calib_reset(None, None),
        "espace_build_projection": lambda: L.espace_build_projection(None, x, 64, 8, None, ctypes.byref(out)),
        "espace_build_projection_go": lambda: L.espace_build_projection_go(None, x, 64, 8, None, ctypes.byref(out)),
        "espace_build_projection_tp": lambda: L.espace_build_projection_tp(None, x, 64, 64, esp.TP_ROW, 2, None,
                                                                          ctypes.byref(out)),
        "espace_proj_tp_info": lambda: L.espace_proj_tp_info(None, ctypes.byref(i), ctypes.byref(i)),
        "espace_proj_shape": lambda: L.espace_proj_shape(None, ctypes.byref(i64), ctypes.byref(i64), ctypes.byref(i64)),
        "espace_proj_eigenvalues": lambda: L.espace_proj_eigenvalues(None, None),
        "espace_proj_read_P": lambda: L.espace_proj_read_P(None, None),
        "espace_proj_read_Wfold": lambda: L.espace_proj_read_Wfold(None, None),
        "espace_proj_export": lambda: L.espace_proj_export(None, None, None, None),
        "espace_linear_forward": lambda: L.espace_linear_forward(None, x, 8, x, None),
        "espace_linear_forward_path": lambda: L.espace_linear_forward_path(None, x, 8, x, None, 0),
        "espace_linear_forward_noalloc": lambda: L.espace_linear_forward_noalloc(None, x, 8, x, None),
        "espace_linear_forward_host": lambda: L.espace_linear_forward_host(None, x, 8, x, None),
        "espace_linear_forward_host_async": lambda: L.espace_linear_forward_host_async(None, x, 8, x, None),
        "espace_linear_forward_host_many": lambda: L.espace_linear_forward_host_many(
            1, (ctypes.c_void_p * 1)(None), (ctypes.c_void_p * 1)(x), (ctypes.c_int64 * 1)(8),
            (ctypes.c_void_p * 1)(x), None),
        "espace_proj_refold": lambda: L.espace_proj_refold(None, x, None),
        "espace_train_forward": lambda: L.espace_train_forward(None, x, 8, x, x, None),
        "espace_train_backward": lambda: L.espace_train_backward(None, x, x, 8, x, None),
        "espace_train_weight_grad": lambda: L.espace_train_weight_grad(None, x, None),
        "espace_dense_forward": lambda: L.espace_dense_forward(None, 8, 64, x, 64, x, None),
        "espace_dense_backward": lambda: L.espace_dense_backward(None, 8, x, 64, x, 64, x, x, 0, None),
    }
    codes = {name: call() for name, call in calls.items()}
    assert all(c == 1 for c in codes.values()), codes
    assert out.value is None
    assert L.espace_linear_forward_launches(None, 8, 0) == -1
    assert L.espace_dense_forward(x, -1, 64, x, 64, x, None) == 2          # N < 0
    assert L.espace_dense_forward(x, 8, 12, x, 64, x, None) == 2           # K not a multiple of 8
    odd = ctypes.c_void_p(264)                                              # 8-byte aligned only
    assert L.espace_dense_forward(odd, 8, 64, x, 64, x, None) == 3          # ESPACE_ERR_ALIGN
    # several layers through one pipeline: the count and the arrays are checked first
    arr = (ctypes.c_void_p * 1)(x)
    assert L.espace_linear_forward_host_many(0, None, None, None, None, None) == 0   # nothing to do
    assert L.espace_linear_forward_host_many(-1, arr, arr, (ctypes.c_int64 * 1)(8), arr, None) == 1
    assert L.espace_linear_forward_host_many(17, arr, arr, (ctypes.c_int64 * 1)(8), arr, None) == 1
    assert L.espace_linear_forward_host_many(1, None, arr, (ctypes.c_int64 * 1)(8), arr, None) == 1


@pytest.mark.parametrize("K", [1, 2, 9, 64, 200])
def test_host_eigh_matches_oracle_jacobi(K):
    import paper_2410_05437_gb300 as esp
    r = np.random.default_rng(K)
    B = r.standard_normal((K, K))
    C = B @ B.T / K + np.diag(np.linspace(0, 2, K))
    w_o, V_o, _ = oracle.eigh(C)
    w, V = esp.espace_host_eigh(C)
    scale = max(1.0, abs(w_o).max())
    assert np.allclose(w, w_o, rtol=0, atol=1e-12 * scale)
    assert np.allclose(V.T @ V, np.eye(K), atol=1e-12)
    assert np.allclose(V @ np.diag(w) @ V.T, C, atol=1e-11 * scale)
    # same sign convention: the largest-magnitude entry of every column is positive
    idx = np.argmax(np.abs(V), axis=0)
    assert np.all(V[idx, np.arange(K)] > 0)
    V_on = oracle.normalize_signs(V_o)
    gaps = np.minimum(np.abs(np.diff(w_o, prepend=np.inf)), np.abs(np.diff(w_o, append=-np.inf)))
    sep = gaps > 1e-6 * scale
    assert np.allclose(V[:, sep], V_on[:, sep], atol=1e-8)


def test_host_eigh_degenerate_and_calibration_spectrum():
    import synth
    import paper_2410_05437_gb300 as esp
    # repeated eigenvalues: the projector onto each eigenspace is still unique
    Q = synth.haar_orthonormal(np.random.default_rng(3), 12, 12)
    lam = np.array([5, 5, 5, 3, 3, 1, 1, 1, 1, 0.5, 0, 0], dtype=float)
    C = Q @ np.diag(lam) @ Q.T
    w, V = esp.espace_host_eigh(C)
    assert np.allclose(w, lam, atol=1e-12)
    P3 = V[:, :3] @ V[:, :3].T
    assert np.allclose(P3, Q[:, :3] @ Q[:, :3].T, atol=1e-10)
    # an autocorrelation of the synthetic activations (outliers, power-law spectrum)
    model = synth.ActivationModel(96, seed=5, outliers=2)
    X = synth.bf16_to_f64(model.sample(3000))
    S = oracle.autocorr_sum(X) / 3000
    w_o, _, _ = oracle.eigh(S)
    w2 = esp.espace_host_eigh(S, vectors=False)
    assert np.allclose(w2, w_o, rtol=0, atol=1e-12 * w_o[0])


@pytest.mark.parametrize("kind", ["graded", "degenerate", "calibration"])
def test_host_eigh_divide_and_conquer_sizes(kind):
    """K = 1100: the tridiagonal problem is torn above 512 rows (parallel joins), the panel
    reduction runs its threaded matrix-vector products. Eigenvalues against LAPACK's (numpy,
    a test witness), orthogonality and the residual C V = V diag(w) of all K vectors."""
    import synth
    import paper_2410_05437_gb300 as esp
    K = 1100
    r = np.random.default_rng(11)
    if kind == "calibration":
        model = synth.ActivationModel(K, seed=9)
        X = synth.bf16_to_f64(model.sample(4 * K))
        C = X.T @ X / (4 * K)
    else:
        Q = synth.haar_orthonormal(r, K, K)
        lam = (np.arange(1, K + 1) ** -1.6 if kind == "graded"
               else np.repeat(r.standard_normal((K + 7) // 8), 8)[:K])
        C = (Q * lam) @ Q.T
        C = (C + C.T) / 2
    w, V = esp.espace_host_eigh(C)
    w_ref = np.linalg.eigvalsh(C)[::-1]
    scale = np.abs(w_ref).max()
    assert np.all(np.diff(w) <= 0)
    assert np.allclose(w, w_ref, rtol=0, atol=1e-13 * scale * 10)
    assert np.abs(V.T @ V - np.eye(K)).max() < 1e-12
    assert np.abs(C @ V - V * w).max() < 1e-12 * scale
