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
