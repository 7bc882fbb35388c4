"""Python binding of the GB300 (sm_103a) ESPACE projected-linear library.

Argument marshalling only: every function below forwards to the C ABI of the same name in
``include/espace.h`` (loaded from ``_build/libespace.so`` with ctypes), turning torch
tensors into device pointers, streams into ``cudaStream_t`` handles and non-zero return
codes into :class:`EspaceError`. All arithmetic runs in the library's CUDA kernels (and its
host eigen-solver); there is no Python or CPU fallback, and importing this package fails if
the library has not been built (``python paper_2410_05437_gb300/build.py``).

Layouts follow the ABI: ``X`` is ``[N, K]``, ``W`` is ``[M, K]`` (``nn.Linear``), ``Y`` is
``[N, M]``, all bf16 and contiguous on the GPU.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build import LIB as LIBRARY_PATH

__all__ = [
    "EspaceError", "LIBRARY_PATH", "lib",
    "espace_version", "espace_calib_create", "espace_calib_accumulate",
    "espace_calib_accumulate_normalized", "espace_calib_read", "espace_calib_export",
    "espace_calib_import", "espace_calib_reset", "espace_calib_destroy",
    "espace_build_projection", "espace_build_projection_go", "espace_proj_from_host", "espace_proj_from_device",
    "espace_proj_shape",
    "espace_proj_eigenvalues", "espace_proj_read_P", "espace_proj_read_Wfold",
    "espace_proj_export", "espace_proj_import", "espace_proj_destroy",
    "espace_linear_forward", "espace_linear_forward_path", "espace_linear_forward_noalloc",
    "espace_dense_forward",
    "espace_check", "espace_debug_wait_timeout", "espace_debug_occupy", "espace_set_wait_limit_ns", "espace_set_phase_event",
    "espace_host_eigh",
    "PATH_AUTO", "PATH_TENSOR", "PATH_SMALL_N", "PATH_TENSOR_SPLIT", "EXPORTED_SYMBOLS",
    "TP_COLUMN", "TP_ROW", "espace_proj_tp_from_host", "espace_build_projection_tp", "espace_proj_tp_info",
    "espace_calib_accumulate_nl", "espace_proj_refold", "espace_train_forward", "espace_train_backward",
    "espace_train_weight_grad", "espace_linear_forward_host", "espace_linear_forward_host_async",
    "espace_linear_forward_host_many",
    "espace_dense_backward",
    "espace_linear_forward_launches",
]

PATH_AUTO, PATH_TENSOR, PATH_SMALL_N, PATH_TENSOR_SPLIT = 0, 1, 2, 3
TP_COLUMN, TP_ROW = 1, 2

ERROR_NAMES = {1: "ARG", 2: "SHAPE", 3: "ALIGN", 4: "CUDA", 5: "TIMEOUT", 6: "STATE",
               7: "NOMEM", 8: "NUMERIC"}


class EspaceError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"ESPACE_ERR_{ERROR_NAMES.get(code, code)}: {message}")
        self.code = code


if not os.path.exists(LIBRARY_PATH):
    raise ImportError(
        f"{LIBRARY_PATH} is missing: build the CUDA library first "
        "(python paper_2410_05437_gb300/build.py, or __graft_entry__.build())")

lib = ctypes.CDLL(LIBRARY_PATH)

_vp = ctypes.c_void_p
_i64 = ctypes.c_int64
_pi64 = ctypes.POINTER(ctypes.c_int64)
_pd = ctypes.POINTER(ctypes.c_double)
_pf = ctypes.POINTER(ctypes.c_float)
_pu16 = ctypes.POINTER(ctypes.c_uint16)

# name -> (restype, argtypes)
_SIGNATURES = {
    "espace_version": (ctypes.c_int, []),
    "espace_last_error": (ctypes.c_char_p, []),
    "espace_calib_create": (ctypes.c_int, [_i64, ctypes.POINTER(_vp)]),
    "espace_calib_accumulate": (ctypes.c_int, [_vp, _vp, _i64, _vp]),
    "espace_calib_accumulate_normalized": (ctypes.c_int, [_vp, _vp, _i64, _vp]),
    "espace_calib_accumulate_nl": (ctypes.c_int, [_vp, _vp, _vp, _i64, ctypes.c_int, _vp]),
    "espace_calib_read": (ctypes.c_int, [_vp, _pd, _pi64, _vp]),
    "espace_calib_export": (ctypes.c_int, [_vp, _pf, _pi64, _vp]),
    "espace_calib_import": (ctypes.c_int, [_vp, _pf, _i64, _vp]),
    "espace_calib_reset": (ctypes.c_int, [_vp, _vp]),
    "espace_calib_destroy": (None, [_vp]),
    "espace_build_projection": (ctypes.c_int, [_vp, _vp, _i64, _i64, _vp, ctypes.POINTER(_vp)]),
    "espace_proj_from_host": (ctypes.c_int, [_i64, _i64, _i64, _pd, _vp, _vp, ctypes.POINTER(_vp)]),
    "espace_proj_from_device": (ctypes.c_int, [_i64, _i64, _i64, _vp, _vp, _vp, ctypes.POINTER(_vp)]),
    "espace_build_projection_go": (ctypes.c_int, [_vp, _vp, _i64, _i64, _vp, ctypes.POINTER(_vp)]),
    "espace_proj_tp_from_host": (ctypes.c_int, [ctypes.c_int, ctypes.c_int, _i64, _i64, _i64, _pd, _vp, _vp,
                                                ctypes.POINTER(_vp)]),
    "espace_build_projection_tp": (ctypes.c_int, [_vp, _vp, _i64, _i64, ctypes.c_int, ctypes.c_int, _vp,
                                                  ctypes.POINTER(_vp)]),
    "espace_proj_tp_info": (ctypes.c_int, [_vp, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int)]),
    "espace_proj_shape": (ctypes.c_int, [_vp, _pi64, _pi64, _pi64]),
    "espace_proj_eigenvalues": (ctypes.c_int, [_vp, _pd]),
    "espace_proj_read_P": (ctypes.c_int, [_vp, _pu16]),
    "espace_proj_read_Wfold": (ctypes.c_int, [_vp, _pu16]),
    "espace_proj_export": (ctypes.c_int, [_vp, _pu16, _pu16, _pd]),
    "espace_proj_import": (ctypes.c_int, [_i64, _i64, _i64, _pu16, _pu16, _pd, ctypes.POINTER(_vp)]),
    "espace_proj_destroy": (None, [_vp]),
    "espace_linear_forward": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp]),
    "espace_linear_forward_path": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp, ctypes.c_int]),
    "espace_linear_forward_noalloc": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp]),
    "espace_linear_forward_host": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp]),
    "espace_linear_forward_host_async": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp]),
    "espace_linear_forward_host_many": (ctypes.c_int, [ctypes.c_int, _vp, _vp, _vp, _vp, _vp]),
    "espace_linear_forward_launches": (ctypes.c_int, [_vp, _i64, ctypes.c_int]),
    "espace_dense_forward": (ctypes.c_int, [_vp, _i64, _i64, _vp, _i64, _vp, _vp]),
    "espace_proj_refold": (ctypes.c_int, [_vp, _vp, _vp]),
    "espace_train_forward": (ctypes.c_int, [_vp, _vp, _i64, _vp, _vp, _vp]),
    "espace_train_backward": (ctypes.c_int, [_vp, _vp, _vp, _i64, _vp, _vp]),
    "espace_train_weight_grad": (ctypes.c_int, [_vp, _vp, _vp]),
    "espace_dense_backward": (ctypes.c_int, [_vp, _i64, _vp, _i64, _vp, _i64, _vp, _vp, ctypes.c_int, _vp]),
    "espace_check": (ctypes.c_int, [_vp]),
    "espace_debug_wait_timeout": (ctypes.c_int, [ctypes.c_uint64, _vp]),
    "espace_debug_occupy": (ctypes.c_int, [ctypes.c_int, ctypes.c_uint64, _vp]),
    "espace_set_wait_limit_ns": (ctypes.c_int, [ctypes.c_uint64]),
    "espace_set_phase_event": (ctypes.c_int, [_vp]),
    "espace_host_eigh": (ctypes.c_int, [_pd, _i64, _pd, _pd, ctypes.c_int]),
}
EXPORTED_SYMBOLS = tuple(_SIGNATURES)

for _name, (_res, _args) in _SIGNATURES.items():
    _fn = getattr(lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


def _check(rc: int) -> None:
    if rc != 0:
        raise EspaceError(rc, lib.espace_last_error().decode(errors="replace"))


def _stream(stream) -> int | None:
    """cudaStream_t of a torch stream (None -> torch's current stream on the current device)."""
    if isinstance(stream, int):
        return stream
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _dev_ptr(t, dtype_name: str = "bfloat16") -> int:
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch tensor")
    if not t.is_cuda:
        raise ValueError("tensor must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    if str(t.dtype) != f"torch.{dtype_name}":
        raise ValueError(f"expected {dtype_name}, got {t.dtype}")
    return t.data_ptr()


def _host_ptr(t, dtype_name: str = "bfloat16") -> int:
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch tensor")
    if t.is_cuda:
        raise ValueError("tensor must live in host memory")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    if str(t.dtype) != f"torch.{dtype_name}":
        raise ValueError(f"expected {dtype_name}, got {t.dtype}")
    return t.data_ptr()


def _np_ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


# ----------------------------------------------------------------------------- wrappers

def espace_version() -> int:
    return lib.espace_version()


def espace_set_wait_limit_ns(ns: int) -> None:
    _check(lib.espace_set_wait_limit_ns(int(ns)))


def espace_set_phase_event(event) -> None:
    """``event``: a recorded ``torch.cuda.Event`` (or a raw cudaEvent_t as int, or None)."""
    if event is not None and not isinstance(event, int):
        event = event.cuda_event
    _check(lib.espace_set_phase_event(event))


def espace_check(stream=None) -> None:
    _check(lib.espace_check(_stream(stream)))


def espace_debug_wait_timeout(limit_ns: int, stream=None) -> None:
    _check(lib.espace_debug_wait_timeout(int(limit_ns), _stream(stream)))


def espace_debug_occupy(ctas: int, hold_ns: int, stream=None) -> None:
    _check(lib.espace_debug_occupy(int(ctas), int(hold_ns), _stream(stream)))


def espace_host_eigh(A: np.ndarray, threads: int = 0, vectors: bool = True):
    A = np.ascontiguousarray(A, dtype=np.float64)
    K = A.shape[0]
    w = np.zeros(K)
    V = np.zeros((K, K)) if vectors else None
    _check(lib.espace_host_eigh(_np_ptr(A, ctypes.c_double), K, _np_ptr(w, ctypes.c_double),
                                _np_ptr(V, ctypes.c_double) if vectors else None, int(threads)))
    return (w, V) if vectors else w


def espace_calib_create(K: int) -> int:
    h = _vp()
    _check(lib.espace_calib_create(int(K), ctypes.byref(h)))
    return h.value


def espace_calib_accumulate(h: int, X, N: int | None = None, stream=None) -> None:
    N = X.shape[0] if N is None else N
    _check(lib.espace_calib_accumulate(h, _dev_ptr(X), int(N), _stream(stream)))


def espace_calib_accumulate_normalized(h: int, X, N: int | None = None, stream=None) -> None:
    N = X.shape[0] if N is None else N
    _check(lib.espace_calib_accumulate_normalized(h, _dev_ptr(X), int(N), _stream(stream)))


def espace_calib_accumulate_nl(h: int, X, G, normalized: bool = False, stream=None) -> None:
    """One NL-MSE calibration sequence: X, G device bf16 [T][K] (activations and the loss
    gradients with respect to them)."""
    assert tuple(X.shape) == tuple(G.shape)
    _check(lib.espace_calib_accumulate_nl(h, _dev_ptr(X), _dev_ptr(G), int(X.shape[0]), int(bool(normalized)),
                                          _stream(stream)))


def espace_calib_read(h: int, K: int, stream=None):
    """Returns ``(C, n)``: C = S / n as a fp64 ``[K, K]`` numpy array."""
    C = np.zeros((K, K))
    n = ctypes.c_int64()
    _check(lib.espace_calib_read(h, _np_ptr(C, ctypes.c_double), ctypes.byref(n), _stream(stream)))
    return C, n.value


def espace_calib_export(h: int, K: int, stream=None):
    S = np.zeros((K, K), dtype=np.float32)
    n = ctypes.c_int64()
    _check(lib.espace_calib_export(h, _np_ptr(S, ctypes.c_float), ctypes.byref(n), _stream(stream)))
    return S, n.value


def espace_calib_import(h: int, S: np.ndarray, n: int, stream=None) -> None:
    S = np.ascontiguousarray(S, dtype=np.float32)
    _check(lib.espace_calib_import(h, _np_ptr(S, ctypes.c_float), int(n), _stream(stream)))


def espace_calib_reset(h: int, stream=None) -> None:
    _check(lib.espace_calib_reset(h, _stream(stream)))


def espace_calib_destroy(h: int) -> None:
    lib.espace_calib_destroy(h)


def espace_build_projection(h: int, W, L: int, stream=None) -> int:
    p = _vp()
    _check(lib.espace_build_projection(h, _dev_ptr(W), int(W.shape[0]), int(L), _stream(stream),
                                       ctypes.byref(p)))
    return p.value


def espace_build_projection_go(h: int, W, L: int, stream=None) -> int:
    p = _vp()
    _check(lib.espace_build_projection_go(h, _dev_ptr(W), int(W.shape[0]), int(L), _stream(stream),
                                          ctypes.byref(p)))
    return p.value


def espace_proj_from_host(P: np.ndarray, W, stream=None) -> int:
    P = np.ascontiguousarray(P, dtype=np.float64)
    K, L = P.shape
    p = _vp()
    _check(lib.espace_proj_from_host(K, int(W.shape[0]), L, _np_ptr(P, ctypes.c_double),
                                     _dev_ptr(W), _stream(stream), ctypes.byref(p)))
    return p.value


def espace_proj_tp_from_host(kind: int, P: np.ndarray, W, stream=None) -> int:
    """P: fp64 [tp][Kr][L], one projection per tensor-parallel rank (Kr = K for TP_COLUMN,
    K / tp for TP_ROW); W: device bf16 [M][K]."""
    P = np.ascontiguousarray(P, dtype=np.float64)
    tp, Kr, L = P.shape
    K = int(W.shape[1])
    p = _vp()
    _check(lib.espace_proj_tp_from_host(int(kind), int(tp), K, int(W.shape[0]), int(L), _np_ptr(P, ctypes.c_double),
                                        _dev_ptr(W), _stream(stream), ctypes.byref(p)))
    return p.value


def espace_build_projection_tp(h: int, W, L: int, kind: int, tp: int, stream=None) -> int:
    p = _vp()
    _check(lib.espace_build_projection_tp(h, _dev_ptr(W), int(W.shape[0]), int(L), int(kind), int(tp),
                                          _stream(stream), ctypes.byref(p)))
    return p.value


def espace_proj_tp_info(p: int):
    """(kind, tp): 0 and 1 for a plain layer."""
    kind, tp = ctypes.c_int(), ctypes.c_int()
    _check(lib.espace_proj_tp_info(p, ctypes.byref(kind), ctypes.byref(tp)))
    return kind.value, tp.value


def espace_proj_from_device(PT, W, stream=None) -> int:
    """PT: device bf16 [L][K] (P_b^T), W: device bf16 [M][K]."""
    L, K = int(PT.shape[0]), int(PT.shape[1])
    p = _vp()
    _check(lib.espace_proj_from_device(K, int(W.shape[0]), L, _dev_ptr(PT), _dev_ptr(W), _stream(stream),
                                       ctypes.byref(p)))
    return p.value


def espace_proj_shape(p: int):
    K, M, L = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(lib.espace_proj_shape(p, ctypes.byref(K), ctypes.byref(M), ctypes.byref(L)))
    return K.value, M.value, L.value


def espace_proj_eigenvalues(p: int) -> np.ndarray:
    K, _, _ = espace_proj_shape(p)
    w = np.zeros(K)
    _check(lib.espace_proj_eigenvalues(p, _np_ptr(w, ctypes.c_double)))
    return w


def espace_proj_read_P(p: int) -> np.ndarray:
    """P as raw bf16 bits, ``uint16 [K, L]``; for a tensor-parallel layer the ranks'
    projections, ``uint16 [tp, Kr, L]`` (Kr = K, or K / tp for TP_ROW)."""
    K, _, L = espace_proj_shape(p)
    kind, tp = espace_proj_tp_info(p)
    shape = (K, L) if kind == 0 else (tp, K // tp if kind == TP_ROW else K, L)
    out = np.zeros(shape, dtype=np.uint16)
    _check(lib.espace_proj_read_P(p, _np_ptr(out, ctypes.c_uint16)))
    return out


def espace_proj_read_Wfold(p: int) -> np.ndarray:
    """W' = P^T W as raw bf16 bits, ``uint16 [L, M]``."""
    _, M, L = espace_proj_shape(p)
    out = np.zeros((L, M), dtype=np.uint16)
    _check(lib.espace_proj_read_Wfold(p, _np_ptr(out, ctypes.c_uint16)))
    return out


def espace_proj_export(p: int):
    K, M, L = espace_proj_shape(p)
    Lp = (L + 63) // 64 * 64
    PT = np.zeros((Lp, K), dtype=np.uint16)
    WfT = np.zeros((M, Lp), dtype=np.uint16)
    ev = np.zeros(K)
    _check(lib.espace_proj_export(p, _np_ptr(PT, ctypes.c_uint16), _np_ptr(WfT, ctypes.c_uint16),
                                  _np_ptr(ev, ctypes.c_double)))
    return PT, WfT, ev


def espace_proj_import(K: int, M: int, L: int, PT: np.ndarray, WfT: np.ndarray, evals=None) -> int:
    PT = np.ascontiguousarray(PT, dtype=np.uint16)
    WfT = np.ascontiguousarray(WfT, dtype=np.uint16)
    ev = None if evals is None else np.ascontiguousarray(evals, dtype=np.float64)
    p = _vp()
    _check(lib.espace_proj_import(int(K), int(M), int(L), _np_ptr(PT, ctypes.c_uint16),
                                  _np_ptr(WfT, ctypes.c_uint16),
                                  None if ev is None else _np_ptr(ev, ctypes.c_double),
                                  ctypes.byref(p)))
    return p.value


def espace_proj_destroy(p: int) -> None:
    lib.espace_proj_destroy(p)


def espace_linear_forward(p: int, X, Y, N: int | None = None, stream=None) -> None:
    N = X.shape[0] if N is None else N
    _check(lib.espace_linear_forward(p, _dev_ptr(X), int(N), _dev_ptr(Y), _stream(stream)))


def espace_linear_forward_path(p: int, X, Y, path: int, N: int | None = None, stream=None) -> None:
    N = X.shape[0] if N is None else N
    _check(lib.espace_linear_forward_path(p, _dev_ptr(X), int(N), _dev_ptr(Y), _stream(stream),
                                          int(path)))


def espace_linear_forward_launches(p: int, N: int, path: int = PATH_AUTO) -> int:
    return lib.espace_linear_forward_launches(p, int(N), int(path))


def espace_linear_forward_host(p: int, X, Y, stream=None) -> None:
    """X [N][K] and Y [N][M]: host bf16 tensors (pinned for overlapped copies)."""
    _check(lib.espace_linear_forward_host(p, _host_ptr(X), int(X.shape[0]), _host_ptr(Y), _stream(stream)))


def espace_linear_forward_host_async(p: int, X, Y, stream=None) -> None:
    """As espace_linear_forward_host, returning once queued: Y is filled (and X may change)
    only when the stream has passed this point."""
    _check(lib.espace_linear_forward_host_async(p, _host_ptr(X), int(X.shape[0]), _host_ptr(Y),
                                                _stream(stream)))


def espace_linear_forward_host_many(layers, Xs, Ys, stream=None) -> None:
    """Several independent layers from host buffers in one pipeline: layers[i] maps the host
    bf16 tensor Xs[i] [N_i][K_i] into Ys[i] [N_i][M_i] (pinned for overlapped copies)."""
    n = len(layers)
    if len(Xs) != n or len(Ys) != n:
        raise ValueError("layers, Xs and Ys must have the same length")
    hs = (ctypes.c_void_p * max(n, 1))(*[int(h) for h in layers])
    xs = (ctypes.c_void_p * max(n, 1))(*[_host_ptr(x) for x in Xs])
    ys = (ctypes.c_void_p * max(n, 1))(*[_host_ptr(y) for y in Ys])
    ns = (ctypes.c_int64 * max(n, 1))(*[int(x.shape[0]) for x in Xs])
    _check(lib.espace_linear_forward_host_many(n, hs, xs, ns, ys, _stream(stream)))


def espace_linear_forward_noalloc(p: int, X, Y, N: int | None = None, stream=None) -> None:
    """Forward that allocates nothing during the call (fixed library-owned Z scratch); for
    callers that may not allocate device memory at that point. See include/espace.h."""
    N = X.shape[0] if N is None else N
    _check(lib.espace_linear_forward_noalloc(p, _dev_ptr(X), int(N), _dev_ptr(Y), _stream(stream)))


def espace_dense_forward(X, W, Y, stream=None) -> None:
    N, K = X.shape
    M = W.shape[0]
    _check(lib.espace_dense_forward(_dev_ptr(X), N, K, _dev_ptr(W), M, _dev_ptr(Y), _stream(stream)))


def espace_proj_refold(p: int, W, stream=None) -> None:
    _check(lib.espace_proj_refold(p, _dev_ptr(W), _stream(stream)))


def espace_train_forward(p: int, X, Z, Y, stream=None) -> None:
    """X [N][K], Z [N][Lp] (kept for the backward pass), Y [N][M]: device bf16."""
    _check(lib.espace_train_forward(p, _dev_ptr(X), int(X.shape[0]), _dev_ptr(Z), _dev_ptr(Y), _stream(stream)))


def espace_train_backward(p: int, dY, Z, dX, stream=None) -> None:
    """dY [N][M], Z [N][Lp], dX [N][K] device bf16; the weight gradient accumulates on the
    handle until espace_train_weight_grad."""
    _check(lib.espace_train_backward(p, _dev_ptr(dY), _dev_ptr(Z), int(dY.shape[0]), _dev_ptr(dX), _stream(stream)))


def espace_train_weight_grad(p: int, dW, stream=None) -> None:
    """dW [M][K] device fp32 (overwritten): the step's weight gradient."""
    _check(lib.espace_train_weight_grad(p, _dev_ptr(dW, "float32"), _stream(stream)))


def espace_dense_backward(dY, X, W, dX, dW, accumulate: bool = False, stream=None) -> None:
    """dY [N][M], X [N][K], W [M][K], dX [N][K] device bf16; dW [M][K] device fp32
    (overwritten, or added to with accumulate)."""
    _check(lib.espace_dense_backward(_dev_ptr(dY), int(dY.shape[0]), _dev_ptr(X), int(X.shape[1]), _dev_ptr(W),
                                     int(W.shape[0]), _dev_ptr(dX), _dev_ptr(dW, "float32"), int(bool(accumulate)),
                                     _stream(stream)))
