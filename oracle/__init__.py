"""CPU oracle for the WHTMix token mixer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference legs may
import this package.  The product path (the C-ABI library and its Python binding) never does.

The arithmetic lives in ``whtmix_oracle.c`` (plain C, float64 / uint32, single-threaded); this
module only compiles it with gcc and marshals numpy arrays.  See the C file's header for what is
computed and which passage of the paper (Section III-B, Eq. 1-4) each step follows.

Every function here is pinned by ``tests/test_oracle.py`` against dense Sylvester-Hadamard
products built independently (popcount definition, Sylvester recursion, scipy.linalg.hadamard),
closed forms (delta inputs, single-frequency gains, unit gains), invariants (self-inverse,
Parseval, linearity, adjointness) and finite differences.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "whtmix_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, no fast-math: IEEE float64 as written)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-std=c11", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fopenmp", "-fPIC",
                        "-shared", "-o", tmp, _SRC], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            i64, p = ctypes.c_int64, ctypes.c_void_p
            for name in ("oracle_fwht_f64", "oracle_fwht_u32"):
                getattr(lib, name).argtypes = [p, i64, i64]
                getattr(lib, name).restype = None
            lib.oracle_wht2d_f64.argtypes = [p, p, i64, i64, i64]
            for name in ("oracle_forward_f64", "oracle_forward_u32"):
                getattr(lib, name).argtypes = [p, p, p, i64, i64, i64]
            for name in ("oracle_backward_f64", "oracle_backward_u32"):
                getattr(lib, name).argtypes = [p, p, p, p, p, i64, i64, i64]
            for name in ("oracle_wht2d_f64", "oracle_forward_f64", "oracle_forward_u32",
                         "oracle_backward_f64", "oracle_backward_u32"):
                getattr(lib, name).restype = ctypes.c_int
            lib.oracle_set_threads.argtypes = [ctypes.c_int]
            lib.oracle_set_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _shape3(x: np.ndarray):
    if x.ndim == 2:
        return 1, x.shape[0], x.shape[1]
    if x.ndim != 3:
        raise ValueError("x must be [N, C] or [B, N, C]")
    return x.shape


def _check(rc: int):
    if rc != 0:
        raise ValueError(f"oracle error {rc} (N and C must be powers of two)")


def set_threads(k: int) -> int:
    """Threads for the float64 calls that follow (1, the default: single-threaded).  Only the timed
    all-core CPU baseline uses more; the results are bit-identical either way.  Returns the count
    in effect."""
    return _load().oracle_set_threads(int(k))


def fwht(v: np.ndarray) -> np.ndarray:
    """Unnormalised FWHT of a 1D vector (float64, or uint32 with wrap-around)."""
    lib = _load()
    if v.dtype == np.uint32:
        out = np.ascontiguousarray(v, dtype=np.uint32).copy()
        lib.oracle_fwht_u32(_ptr(out), out.size, 1)
    else:
        out = np.ascontiguousarray(v, dtype=np.float64).copy()
        lib.oracle_fwht_f64(_ptr(out), out.size, 1)
    return out


def wht2d(x: np.ndarray) -> np.ndarray:
    """H_N X_b H_C for each plane (float64, unnormalised)."""
    lib = _load()
    B, N, C = _shape3(x)
    xx = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty_like(xx)
    _check(lib.oracle_wht2d_f64(_ptr(xx), _ptr(out), B, N, C))
    return out


def forward(x: np.ndarray, g: np.ndarray) -> np.ndarray:
    """WHTMix forward.  float inputs -> float64 orthonormal map; int32/uint32 -> integer mode
    (unnormalised, mod 2^32) returned as int32."""
    lib = _load()
    B, N, C = _shape3(x)
    if np.issubdtype(x.dtype, np.integer):
        xx = np.ascontiguousarray(x).astype(np.uint32)
        gg = np.ascontiguousarray(g).astype(np.uint32)
        y = np.empty_like(xx)
        _check(lib.oracle_forward_u32(_ptr(xx), _ptr(gg), _ptr(y), B, N, C))
        return y.view(np.int32).reshape(x.shape)
    xx = np.ascontiguousarray(x, dtype=np.float64)
    gg = np.ascontiguousarray(g, dtype=np.float64)
    y = np.empty_like(xx)
    _check(lib.oracle_forward_f64(_ptr(xx), _ptr(gg), _ptr(y), B, N, C))
    return y.reshape(x.shape)


def backward(x: np.ndarray, g: np.ndarray, dy: np.ndarray):
    """WHTMix backward: returns (dX, dG) with dG summed over the batch in ascending order."""
    lib = _load()
    B, N, C = _shape3(x)
    if np.issubdtype(x.dtype, np.integer):
        xx = np.ascontiguousarray(x).astype(np.uint32)
        gg = np.ascontiguousarray(g).astype(np.uint32)
        dd = np.ascontiguousarray(dy).astype(np.uint32)
        dx = np.empty_like(xx)
        dg = np.empty((N, C), dtype=np.uint32)
        _check(lib.oracle_backward_u32(_ptr(xx), _ptr(gg), _ptr(dd), _ptr(dx), _ptr(dg), B, N, C))
        return dx.view(np.int32).reshape(x.shape), dg.view(np.int32)
    xx = np.ascontiguousarray(x, dtype=np.float64)
    gg = np.ascontiguousarray(g, dtype=np.float64)
    dd = np.ascontiguousarray(dy, dtype=np.float64)
    dx = np.empty_like(xx)
    dg = np.empty((N, C), dtype=np.float64)
    _check(lib.oracle_backward_f64(_ptr(xx), _ptr(gg), _ptr(dd), _ptr(dx), _ptr(dg), B, N, C))
    return dx.reshape(x.shape), dg


def separable_gains(g_t: np.ndarray, g_c: np.ndarray) -> np.ndarray:
    """G[n, c] = exp(g_t[n]) exp(g_c[c]) in float64: the per-frequency log gains of the token mix
    (Eq. 3) and of the channel mix (Eq. 2), Section III-B, combined into the one 2D gain plane they
    amount to (the two mixes act on different axes)."""
    return np.outer(np.exp(np.asarray(g_t, dtype=np.float64)), np.exp(np.asarray(g_c, dtype=np.float64)))


def forward_separable(x: np.ndarray, g_t: np.ndarray, g_c: np.ndarray) -> np.ndarray:
    """WHTMix forward with the log-domain gains (float64)."""
    return forward(np.asarray(x, dtype=np.float64), separable_gains(g_t, g_c))


def backward_separable(x: np.ndarray, g_t: np.ndarray, g_c: np.ndarray, dy: np.ndarray):
    """(dX, dg_t, dg_c) of forward_separable: dX as in backward(); by the chain rule through
    G = exp(g_t) exp(g_c)^T, dg_t[n] = sum_c dG[n, c] G[n, c] and dg_c[c] = sum_n dG[n, c] G[n, c]."""
    G = separable_gains(g_t, g_c)
    dx, dG = backward(np.asarray(x, dtype=np.float64), G, np.asarray(dy, dtype=np.float64))
    return dx, (dG * G).sum(axis=1), (dG * G).sum(axis=0)


def block_forward(x: np.ndarray, w_in: np.ndarray, g: np.ndarray, w_out: np.ndarray) -> np.ndarray:
    """The whole mixer block of Section III-B, Eq. 1-4, in float64: Z = X W_in^T per token (the input
    projection), the 2D WHT mixer of Z with gains G, then the output projection M W_out^T.  The
    weights are stored (out, in), as a linear layer's."""
    x = np.asarray(x, dtype=np.float64)
    z = x @ np.asarray(w_in, dtype=np.float64).T
    return forward(z, np.asarray(g, dtype=np.float64)) @ np.asarray(w_out, dtype=np.float64).T


def block_backward(x: np.ndarray, w_in: np.ndarray, g: np.ndarray, w_out: np.ndarray, dy: np.ndarray):
    """Gradients of the mixer block of Section III-B, Eq. 1-4, Y = mix(X W_in^T) W_out^T, in
    float64, for the loss <Y, dY>.  By the chain rule through the three linear steps (Z = X W_in^T,
    M = mix(Z), Y = M W_out^T), with token rows t over every plane:
        dM = dY W_out,   (dZ, dG) = the mixer's backward at (Z, G, dM),   dX = dZ W_in,
        dW_out = sum_t dY[t]^T M[t],   dW_in = sum_t dZ[t]^T X[t].
    Returns (dX, dW_in, dG, dW_out); the weights are (out, in) like a linear layer's."""
    x = np.asarray(x, dtype=np.float64)
    w_in = np.asarray(w_in, dtype=np.float64)
    w_out = np.asarray(w_out, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    dy = np.asarray(dy, dtype=np.float64)
    C = x.shape[-1]
    z = x @ w_in.T
    m = forward(z, g)
    dm = dy @ w_out
    dz, dg = backward(z, g, dm)
    dx = dz @ w_in
    dw_out = dy.reshape(-1, C).T @ m.reshape(-1, C)
    dw_in = dz.reshape(-1, C).T @ x.reshape(-1, C)
    return dx, dw_in, dg, dw_out
