"""ctypes front end of the float64 Gauss-sum oracle (test infrastructure only).

``gauss_oracle.c`` is compiled with the host C compiler into
``oracle/_build/libgauss_oracle.so`` on first use (or by ``build_oracle()``).
Inputs are converted to contiguous float64 arrays here; all arithmetic
happens in the C file.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gauss_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libgauss_oracle.so")

_lock = threading.Lock()
_lib = None


def oracle_library_path() -> str:
    return _LIB_PATH


def build_oracle(src: str | None = None, out: str | None = None, force: bool = False) -> str:
    """Compile the oracle C source into a shared library and return its path.

    ``src``/``out`` default to the committed oracle; tests that plant a
    mistake in a copy of the source pass their own paths.
    """
    src = src or _SRC
    out = out or _LIB_PATH
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(src)):
        return out
    cc = os.environ.get("CC", "gcc")
    tmp = out + f".tmp{os.getpid()}"
    cmd = [cc, "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def _load(path: str | None = None):
    global _lib
    if path is not None:
        lib = ctypes.CDLL(path)
        _declare(lib)
        return lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build_oracle())
            _declare(lib)
            _lib = lib
    return _lib


def _declare(lib):
    dp = ctypes.POINTER(ctypes.c_double)
    ip = ctypes.POINTER(ctypes.c_int64)
    i64 = ctypes.c_int64
    lib.gs_oracle_sum.argtypes = [dp, dp, dp, ctypes.c_double, i64, i64, i64, i64,
                                  ip, i64, dp, dp, ctypes.c_int]
    lib.gs_oracle_sum.restype = ctypes.c_int
    lib.gs_oracle_grad_q.argtypes = [dp, dp, dp, ctypes.c_double, i64, i64, i64,
                                     ip, i64, dp, dp, dp, dp, ctypes.c_int]
    lib.gs_oracle_grad_q.restype = ctypes.c_int
    lib.gs_oracle_vjp.argtypes = [dp, dp, dp, dp, ctypes.c_double, i64, i64, i64, i64,
                                  ip, i64, ip, i64, dp, dp, dp, dp, dp, dp, ctypes.c_int]
    lib.gs_oracle_vjp.restype = ctypes.c_int
    lib.gs_oracle_max_threads.argtypes = []
    lib.gs_oracle_max_threads.restype = ctypes.c_int


def _f64(a, shape):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float64)).reshape(shape)
    return a


def _ptr(a):
    if a is None:
        return None
    ctype = ctypes.c_int64 if a.dtype == np.int64 else ctypes.c_double
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _threads(nthreads):
    if nthreads is None:
        return max(1, len(os.sched_getaffinity(0)))
    return int(nthreads)


def oracle_max_threads(lib_path: str | None = None) -> int:
    return int(_load(lib_path).gs_oracle_max_threads())


def oracle_sum(q, k, v, tau, rows=None, nthreads=None, lib_path=None):
    """Eq. 1 in float64.  Returns (s, den) with s, den of shape (R, C).

    q: (M, D), k: (N, D), v: (N, C) -- any real dtype, upcast to float64.
    rows: optional sequence of row indices (default: all M rows).
    den[r, c] = sum_n Phi |v[n, c]| is the scale used for relative errors.
    """
    q = np.asarray(q)
    k = np.asarray(k)
    v = np.asarray(v)
    M, D = q.shape
    N = k.shape[0]
    if v.ndim == 1:
        v = v.reshape(N, 1)
    C = v.shape[1]
    q64 = _f64(q, (M, D))
    k64 = _f64(k, (N, D))
    v64 = _f64(v, (N, C))
    if rows is None:
        R = M
        rows_a = None
    else:
        rows_a = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
        R = rows_a.shape[0]
    s = np.empty((R, C), dtype=np.float64)
    den = np.empty((R, C), dtype=np.float64)
    rc = _load(lib_path).gs_oracle_sum(_ptr(q64), _ptr(k64), _ptr(v64), float(tau), M, N, D, C,
                                       _ptr(rows_a), R, _ptr(s), _ptr(den), _threads(nthreads))
    if rc != 0:
        raise ValueError("gs_oracle_sum rejected its arguments")
    return s, den


def oracle_grad_q(q, k, v, tau, rows=None, nthreads=None, lib_path=None):
    """Sec. 3 q-gradient in float64 for scalar weights.

    Returns (g, s, den, den_shift): g, den, den_shift of shape (R, D), s of
    shape (R,).
    """
    q = np.asarray(q)
    k = np.asarray(k)
    v = np.asarray(v).reshape(-1)
    M, D = q.shape
    N = k.shape[0]
    q64 = _f64(q, (M, D))
    k64 = _f64(k, (N, D))
    v64 = _f64(v, (N,))
    if rows is None:
        R = M
        rows_a = None
    else:
        rows_a = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
        R = rows_a.shape[0]
    g = np.empty((R, D), dtype=np.float64)
    s = np.empty((R,), dtype=np.float64)
    den = np.empty((R, D), dtype=np.float64)
    dsh = np.empty((R, D), dtype=np.float64)
    rc = _load(lib_path).gs_oracle_grad_q(_ptr(q64), _ptr(k64), _ptr(v64), float(tau), M, N, D,
                                          _ptr(rows_a), R, _ptr(g), _ptr(s), _ptr(den), _ptr(dsh),
                                          _threads(nthreads))
    if rc != 0:
        raise ValueError("gs_oracle_grad_q rejected its arguments")
    return g, s, den, dsh


def oracle_mmd2(x, v, tau, nthreads=None, lib_path=None):
    """Squared MMD of Sec. 3 (Maximum mean discrepancy) for the signed
    measure sum_n v_n delta_{x_n}: sum_m v_m s_m with s the Gauss sum of
    Eq. 1 for q = k = x and C = 1.  Returns (mmd2, den) with
    den = sum_m |v_m| sum_n Phi(x_m, x_n) |v_n|, the error scale of a
    computed s carried through the weighted sum.  x: (N, D), v: (N,)."""
    x = np.asarray(x, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64).reshape(-1)
    s, den = oracle_sum(x, x, v.reshape(-1, 1), tau, nthreads=nthreads, lib_path=lib_path)
    return float(np.dot(v, s[:, 0])), float(np.dot(np.abs(v), den[:, 0]))


def _rows(rows):
    if rows is None:
        return None
    return np.ascontiguousarray(np.asarray(rows, dtype=np.int64))


def oracle_vjp(q, k, v, g, tau, rows_q=None, rows_k=None, nthreads=None, lib_path=None):
    """Vector-Jacobian product of Eq. 1 in float64: the gradients of
    L = sum_m g_m . s_m with respect to q, k and v.

    q: (M, D), k: (N, D), v: (N, C), g: (M, C).  rows_q / rows_k select the
    rows of dL/dq and of dL/dk, dL/dv (default: all).  Returns a dict with
    gq (Rq, D), gk (Rk, D), gv (Rk, C) and their error scales dq, dk, dv of
    the same shapes (see gauss_oracle.c).
    """
    q = np.asarray(q)
    k = np.asarray(k)
    M, D = q.shape
    N = k.shape[0]
    v = np.asarray(v).reshape(N, -1)
    C = v.shape[1]
    g = np.asarray(g).reshape(M, C)
    q64, k64 = _f64(q, (M, D)), _f64(k, (N, D))
    v64, g64 = _f64(v, (N, C)), _f64(g, (M, C))
    rq, rk = _rows(rows_q), _rows(rows_k)
    Rq = M if rq is None else rq.shape[0]
    Rk = N if rk is None else rk.shape[0]
    out = {
        "gq": np.empty((Rq, D)), "dq": np.empty((Rq, D)),
        "gk": np.empty((Rk, D)), "dk": np.empty((Rk, D)),
        "gv": np.empty((Rk, C)), "dv": np.empty((Rk, C)),
    }
    rc = _load(lib_path).gs_oracle_vjp(
        _ptr(q64), _ptr(k64), _ptr(v64), _ptr(g64), float(tau), M, N, D, C,
        _ptr(rq), Rq, _ptr(rk), Rk, _ptr(out["gq"]), _ptr(out["gk"]), _ptr(out["gv"]),
        _ptr(out["dq"]), _ptr(out["dk"]), _ptr(out["dv"]), _threads(nthreads))
    if rc != 0:
        raise ValueError("gs_oracle_vjp rejected its arguments")
    return out
