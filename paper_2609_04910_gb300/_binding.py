"""Thin ctypes binding of the C ABI in ``include/gauss_sum.h``.

Only argument marshalling happens here: torch tensors are reduced to device
pointers, sizes, a dtype code and the current CUDA stream, and every step of
the computation runs in the library's CUDA kernels.  There is no fallback:
if ``libgauss_sum.so`` has not been built, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from .build import LIB_PATH

GS_FP32, GS_FP16, GS_BF16 = 0, 1, 2
GS_PATH_AUTO, GS_PATH_TENSOR, GS_PATH_SIMT = 0, 1, 2
STATUS_NAMES = {
    0: "GS_OK", 1: "GS_ERR_INVALID_ARGUMENT", 2: "GS_ERR_UNSUPPORTED",
    3: "GS_ERR_OUT_OF_MEMORY", 4: "GS_ERR_CUDA", 5: "GS_ERR_DEVICE_TIMEOUT",
}

# Every symbol include/gauss_sum.h declares.
EXPORTS = (
    "gauss_sum_default_options", "gauss_sum", "gauss_sum_ex", "gauss_sum_grad_q",
    "gauss_sum_grad_q_ex", "gauss_sum_workspace_size", "gauss_sum_device_status",
    "gauss_sum_last_error", "gauss_sum_status_string", "gauss_sum_probe_ex2_rate",
    "gauss_sum_noalloc", "gauss_sum_kernel_launches", "gauss_sum_batched", "gauss_sum_mmd2",
    "gauss_sum_vjp", "gauss_sum_probe_ex2_mix_rate",
)
# Test hooks declared in include/gauss_sum_testing.h.
TESTING_EXPORTS = ("gauss_sum_testing_fail_allocations", "gauss_sum_testing_request_stall",
                   "gauss_sum_testing_last_fma_variant")

# Bytes of the static scratch array behind gauss_sum_noalloc
# (GS_NOALLOC_SCRATCH_BYTES in include/gauss_sum.h).
NOALLOC_SCRATCH_BYTES = 32 * 1024 * 1024


class GaussSumError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status
        self.message = message


class GsOptions(ctypes.Structure):
    _fields_ = [("center", ctypes.c_int), ("split_n", ctypes.c_int),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
                ("path", ctypes.c_int), ("main_events", ctypes.c_void_p * 2),
                ("exp2_fma", ctypes.c_int)]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return LIB_PATH


def load_library(path: str | None = None):
    """Load (once) and return the ctypes handle of libgauss_sum.so."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(
                f"{p} is missing: build the CUDA library first "
                "(python -m paper_2609_04910_gb300.build or __graft_entry__.build())")
        lib = ctypes.CDLL(p)
        _declare(lib)
        if path is None:
            _lib = lib
        return lib


def _declare(lib):
    vp, i64, f = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    d = ctypes.c_double
    lib.gauss_sum_default_options.argtypes = [ctypes.POINTER(GsOptions)]
    lib.gauss_sum_default_options.restype = None
    lib.gauss_sum.argtypes = [vp, vp, vp, d, i64, i64, i64, i64, f, vp, vp]
    lib.gauss_sum.restype = f
    lib.gauss_sum_ex.argtypes = [vp, vp, vp, d, i64, i64, i64, i64, f, vp, vp,
                                 ctypes.POINTER(GsOptions)]
    lib.gauss_sum_ex.restype = f
    lib.gauss_sum_grad_q.argtypes = [vp, vp, vp, d, i64, i64, i64, f, vp, vp, vp]
    lib.gauss_sum_grad_q.restype = f
    lib.gauss_sum_grad_q_ex.argtypes = [vp, vp, vp, d, i64, i64, i64, f, vp, vp, vp,
                                        ctypes.POINTER(GsOptions)]
    lib.gauss_sum_grad_q_ex.restype = f
    lib.gauss_sum_workspace_size.argtypes = [i64, i64, i64, i64, f, f, ctypes.POINTER(GsOptions)]
    lib.gauss_sum_workspace_size.restype = ctypes.c_size_t
    lib.gauss_sum_device_status.argtypes = [vp]
    lib.gauss_sum_device_status.restype = f
    lib.gauss_sum_last_error.argtypes = []
    lib.gauss_sum_last_error.restype = ctypes.c_char_p
    lib.gauss_sum_status_string.argtypes = [f]
    lib.gauss_sum_status_string.restype = ctypes.c_char_p
    lib.gauss_sum_probe_ex2_rate.argtypes = [vp, ctypes.POINTER(ctypes.c_double)]
    lib.gauss_sum_probe_ex2_rate.restype = f
    lib.gauss_sum_probe_ex2_mix_rate.argtypes = [vp, ctypes.POINTER(ctypes.c_double)]
    lib.gauss_sum_probe_ex2_mix_rate.restype = f
    lib.gauss_sum_noalloc.argtypes = [vp, vp, vp, d, i64, i64, i64, i64, f, vp, vp]
    lib.gauss_sum_noalloc.restype = f
    lib.gauss_sum_kernel_launches.argtypes = []
    lib.gauss_sum_kernel_launches.restype = ctypes.c_uint64
    lib.gauss_sum_batched.argtypes = [vp, vp, vp, d, i64, i64, i64, i64, i64, f, vp, vp]
    lib.gauss_sum_batched.restype = f
    lib.gauss_sum_mmd2.argtypes = [vp, vp, d, i64, i64, i64, f, vp, vp]
    lib.gauss_sum_mmd2.restype = f
    lib.gauss_sum_vjp.argtypes = [vp, vp, vp, vp, d, i64, i64, i64, i64, f, vp, vp, vp, vp]
    lib.gauss_sum_vjp.restype = f
    lib.gauss_sum_testing_fail_allocations.argtypes = [f]
    lib.gauss_sum_testing_fail_allocations.restype = None
    lib.gauss_sum_testing_request_stall.argtypes = [vp]
    lib.gauss_sum_testing_request_stall.restype = f
    lib.gauss_sum_testing_last_fma_variant.argtypes = []
    lib.gauss_sum_testing_last_fma_variant.restype = f


def _check(lib, status: int):
    if status != 0:
        raise GaussSumError(status, lib.gauss_sum_last_error().decode())


def options(center=True, split_n=0, workspace=None, workspace_bytes=0, path=GS_PATH_AUTO,
            main_events=None, exp2_fma=0):
    """gs_options; ``main_events`` is an optional pair of torch.cuda.Event
    (already recorded once, so that their CUDA events exist) that the call
    records around its main kernel."""
    o = GsOptions()
    load_library().gauss_sum_default_options(ctypes.byref(o))
    o.center = 1 if center else 0
    o.split_n = int(split_n)
    o.workspace = workspace
    o.workspace_bytes = int(workspace_bytes)
    o.path = int(path)
    o.exp2_fma = int(exp2_fma)
    if main_events is not None:
        o.main_events[0] = main_events[0].cuda_event
        o.main_events[1] = main_events[1].cuda_event
    return o


def _dtype_code(t):
    import torch
    if t.dtype == torch.float32:
        return GS_FP32
    if t.dtype == torch.float16:
        return GS_FP16
    if t.dtype == torch.bfloat16:
        return GS_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _stream_ptr(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _check_tensor(t, name):
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def gauss_sum(q, k, v, tau, out=None, stream=None, center=True, split_n=0, workspace=None,
              main_events=None, path=GS_PATH_AUTO, exp2_fma=0):
    """Eq. 1: s[m] = sum_n exp(-tau/2 ||q_m - k_n||^2) v[n] as an (M, C) fp32 tensor.

    q: (M, D), k: (N, D), v: (N, C) or (N,) CUDA tensors of one dtype
    (fp32, fp16 or bf16).  ``q`` may be the same tensor as ``k``.
    ``exp2_fma`` (0..4) moves a share of the exponentials to the FMA pipe
    (gs_options.exp2_fma).
    """
    import torch
    lib = load_library()
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _check_tensor(t, n)
    M, D = q.shape
    N = k.shape[0]
    C = 1 if v.dim() == 1 else v.shape[1]
    if out is None:
        out = torch.empty((M, C), dtype=torch.float32, device=q.device)
    opt = options(center=center, split_n=split_n,
                  workspace=None if workspace is None else workspace.data_ptr(),
                  workspace_bytes=0 if workspace is None else workspace.numel() * workspace.element_size(),
                  main_events=main_events, path=path, exp2_fma=exp2_fma)
    st = lib.gauss_sum_ex(_ptr(q), _ptr(k), _ptr(v), float(tau), M, N, D, C, _dtype_code(q),
                          _ptr(out), _stream_ptr(stream), ctypes.byref(opt))
    _check(lib, st)
    return out


def gauss_sum_batched(q, k, v, tau, out=None, stream=None):
    """A batch of independent problems of Eq. 1: q (B, M, D), k (B, N, D),
    v (B, N, C) or (B, N) CUDA tensors of one dtype; returns (B, M, C)
    fp32.  ``q`` may be the same tensor as ``k``."""
    import torch
    lib = load_library()
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _check_tensor(t, n)
    B, M, D = q.shape
    N = k.shape[1]
    C = 1 if v.dim() == 2 else v.shape[2]
    if out is None:
        out = torch.empty((B, M, C), dtype=torch.float32, device=q.device)
    st = lib.gauss_sum_batched(_ptr(q), _ptr(k), _ptr(v), float(tau), B, M, N, D, C,
                               _dtype_code(q), _ptr(out), _stream_ptr(stream))
    _check(lib, st)
    return out


def gauss_sum_mmd2(x, v, tau, out=None, stream=None):
    """Squared MMD of Sec. 3: x (B, N, D) or (N, D) points with signed
    weights v (B, N) or (N,); returns (B,) fp32 (a 1-element tensor for
    unbatched input) with mmd2[b] = v_b^T K(x_b, x_b) v_b."""
    import torch
    lib = load_library()
    for t, n in ((x, "x"), (v, "v")):
        _check_tensor(t, n)
    if x.dim() == 2:
        B, (N, D) = 1, x.shape
    else:
        B, N, D = x.shape
    if out is None:
        out = torch.empty((B,), dtype=torch.float32, device=x.device)
    st = lib.gauss_sum_mmd2(_ptr(x), _ptr(v), float(tau), B, N, D, _dtype_code(x), _ptr(out),
                            _stream_ptr(stream))
    _check(lib, st)
    return out


def gauss_sum_vjp(q, k, v, g, tau, want=("q", "k", "v"), grad_q=None, grad_k=None,
                  grad_v=None, stream=None):
    """Vector-Jacobian product of Eq. 1 for the upstream g (M, C) fp32:
    returns (grad_q (M, D), grad_k (N, D), grad_v (N, C)) as fp32 tensors,
    None for the outputs not named in ``want``."""
    import torch
    lib = load_library()
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (g, "g")):
        _check_tensor(t, n)
    if g.dtype != torch.float32:
        raise ValueError("g must be float32")
    M, D = q.shape
    N = k.shape[0]
    C = 1 if v.dim() == 1 else v.shape[1]

    def out(given, name, shape):
        if given is None and name in want:
            given = torch.empty(shape, dtype=torch.float32, device=q.device)
        return given

    grad_q = out(grad_q, "q", (M, D))
    grad_k = out(grad_k, "k", (N, D))
    grad_v = out(grad_v, "v", (N, C))
    st = lib.gauss_sum_vjp(_ptr(q), _ptr(k), _ptr(v), _ptr(g), float(tau), M, N, D, C,
                           _dtype_code(q), _ptr(grad_q), _ptr(grad_k), _ptr(grad_v),
                           _stream_ptr(stream))
    _check(lib, st)
    return grad_q, grad_k, grad_v


def gauss_sum_noalloc(q, k, v, tau, out=None, stream=None):
    """Eq. 1 like ``gauss_sum`` but without any device allocation by the
    library: its scratch lives in a static 32 MiB device array (see
    ``gauss_sum_noalloc`` in include/gauss_sum.h for the rules of use).
    ``out`` should be passed by callers that must not allocate at all."""
    import torch
    lib = load_library()
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _check_tensor(t, n)
    M, D = q.shape
    N = k.shape[0]
    C = 1 if v.dim() == 1 else v.shape[1]
    if out is None:
        out = torch.empty((M, C), dtype=torch.float32, device=q.device)
    st = lib.gauss_sum_noalloc(_ptr(q), _ptr(k), _ptr(v), float(tau), M, N, D, C, _dtype_code(q),
                               _ptr(out), _stream_ptr(stream))
    _check(lib, st)
    return out


def gauss_sum_grad_q(q, k, v, tau, grad=None, s_out=None, want_s=True, stream=None,
                     center=True, split_n=0, workspace=None, main_events=None):
    """Sec. 3 q-gradient for scalar weights.  Returns (grad (M, D), s (M,) or None)."""
    import torch
    lib = load_library()
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _check_tensor(t, n)
    M, D = q.shape
    N = k.shape[0]
    if grad is None:
        grad = torch.empty((M, D), dtype=torch.float32, device=q.device)
    if s_out is None and want_s:
        s_out = torch.empty((M,), dtype=torch.float32, device=q.device)
    opt = options(center=center, split_n=split_n,
                  workspace=None if workspace is None else workspace.data_ptr(),
                  workspace_bytes=0 if workspace is None else workspace.numel() * workspace.element_size(),
                  main_events=main_events)
    st = lib.gauss_sum_grad_q_ex(_ptr(q), _ptr(k), _ptr(v), float(tau), M, N, D, _dtype_code(q),
                                 _ptr(grad), _ptr(s_out), _stream_ptr(stream), ctypes.byref(opt))
    _check(lib, st)
    return grad, s_out


def gauss_sum_workspace_size(M, N, D, C, dtype_code, grad=False, center=True, split_n=0,
                             path=GS_PATH_AUTO):
    lib = load_library()
    opt = options(center=center, split_n=split_n, path=path)
    return int(lib.gauss_sum_workspace_size(M, N, D, C, dtype_code, 1 if grad else 0,
                                            ctypes.byref(opt)))


def gauss_sum_device_status(stream=None):
    """Synchronise and return (and clear) the device status; raises on a timeout."""
    lib = load_library()
    st = lib.gauss_sum_device_status(_stream_ptr(stream))
    _check(lib, st)
    return st


def gauss_sum_probe_ex2_rate(stream=None) -> float:
    lib = load_library()
    r = ctypes.c_double(0.0)
    _check(lib, lib.gauss_sum_probe_ex2_rate(_stream_ptr(stream), ctypes.byref(r)))
    return r.value


def gauss_sum_probe_ex2_mix_rate(stream=None) -> float:
    """exp2 rate reachable with the FMA kernel's exponent-loop instruction
    mix (see include/gauss_sum.h), in exponentials per second."""
    lib = load_library()
    r = ctypes.c_double(0.0)
    _check(lib, lib.gauss_sum_probe_ex2_mix_rate(_stream_ptr(stream), ctypes.byref(r)))
    return r.value


def gauss_sum_kernel_launches() -> int:
    """Kernels the library has launched in this process (all devices)."""
    return int(load_library().gauss_sum_kernel_launches())


def testing_fail_allocations(on: bool) -> None:
    """Test hook: make the library's workspace allocations fail (or not)."""
    load_library().gauss_sum_testing_fail_allocations(1 if on else 0)


def testing_last_fma_variant() -> int:
    """Bit flags of the last fused FMA-kernel launch (test hook): 1 =
    overlapped segment transitions, 2 = banded key order, 4 = q^ in TMEM;
    -1 before the first launch."""
    return int(load_library().gauss_sum_testing_last_fma_variant())


def testing_request_stall(stream=None) -> None:
    """Test hook: the next FMA-kernel launch gives up one bounded wait."""
    lib = load_library()
    _check(lib, lib.gauss_sum_testing_request_stall(_stream_ptr(stream)))
