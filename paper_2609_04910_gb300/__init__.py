"""GB300-native exact Gauss kernel sums (arXiv 2609.04910).

The computation lives in ``libgauss_sum.so`` (C ABI: ``include/gauss_sum.h``),
built from ``csrc/`` by ``build.build_library()``.  This package holds the
ctypes binding (argument marshalling only) and the seeded workload
generators.  The library is loaded on first use; if it is missing, calls
raise instead of falling back to anything else.
"""
from ._binding import (GS_BF16, GS_FP16, GS_FP32, GS_PATH_AUTO, GS_PATH_SIMT, GS_PATH_TENSOR,
                       EXPORTS, GaussSumError, gauss_sum, gauss_sum_batched, gauss_sum_device_status,
                       gauss_sum_mmd2, gauss_sum_noalloc, gauss_sum_vjp,
                       gauss_sum_grad_q, gauss_sum_kernel_launches, gauss_sum_probe_ex2_mix_rate,
                       gauss_sum_probe_ex2_rate,
                       gauss_sum_workspace_size,
                       library_path, load_library)

__all__ = [
    "GS_BF16", "GS_FP16", "GS_FP32", "GS_PATH_AUTO", "GS_PATH_SIMT", "GS_PATH_TENSOR",
    "EXPORTS", "GaussSumError", "gauss_sum", "gauss_sum_device_status", "gauss_sum_grad_q",
    "gauss_sum_batched", "gauss_sum_kernel_launches", "gauss_sum_mmd2", "gauss_sum_noalloc",
    "gauss_sum_probe_ex2_mix_rate", "gauss_sum_probe_ex2_rate", "gauss_sum_vjp", "gauss_sum_workspace_size", "library_path",
    "load_library",
]
