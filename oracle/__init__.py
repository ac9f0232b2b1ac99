"""Float64 CPU oracle for the Gauss kernel sum -- TEST INFRASTRUCTURE ONLY.

The oracle evaluates Eq. 1 of arXiv 2609.04910 (the Gauss kernel sum) and
the q-gradient of Sec. 3 and the vector-Jacobian product of Eq. 1 (the
gradients of sum_m g_m . s_m in q, k and v) with plain loops in C
(``gauss_oracle.c``),
and the squared MMD of Sec. 3 as v^T s on top of that sum,
from the dtype-rounded inputs upcast to float64.  It shares no code with the
CUDA library and is only used by ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py``.  The library itself never imports it.

Parity status: every function here is pinned by CPU tests against closed
forms, symmetry, two independent algebraic routes (Alg. 1 and Alg. 2 written
out in float64), finite differences, a Monte-Carlo expectation and brute
force on tiny inputs (``tests/test_oracle_pins.py``).
"""
from .oracle import (build_oracle, oracle_sum, oracle_grad_q, oracle_mmd2, oracle_vjp,
                     oracle_max_threads, oracle_library_path)

__all__ = ["build_oracle", "oracle_sum", "oracle_grad_q", "oracle_mmd2", "oracle_vjp",
           "oracle_max_threads", "oracle_library_path"]
