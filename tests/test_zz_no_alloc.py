"""gauss_sum_noalloc, the allocation-free entry point, against gauss_sum.

Callers that cannot allocate device memory at the point of the call (code
inside a framework that owns all device allocations, or that has reserved
all free memory up front) use gauss_sum_noalloc, which runs the same
kernels with the library's static 16 MiB scratch array instead of an
allocated workspace.  This file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest

from tests.gpu_helpers import TOL, case
from paper_2609_04910_gb300.workloads import device_inputs, generate

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


def _noalloc_call(q, k, v, tau, out):
    """Call gauss_sum_noalloc directly through the C ABI."""
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300._binding import _dtype_code
    lib = gs.load_library()
    M, D = q.shape
    N = k.shape[0]
    C = v.shape[1]
    st = lib.gauss_sum_noalloc(ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()),
                               ctypes.c_void_p(v.data_ptr()), float(tau), M, N, D, C,
                               _dtype_code(q), ctypes.c_void_p(out.data_ptr()),
                               ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return st, lib


def test_noalloc_matches_gauss_sum_on_two_calls_in_a_row():
    """Two consecutive calls with different inputs (the second one reuses
    the scratch the first one left behind) agree with gauss_sum within the
    parity tolerance, measured against the oracle's scale sum_n Phi |v|."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    cases = [case(700, 700, 64, 1, "fp16", kind="mmd", q_is_k=True),
             case(257, 515, 48, 3, "fp16")]
    for w in cases:
        inp = generate(w, seed=3)
        q, k, v = device_inputs(inp)
        ref = gs.gauss_sum(q, k, v, w.tau)
        out = torch.full((w.M, w.C), float("nan"), device="cuda")
        st, lib = _noalloc_call(q, k, v, w.tau, out)
        assert st == 0, lib.gauss_sum_last_error()
        gs.gauss_sum_device_status()
        _, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
        rel = np.max(np.abs(out.cpu().numpy() - ref.cpu().numpy()) / (den + 1e-30))
        assert rel <= TOL[w.dtype], f"{w.name}: rel {rel:.3e}"


def test_noalloc_rejects_calls_beyond_the_static_scratch():
    q = torch.zeros((262144, 128), dtype=torch.float16, device="cuda")
    v = torch.zeros((262144, 1), dtype=torch.float16, device="cuda")
    out = torch.empty((262144, 1), dtype=torch.float32, device="cuda")
    st, lib = _noalloc_call(q, q, v, 0.1, out)
    assert st == 2  # GS_ERR_UNSUPPORTED
    assert b"static scratch" in lib.gauss_sum_last_error()
