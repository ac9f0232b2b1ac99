"""gauss_sum_noalloc, the allocation-free entry point.

Some callers cannot allocate device memory at the point of the call: code
inside a framework that owns every device allocation through its own pool,
or code that has reserved all free device memory up front.  They call
gauss_sum_noalloc, which runs the same kernels as gauss_sum with the
library's static 32 MiB scratch array as its workspace.  The checks here:
two calls in a row (the second one reuses the scratch the first one left
behind) match gauss_sum and the float64 oracle, on the FMA kernel (C <= 4)
and on the two-MMA kernel (C > 4, whose per-channel maximum is the one
scratch accumulator a call must clear itself); the calls succeed while every
library allocation is made to fail (so none is attempted); and sizes beyond
the array are rejected.  This file is named so that pytest collects it last.
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


# Two calls in a row per group: FMA kernel (C <= 4; the first case is the
# q = k MMD form), then the two-MMA kernel (C > 4) twice with different
# value magnitudes, so that a per-channel maximum left in the scratch by the
# first call would spoil the second one's value scaling.
CASES = [
    (case(700, 700, 64, 1, "fp16", kind="mmd", q_is_k=True), 3, 1.0),
    (case(257, 515, 48, 3, "fp16"), 3, 1.0),
    (case(300, 470, 40, 20, "fp16"), 4, 1000.0),
    (case(300, 470, 40, 20, "fp16"), 5, 0.001),
    (case(200, 333, 32, 9, "bf16"), 6, 1.0),
]


@pytest.mark.parametrize("fail_allocations", [False, True])
def test_noalloc_matches_gauss_sum_and_the_oracle_on_calls_in_a_row(fail_allocations):
    """Every call agrees with gauss_sum and with the oracle within the parity
    tolerance, measured against the oracle's scale sum_n Phi |v|.  With every
    library allocation made to fail, gauss_sum_noalloc still succeeds: it
    allocates nothing."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300._binding import testing_fail_allocations
    for w, seed, vscale in CASES:
        inp = generate(w, seed=seed)
        q, k, v = device_inputs(inp)
        v = (v.float() * vscale).to(v.dtype)
        v64 = v.double().cpu().numpy()
        ref = gs.gauss_sum(q, k, v, w.tau)
        gs.gauss_sum_device_status()
        out = torch.full((w.M, w.C), float("nan"), device="cuda")
        testing_fail_allocations(fail_allocations)
        try:
            st, lib = _noalloc_call(q, k, v, w.tau, out)
        finally:
            testing_fail_allocations(False)
        assert st == 0, lib.gauss_sum_last_error()
        gs.gauss_sum_device_status()
        want, den = oracle_sum(inp["q64"], inp["k64"], v64, w.tau)
        got = out.cpu().numpy()
        rel_ref = np.max(np.abs(got - ref.cpu().numpy()) / (den + 1e-30))
        rel_oracle = np.max(np.abs(got - want) / (den + 1e-30))
        assert rel_ref <= TOL[w.dtype], f"{w.name}: against gauss_sum rel {rel_ref:.3e}"
        assert rel_oracle <= TOL[w.dtype], f"{w.name}: against the oracle rel {rel_oracle:.3e}"


def test_noalloc_runs_the_bench_workload_like_gauss_sum():
    """The 65536 x 65536, D = 64, C = 1 fp16 workload (21 MiB of scratch)
    fits the array; the same kernels in the same order give the same bits
    as gauss_sum, twice in a row."""
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import WORKLOADS
    w = WORKLOADS["mmd_d64"]
    q, k, v = device_inputs(generate(w, seed=0))
    ref = gs.gauss_sum(q, k, v, w.tau)
    for _ in range(2):
        out = torch.full((w.M, w.C), float("nan"), device="cuda")
        st, lib = _noalloc_call(q, k, v, w.tau, out)
        assert st == 0, lib.gauss_sum_last_error()
        gs.gauss_sum_device_status()
        assert torch.equal(out, ref)


def test_noalloc_rejects_calls_beyond_the_static_scratch():
    q = torch.zeros((262144, 128), dtype=torch.float16, device="cuda")
    v = torch.zeros((262144, 1), dtype=torch.float16, device="cuda")
    out = torch.empty((262144, 1), dtype=torch.float32, device="cuda")
    st, lib = _noalloc_call(q, q, v, 0.1, out)
    assert st == 2  # GS_ERR_UNSUPPORTED
    assert b"static scratch" in lib.gauss_sum_last_error()
