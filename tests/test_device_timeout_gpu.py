"""A device-side wait that runs out of time, without faulting the GPU.

Every mbarrier wait of the fused kernels is bounded (2 s of globaltimer);
when one runs out, the kernel writes GS_ERR_DEVICE_TIMEOUT and where it
happened into the device status words, raises an abort flag that every
other role of the CTA polls, frees its tensor memory and returns.  The test
hook gauss_sum_testing_request_stall makes one control warp of CTA 0 wait on a barrier
that nothing arrives on; the test checks that gauss_sum_device_status
reports the timeout and that the next call on the same context runs
normally (its result matches the oracle).
"""
import numpy as np
import pytest

from tests.gpu_helpers import TOL, case, device_inputs, rel_err

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


def test_bounded_wait_runs_out_and_context_stays_usable():
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300.workloads import generate
    w = case(600, 900, 64, 1, "fp16")          # FMA kernel, augmented operands
    inp = generate(w)
    q, k, v = device_inputs(inp)
    gs.gauss_sum_device_status()               # start from a clear status

    from paper_2609_04910_gb300._binding import testing_request_stall
    testing_request_stall()
    gs.gauss_sum(q, k, v, w.tau)               # the launch itself succeeds
    with pytest.raises(gs.GaussSumError) as ei:
        gs.gauss_sum_device_status()
    assert ei.value.status == 5                # GS_ERR_DEVICE_TIMEOUT
    assert "block (0, 0)" in ei.value.message

    gs.gauss_sum_device_status()               # the status was cleared
    out = gs.gauss_sum(q, k, v, w.tau)
    gs.gauss_sum_device_status()
    ref, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
    assert rel_err(out.cpu().numpy(), ref, den) <= TOL["fp16"]
