"""The five workloads at full size, in the launch configuration bench.py
times (default options), checked against the float64 oracle on all rows
(fp32_d16, mmd_d64) or on seeded row samples the oracle computes one by one
(multi_c64: 256 rows, svgd_d32: 4096, offset_d256: 1024 with centring on
and off, the q = k reading of mmd_d64: 1024)."""
import numpy as np
import pytest

from paper_2609_04910_gb300.workloads import WORKLOADS, sample_rows
from tests.gpu_helpers import forward_check, grad_check

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


def test_fp32_d16_all_rows():
    w = WORKLOADS["fp32_d16"]
    rel, *_ = forward_check(w)
    print(f"fp32_d16 max rel {rel:.3e}")


def test_mmd_d64_all_rows():
    """The bench workload (independent q and k draws) on every one of its
    65536 rows."""
    w = WORKLOADS["mmd_d64"]
    rel, got, ref, den = forward_check(w)
    print(f"mmd_d64 all rows max rel {rel:.3e}")


def test_mmd_d64_q_is_k_sampled_rows():
    """The other reading of the MMD workload: q = k = X (one cloud carrying
    the two signed halves), 1024 seeded rows."""
    w = WORKLOADS["mmd_d64_qk"]
    rel, *_ = forward_check(w, rows=sample_rows(w.M, 1024))
    print(f"mmd_d64 (q = k) max rel {rel:.3e}")


def test_multi_c64_256_rows():
    w = WORKLOADS["multi_c64"]
    rel, *_ = forward_check(w, rows=sample_rows(w.M, 256))
    print(f"multi_c64 max rel {rel:.3e}")


def test_svgd_d32_grad_and_sum():
    w = WORKLOADS["svgd_d32"]
    relg, rels = grad_check(w, rows=sample_rows(w.M, 4096))
    print(f"svgd_d32 grad max rel {relg:.3e}, s max rel {rels:.3e}")


@pytest.mark.parametrize("center", [True, False])
def test_offset_d256(center):
    w = WORKLOADS["offset_d256"]
    rel, got, ref, den = forward_check(w, rows=sample_rows(w.M, 1024), center=center)
    print(f"offset_d256 center={center} max rel {rel:.3e}")
