"""The seeded input generators: determinism, shapes and exact dtype rounding."""
import numpy as np
import pytest

from paper_2609_04910_gb300.workloads import WORKLOADS, generate, round_to, sample_rows, to_float64


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_small_versions_are_deterministic(name):
    w = WORKLOADS[name].resized(M=64, N=64)
    a = generate(w, seed=0)
    b = generate(w, seed=0)
    assert a["q"].shape == (w.M, w.D) and a["k"].shape == (w.N, w.D)
    assert a["v"].shape == (w.N, w.C)
    np.testing.assert_array_equal(a["q64"], b["q64"])
    np.testing.assert_array_equal(a["v64"], b["v64"])
    if w.q_is_k:
        assert a["q"] is a["k"]


def test_roundings_are_exact_and_nearest():
    x = np.array([1.0 + 2.0 ** -12, 1.0 + 3 * 2.0 ** -12, 65504.0, 1e-8])
    h = round_to(x, "fp16")
    assert h.dtype == np.float16
    np.testing.assert_array_equal(to_float64(h, "fp16"), [1.0, 1.0 + 2.0 ** -10, 65504.0, 0.0])
    b = round_to(np.array([1.0 + 2.0 ** -9, 1.0 + 3 * 2.0 ** -9, -2.5]), "bf16")
    assert b.dtype == np.uint16
    np.testing.assert_array_equal(to_float64(b, "bf16"), [1.0, 1.0 + 2.0 ** -7, -2.5])


def test_mmd_weights_and_offset_norm():
    w = WORKLOADS["mmd_d64"].resized(M=100, N=100)
    g = generate(w)
    assert np.sum(g["v64"] > 0) == 50 and np.sum(g["v64"] < 0) == 50
    w5 = WORKLOADS["offset_d256"].resized(M=8, N=8)
    g5 = generate(w5)
    mean = g5["k64"].mean(0)
    assert 45 < np.linalg.norm(mean) < 55


def test_sample_rows():
    r = sample_rows(1000, 10)
    assert len(r) == 10 and len(set(r.tolist())) == 10 and np.all(np.diff(r) > 0)
    assert np.array_equal(sample_rows(5, 10), np.arange(5))


def test_fp16_kernel_value_floor_never_binds_on_the_two_mma_workloads():
    """The two-MMA kernel stores each kernel value as fp16(2^(x + 15)), so
    values below 2^-29 lose precision (2^-39 and below flush to zero).  A row
    whose largest kernel value fell below that floor would have all of its
    terms there; on the two workloads that take this kernel (multi_c64,
    svgd_d32) the largest kernel value of every sampled row is far above it,
    so a per-row exponent offset (a row maximum before the exponentials)
    would change nothing there."""
    floor = 2.0 ** -29
    for name in ("multi_c64", "svgd_d32"):
        w = WORKLOADS[name]
        g = generate(w, seed=0)
        rows = sample_rows(w.M, 48, seed=5)
        q = g["q64"][rows]
        k = g["k64"]
        d2 = ((q * q).sum(1)[:, None] - 2.0 * q @ k.T + (k * k).sum(1)[None, :])
        phi_max = np.exp(-0.5 * w.tau * np.maximum(d2.min(axis=1), 0.0))
        assert phi_max.min() > 2.0 ** 10 * floor, (name, phi_max.min())
