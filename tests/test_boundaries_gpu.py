"""GPU parity at the thresholds where the library switches kernels or
layouts, each side of every switch against the float64 oracle.

Switches (plan_tensor / plan_simt): augmented operands of the FMA kernel
(fp16 D + 4 <= 128, bf16 D + 6 <= 128) versus q^ in TMEM; FMA kernel
(C <= 4) versus two-MMA kernel; augmented two-MMA operands
(Dp_aug + Cp <= 128); 128- versus 64-key tiles (Cp <= 128); early S
release (four or more stages) versus one MMA warp; gradient channels in one
launch (D + 1 <= 256) versus two; fp32 register tiles of 16 / 32 / 64 / 128
coordinates; 3xTF32 tensor-core variant (D <= 32, C <= 4); overlapped
segment transitions of the FMA kernel (runs of at most 64 key tiles).  Key
counts straddle one key tile (127, 128, 129).
"""
import pytest

from tests.gpu_helpers import case, forward_check, grad_check

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("D,dtype", [(123, "fp16"), (124, "fp16"), (125, "fp16"),
                                     (121, "bf16"), (122, "bf16"), (123, "bf16")])
@pytest.mark.parametrize("C", [1, 4])
def test_fma_augmented_switch(D, dtype, C):
    forward_check(case(130, 300, D, C, dtype))


@pytest.mark.parametrize("C", [4, 5])
@pytest.mark.parametrize("N", [127, 128, 129])
def test_fma_two_mma_switch(C, N):
    forward_check(case(140, N, 40, C, "fp16"))


@pytest.mark.parametrize("D,C", [(64, 48), (64, 49), (60, 64), (61, 64)])
def test_two_mma_augmented_switch(D, C):
    # fp16 augmented rows: Dp = ceil((D + 4) / 16) 16; augmented when Dp + Cp <= 128.
    forward_check(case(150, 400, D, C, "fp16"))


@pytest.mark.parametrize("C", [128, 129])
def test_key_tile_width_switch(C):
    forward_check(case(150, 300, 32, C, "fp16"))


@pytest.mark.parametrize("D,C,dtype", [(64, 100, "fp16"), (96, 100, "fp16"), (128, 64, "bf16"),
                                       (128, 48, "bf16")])
def test_schedule_switch(D, C, dtype):
    # Four stages (early S release) or three (one MMA warp), near the edge.
    forward_check(case(150, 700, D, C, dtype), split_n=1)


@pytest.mark.parametrize("D", [254, 255, 256])
def test_gradient_channel_chunks(D):
    grad_check(case(70, 200, D, 1, "fp16"))


@pytest.mark.parametrize("D", [16, 17, 32, 33, 64, 65, 128])
def test_fp32_register_tiles(D):
    forward_check(case(100, 129, D, 2, "fp32"))


@pytest.mark.parametrize("D", [16, 17, 64])
def test_fp32_gradient_register_tiles(D):
    grad_check(case(100, 129, D, 1, "fp32"))


@pytest.mark.parametrize("D,C", [(31, 4), (32, 4), (32, 1), (8, 3)])
def test_fp32_tensor_variant_edges(D, C):
    import paper_2609_04910_gb300 as gs
    forward_check(case(130, 257, D, C, "fp32"), path=gs.GS_PATH_TENSOR)


def test_ex2_rate_probes():
    """The MUFU probe stays below 32 exp2 per clock per SM at a 2.2 GHz
    bound, and the probe of the FMA kernel's exponent-loop instruction mix
    (which adds multiplies, loads and FMAs to every exp2) does not exceed it."""
    import torch
    import paper_2609_04910_gb300 as gs
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    plain = gs.gauss_sum_probe_ex2_rate()
    mix = gs.gauss_sum_probe_ex2_mix_rate()
    assert 0 < plain <= 32 * sms * 2.2e9
    assert 0 < mix <= 1.05 * plain


@pytest.mark.parametrize("M,N,overlap,banded", [
    (65536, 8192, True, False),      # 64 key tiles per pair of query tiles: overlapped
    (65536, 8320, False, False),     # 65 key tiles, 110 units per CTA: segment barrier
    (2048, 8320, True, False),       # 65 key tiles but 4 units per CTA: overlapped
    (1024, 524288, True, True),      # keys beyond half the L2: bands of 64 key tiles
])
def test_fma_segment_overlap_switch(M, N, overlap, banded):
    """The FMA kernel overlaps segment transitions when a CTA's runs of key
    tiles for one pair of query tiles are at most 64 tiles long (the
    smaller of the key tiles per pair and the units per CTA, or the band
    length); each side against the oracle on sampled rows."""
    from paper_2609_04910_gb300._binding import testing_last_fma_variant
    from paper_2609_04910_gb300.workloads import sample_rows
    w = case(M, N, 64, 1, "fp16")
    forward_check(w, rows=sample_rows(M, 256))
    flags = testing_last_fma_variant()
    assert bool(flags & 1) == overlap, flags
    assert bool(flags & 2) == banded, flags
