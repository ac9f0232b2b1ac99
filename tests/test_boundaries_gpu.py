"""GPU parity at the thresholds where the library switches kernels or
layouts, each side of every switch against the float64 oracle.

Switches (plan_tensor / plan_simt): augmented operands of the FMA kernel
(fp16 D + 4 <= 128, bf16 D + 6 <= 128) versus q^ in TMEM; FMA kernel
(C <= 4) versus two-MMA kernel, and for three or four channels on
augmented rows the call size (2^28 pairs); augmented two-MMA operands
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


@pytest.mark.parametrize("C", [2, 3, 4])
def test_three_and_four_channels_switch_kernels_at_2_28_pairs(C):
    """From 2^28 pairs a single call with three or four channels on
    augmented rows takes the two-MMA kernel (its value preparation adds
    launches), below it and with two channels the FMA kernel: sampled rows
    of both sides against the oracle."""
    import numpy as np
    import paper_2609_04910_gb300 as gs
    rows = np.arange(0, 16384, 61)
    launches = []
    for N in (16383, 16384):
        before = gs.gauss_sum_kernel_launches()
        forward_check(case(16384, N, 64, C, "fp16"), rows=rows)
        launches.append(gs.gauss_sum_kernel_launches() - before)
    if C == 2:
        assert launches[1] == launches[0]
    else:
        assert launches[1] > launches[0]


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


def _value_pattern(N, pattern, rng):
    """fp16 values with the sign structure the folded-value path
    distinguishes: groups of 32 keys of one sign (no record loads), mixed
    groups, zeros, and magnitudes across the fp16 range."""
    import numpy as np
    if pattern == "halves":          # MMD weights: every group of one sign
        v = np.where(np.arange(N) < N // 2, 1.0, -1.0) / N
    elif pattern == "random":        # mixed groups throughout
        v = rng.standard_normal(N)
    elif pattern == "blocks":        # runs of 32 or 96 keys of one sign, some groups with a zero
        v = np.repeat(np.where(rng.random((N + 31) // 32) < 0.5, 1.0, -1.0), 32)[:N]
        v = v * rng.uniform(0.5, 2.0, N)
        v[rng.choice(N, size=max(1, N // 100), replace=False)] = 0.0
    else:                            # "range": magnitudes from subnormal to near 65504
        v = np.exp2(rng.uniform(-23.0, 15.9, N)) * np.where(rng.random(N) < 0.5, 1.0, -1.0)
    return v.astype(np.float16).reshape(N, 1)


@pytest.mark.parametrize("pattern", ["halves", "random", "blocks", "range"])
@pytest.mark.parametrize("center", [True, False])
def test_folded_value_magnitudes(pattern, center):
    """One fp16 value channel: the value magnitudes are folded into the key
    operands (log2(|v| 2^-16) / c in the key norm term) and the key records
    hold only signs, with a per-32-key-group sign word that lets groups of
    one sign skip the record loads.  Against the oracle for every sign
    pattern, with and without centring (the sign records then come from
    their own kernel rather than the mean launch).  The shape gives every
    CTA long runs of key tiles (65 key tiles, 110 units per CTA), where the
    folded path is used; sampled rows."""
    import numpy as np
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300._binding import testing_last_fma_variant
    from paper_2609_04910_gb300.workloads import sample_rows
    rng = np.random.default_rng(7)
    M, N, D = 65536, 8320, 48
    q = rng.standard_normal((M, D)).astype(np.float16)
    k = rng.standard_normal((N, D)).astype(np.float16)
    v = _value_pattern(N, pattern, rng)
    tau = 1.0 / D
    s = gs.gauss_sum(torch.from_numpy(q).cuda(), torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                     tau, center=center)
    gs.gauss_sum_device_status()
    assert testing_last_fma_variant() & 8, "folded-value path not taken"
    rows = sample_rows(M, 256)
    ref, den = oracle_sum(q, k, v, tau, rows=rows)
    rel = float(np.max(np.abs(s.cpu().numpy()[rows] - ref) / (den + 1e-30)))
    assert rel <= 2e-3, f"{pattern} center={center}: max rel {rel:.3e}"


def test_folded_values_only_for_one_fp16_channel_and_long_runs():
    """bf16 values (range beyond 2^16), C > 1 and short runs of key tiles
    (small problems: the extra launches would cost more than they save)
    keep the value records."""
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300._binding import testing_last_fma_variant
    for n, dtype, C in ((65536, torch.bfloat16, 1), (65536, torch.float16, 2), (300, torch.float16, 1)):
        q = torch.randn(n, 32, device="cuda").to(dtype)
        v = torch.randn(n, C, device="cuda").to(dtype)
        gs.gauss_sum(q, q, v, 1.0 / 32)
        gs.gauss_sum_device_status()
        assert not testing_last_fma_variant() & 8, (n, dtype, C)


def test_folded_values_both_passes_in_one_batch():
    """A batch whose problems differ in sign structure: problems whose
    32-key groups all have values of one sign go through the first pass
    of the fused kernel, the others through the second; together they
    give every problem's sum (against the oracle, problem by problem)."""
    import numpy as np
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300._binding import testing_last_fma_variant
    from paper_2609_04910_gb300.workloads import sample_rows
    rng = np.random.default_rng(11)
    B, M, n, D = 4, 16384, 8320, 32
    q = rng.standard_normal((B, M, D)).astype(np.float16)
    k = rng.standard_normal((B, n, D)).astype(np.float16)
    v = np.stack([_value_pattern(n, pat, rng) for pat in ("halves", "random", "blocks", "range")])
    tau = 1.0 / D
    s = gs.gauss_sum_batched(torch.from_numpy(q).cuda(), torch.from_numpy(k).cuda(),
                             torch.from_numpy(v).cuda(), tau)
    gs.gauss_sum_device_status()
    assert testing_last_fma_variant() & 8, "folded-value path not taken"
    s = s.cpu().numpy()
    rows = sample_rows(M, 128)
    for b in range(B):
        ref, den = oracle_sum(q[b], k[b], v[b], tau, rows=rows)
        rel = float(np.max(np.abs(s[b][rows] - ref) / (den + 1e-30)))
        assert rel <= 2e-3, f"problem {b}: max rel {rel:.3e}"


@pytest.mark.parametrize("dtype,C,tau,folded", [
    ("fp16", 3, 1.0 / 40, True),     # exponent scale folded into the query rows
    ("fp16", 1, 1.0 / 40, True),     # small problem: scale folded, value records kept
    ("fp16", 2, 0.4, False),         # c = tau log2 e > 1/2: rn(c q^) could overflow
    ("bf16", 2, 1.0 / 40, False),    # bf16 rows keep the multiply
])
def test_folded_exponent_scale_switch(dtype, C, tau, folded):
    """fp16 augmented operands of the FMA kernel carry the exponent scale c
    in the query rows (rn(c q^), norm term -||rn(c q^)||^2 / (2c)) when
    2^-14 <= c <= 1/2; each side against the oracle."""
    from paper_2609_04910_gb300._binding import testing_last_fma_variant
    forward_check(case(300, 700, 40, C, dtype, tau=tau))
    assert bool(testing_last_fma_variant() & 16) == folded, testing_last_fma_variant()
