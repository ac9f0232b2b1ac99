"""GPU parity: the CUDA path against the float64 oracle, element by element.

Tolerance (per output): rel = |s_gpu - s_oracle| / (sum_n Phi |v_n| + 1e-30)
must stay <= 2e-3 for fp16/bf16 inputs (fp16/bf16 MMA operands, fp32
accumulation) and <= 1e-5 for the fp32 SIMT path.  Shapes span several row
and key tiles with ragged tails; all calls go through the C ABI.
"""
import numpy as np
import pytest

from oracle import oracle_grad_q, oracle_sum
from paper_2609_04910_gb300.workloads import generate
from tests.gpu_helpers import TOL, case, device_inputs, forward_check, grad_check, rel_err

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


FWD_CASES = [
    # M, N, D, C, dtype
    (1, 1, 1, 1, "fp16"), (7, 130, 3, 1, "fp16"), (128, 128, 16, 16, "fp16"),
    (129, 257, 17, 2, "fp16"), (300, 1000, 64, 1, "fp16"), (257, 300, 100, 33, "fp16"),
    (130, 200, 128, 64, "fp16"), (64, 300, 255, 4, "fp16"), (200, 150, 256, 200, "fp16"),
    (100, 129, 32, 15, "fp16"), (513, 700, 8, 17, "fp16"), (90, 2000, 64, 128, "fp16"),
    (1, 1, 1, 1, "bf16"), (129, 257, 17, 2, "bf16"), (300, 500, 128, 64, "bf16"),
    (77, 260, 256, 1, "bf16"),
    (1, 1, 1, 1, "fp32"), (7, 130, 3, 1, "fp32"), (129, 257, 17, 2, "fp32"),
    (300, 1000, 64, 5, "fp32"), (100, 200, 128, 3, "fp32"), (50, 70, 32, 9, "fp32"),
]


@pytest.mark.parametrize("M,N,D,C,dtype", FWD_CASES)
def test_forward_parity(M, N, D, C, dtype):
    forward_check(case(M, N, D, C, dtype))


TF32_CASES = [
    # M, N, D, C (fp32 inputs on the tensor cores: 3xTF32 S, fp32 exponent and sums)
    (1, 1, 1, 1), (7, 130, 3, 1), (129, 257, 17, 2), (300, 1000, 16, 1), (260, 700, 32, 4),
    (513, 300, 8, 3), (1000, 3000, 16, 1),
]


@pytest.mark.parametrize("M,N,D,C", TF32_CASES)
def test_fp32_tensor_parity(M, N, D, C):
    import paper_2609_04910_gb300 as gs
    forward_check(case(M, N, D, C, "fp32"), path=gs.GS_PATH_TENSOR)


def test_fp32_tensor_aliasing_splits_and_offset():
    import paper_2609_04910_gb300 as gs
    t = gs.GS_PATH_TENSOR
    forward_check(case(300, 300, 16, 1, "fp32", kind="mmd", q_is_k=True), path=t)
    forward_check(case(260, 1500, 24, 3, "fp32"), path=t, split_n=3)
    # A common offset of norm 50: the centring keeps the Gram form exact.
    forward_check(case(200, 600, 32, 2, "fp32", kind="offset", tau=10.0 / 32), path=t)


def test_fp32_tensor_matches_simt():
    """Both fp32 kernels agree with each other within twice the tolerance."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300.workloads import generate
    w = case(700, 900, 16, 2, "fp32")
    q, k, v = device_inputs(generate(w))
    inp = generate(w)
    a = gs.gauss_sum(q, k, v, w.tau, path=gs.GS_PATH_TENSOR)
    b = gs.gauss_sum(q, k, v, w.tau, path=gs.GS_PATH_SIMT)
    gs.gauss_sum_device_status()
    _, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
    assert rel_err(a.cpu().numpy(), b.cpu().numpy(), den) <= 2 * TOL["fp32"]


@pytest.mark.parametrize("dtype", ["fp16", "bf16", "fp32"])
def test_forward_q_aliases_k(dtype):
    forward_check(case(300, 300, 64, 1, dtype, kind="mmd", q_is_k=True))


@pytest.mark.parametrize("split_n", [1, 2, 3, 7])
def test_key_splits(split_n):
    forward_check(case(260, 1500, 64, 3, "fp16"), split_n=split_n)


@pytest.mark.parametrize("D,dtype", [(64, "fp16"), (200, "fp16"), (120, "bf16"), (250, "bf16")])
def test_long_key_range_one_split(D, dtype):
    # One key split: every CTA walks 64 key tiles, so all control warps
    # cycle through their stages and S slots many times (q^ in shared
    # memory for D + 4 <= 128, in TMEM otherwise).
    forward_check(case(256, 8192, D, 3, dtype), split_n=1)


@pytest.mark.parametrize("M,N,D,C,dtype,grad", [
    (300, 5000, 64, 16, "fp16", False),   # BN 128, augmented, early S release (six stages)
    (200, 5000, 64, 100, "fp16", False),  # BN 128, plain operands, early S release (four stages)
    (200, 5000, 128, 64, "bf16", False),  # BN 128, q^ in TMEM buys a fourth stage: early release
    (200, 5000, 128, 96, "fp16", False),  # BN 128, q^ in shared memory (TMEM full), three
                                          # stages: one MMA warp, P-then-S order
    (150, 3000, 160, 48, "fp16", False),  # BN 128, q^ in TMEM buys a third stage: one MMA
                                          # warp, P-then-S order, A operand from TMEM
    (150, 3000, 32, 200, "fp16", False),  # BN 64, early S release
    (100, 3000, 256, 200, "fp16", False), # BN 64, two stages: one MMA warp
    (256, 5000, 32, 1, "fp16", True),     # gradient (33 channels), early S release
    (128, 3000, 100, 1, "bf16", True),    # gradient (101 channels), three stages
])
def test_two_mma_long_key_range(M, N, D, C, dtype, grad):
    """Two-MMA kernel over long key ranges in one split (tens of key tiles
    per CTA, so both S/P buffers and all stages cycle many times) on both
    schedules: the early S release with MMA1 and MMA2 issued by two warps,
    and one MMA warp in P-then-S order.  Repeated calls agree bit for bit
    and match the oracle."""
    import paper_2609_04910_gb300 as gs
    w = case(M, N, D, C, dtype, kind="mmd" if grad else "normal")
    inp = generate(w)
    q, k, v = device_inputs(inp)
    path = gs.GS_PATH_TENSOR
    if grad:
        outs = [gs.gauss_sum_grad_q(q, k, v, w.tau, split_n=1)[0] for _ in range(3)]
    else:
        outs = [gs.gauss_sum(q, k, v, w.tau, split_n=1, path=path) for _ in range(3)]
    gs.gauss_sum_device_status()
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    got = outs[0].cpu().numpy()
    if grad:
        ref, _, den, _ = oracle_grad_q(inp["q64"], inp["k64"], inp["v64"], w.tau)
    else:
        ref, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
    assert rel_err(got, ref, den) <= TOL[dtype]


@pytest.mark.parametrize("N", [100, 256, 300, 500, 640])
@pytest.mark.parametrize("D,C,grad", [(64, 16, False), (32, 200, False), (32, 1, True)])
def test_two_mma_few_key_tiles(N, D, C, grad):
    """One to five key tiles in one split on the early-release schedule
    (BN 128 and BN 64 forward, gradient): the MMA1 warp's first tiles need no
    S release, the second group may have no tile at all, and the MMA2 warp
    ends on either group."""
    if grad:
        grad_check(case(150, N, D, 1, "fp16"), split_n=1)
    else:
        forward_check(case(150, N, D, C, "fp16"), split_n=1)


@pytest.mark.parametrize("dtype", ["fp16", "bf16"])
def test_centering_off(dtype):
    forward_check(case(200, 400, 32, 2, dtype), center=False)


GRAD_CASES = [
    (300, 300, 32, "fp16", True), (129, 200, 17, "fp16", False), (150, 150, 64, "bf16", True),
    (64, 500, 100, "fp16", False), (40, 90, 255, "fp16", False),
    (100, 130, 16, "fp32", False), (64, 64, 64, "fp32", True), (33, 80, 5, "fp32", False),
]


@pytest.mark.parametrize("M,N,D,dtype,alias", GRAD_CASES)
def test_grad_parity(M, N, D, dtype, alias):
    grad_check(case(M, N, D, 1, dtype, kind="mmd" if alias else "normal", q_is_k=alias))


# ---------------------------------------------------------------- edge values
def _call(q, k, v, tau, **kw):
    import paper_2609_04910_gb300 as gs
    s = gs.gauss_sum(q, k, v, tau, **kw)
    gs.gauss_sum_device_status()
    return s


@pytest.mark.parametrize("dtype", ["fp16", "fp32"])
def test_zero_values_give_zero(dtype):
    tdt = {"fp16": torch.float16, "fp32": torch.float32}[dtype]
    q = torch.randn(200, 20, device="cuda", dtype=tdt)
    k = torch.randn(300, 20, device="cuda", dtype=tdt)
    v = torch.zeros(300, 3, device="cuda", dtype=tdt)
    assert torch.count_nonzero(_call(q, k, v, 0.5)).item() == 0


@pytest.mark.parametrize("dtype", ["fp16", "bf16", "fp32"])
def test_tiny_tau_gives_plain_sum(dtype):
    forward_check(case(150, 400, 24, 2, dtype, tau=1e-6))


@pytest.mark.parametrize("dtype", ["fp16", "fp32"])
def test_large_tau_coincident_points(dtype):
    # q = k, tau large: the self pair (exponent exactly 0) dominates.
    forward_check(case(260, 260, 16, 1, dtype, tau=40.0, kind="mmd", q_is_k=True))


def test_far_points_underflow_to_zero():
    q = torch.zeros(130, 8, device="cuda", dtype=torch.float16)
    k = torch.full((140, 8), 60.0, device="cuda", dtype=torch.float16)
    v = torch.ones(140, 2, device="cuda", dtype=torch.float16)
    s = _call(q, k, v, 1.0)
    assert torch.count_nonzero(s).item() == 0


def test_fp16_kernel_value_floor():
    """Kernel values below 2^-29 may be flushed (fp16 P stored with a +15
    exponent shift); the error stays below tol * den + sum of flushed terms."""
    from oracle import oracle_sum
    rng = np.random.default_rng(5)
    M, N, D = 64, 300, 4
    q = rng.standard_normal((M, D)).astype(np.float16)
    k = (rng.standard_normal((N, D)) * 3.0).astype(np.float16)
    v = rng.standard_normal((N, 1)).astype(np.float16)
    tau = 3.0
    s = _call(torch.from_numpy(q).cuda(), torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(), tau)
    ref, den = oracle_sum(q, k, v, tau)
    d2 = ((q.astype(np.float64)[:, None, :] - k.astype(np.float64)[None]) ** 2).sum(-1)
    phi = np.exp(-tau / 2 * d2)
    flushed = (phi * (phi < 2.0 ** -28) * np.abs(v.astype(np.float64)[:, 0])[None]).sum(1)
    err = np.abs(s.cpu().numpy()[:, 0] - ref[:, 0])
    assert np.all(err <= 2e-3 * den[:, 0] + flushed + 1e-30)


@pytest.mark.parametrize("dtype", ["fp16", "bf16"])
def test_norms_beyond_fp16_range(dtype):
    """Two clusters at +-40 per coordinate (D = 64): ||x - mu||^2 ~ 1e5 is
    above the fp16 range, so the folded norm terms need their range factor."""
    from oracle import oracle_sum
    rng = np.random.default_rng(11)
    M, N, D, C = 200, 333, 64, 2
    tdt = {"fp16": torch.float16, "bf16": torch.bfloat16}[dtype]
    def pts(n):
        x = rng.standard_normal((n, D)) + np.where(rng.random((n, 1)) < 0.5, -40.0, 40.0)
        return torch.from_numpy(x).to(tdt)
    q, k = pts(M), pts(N)
    v = torch.from_numpy(rng.standard_normal((N, C))).to(tdt)
    tau = 1.0 / 16
    s = _call(q.cuda(), k.cuda(), v.cuda(), tau).cpu().numpy()
    ref, den = oracle_sum(q.double().numpy(), k.double().numpy(), v.double().numpy(), tau)
    assert rel_err(s, ref, den) <= TOL[dtype]


def test_deterministic_bitwise():
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import generate
    w = case(300, 900, 64, 4, "fp16")
    q, k, v = device_inputs(generate(w))
    a = gs.gauss_sum(q, k, v, w.tau)
    b = gs.gauss_sum(q, k, v, w.tau)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_output_guards_and_prefill():
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import generate
    w = case(130, 260, 32, 3, "fp16")
    q, k, v = device_inputs(generate(w))
    guard = 1024
    buf = torch.full((guard + 130 * 3 + guard,), float("nan"), device="cuda")
    sentinel = 12345.5
    buf[:guard] = sentinel
    buf[-guard:] = sentinel
    out = buf[guard:guard + 130 * 3].view(130, 3)
    gs.gauss_sum(q, k, v, w.tau, out=out)
    gs.gauss_sum_device_status()
    assert torch.all(buf[:guard] == sentinel) and torch.all(buf[-guard:] == sentinel)
    assert not torch.isnan(out).any()


def test_empty_inputs():
    import paper_2609_04910_gb300 as gs
    q = torch.randn(5, 4, device="cuda", dtype=torch.float16)
    k = torch.randn(0, 4, device="cuda", dtype=torch.float16)
    v = torch.randn(0, 2, device="cuda", dtype=torch.float16)
    out = torch.full((5, 2), 7.0, device="cuda")
    gs.gauss_sum(q, k, v, 1.0, out=out)
    torch.cuda.synchronize()
    assert torch.count_nonzero(out).item() == 0
    q0 = torch.randn(0, 4, device="cuda", dtype=torch.float16)
    assert gs.gauss_sum(q0, q, torch.ones(5, 1, device="cuda", dtype=torch.float16), 1.0).shape == (0, 1)


def test_caller_workspace_matches_allocated():
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import generate
    w = case(200, 700, 48, 5, "fp16")
    q, k, v = device_inputs(generate(w))
    a = gs.gauss_sum(q, k, v, w.tau)
    n = gs.gauss_sum_workspace_size(200, 700, 48, 5, gs.GS_FP16)
    ws = torch.empty(n, dtype=torch.uint8, device="cuda")
    b = gs.gauss_sum(q, k, v, w.tau, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    small = torch.empty(max(n // 2, 256), dtype=torch.uint8, device="cuda")
    with pytest.raises(gs.GaussSumError) as ei:
        gs.gauss_sum(q, k, v, w.tau, workspace=small)
    assert ei.value.status == 3


def test_unsupported_shapes_raise():
    import paper_2609_04910_gb300 as gs
    q = torch.randn(4, 300, device="cuda", dtype=torch.float16)
    v = torch.ones(4, 1, device="cuda", dtype=torch.float16)
    with pytest.raises(gs.GaussSumError) as ei:
        gs.gauss_sum(q, q, v, 1.0)
    assert ei.value.status == 2


def test_forced_allocation_failure():
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300._binding import testing_fail_allocations
    q = torch.randn(4, 8, device="cuda", dtype=torch.float16)
    v = torch.ones(4, 1, device="cuda", dtype=torch.float16)
    testing_fail_allocations(True)
    try:
        with pytest.raises(gs.GaussSumError) as ei:
            gs.gauss_sum(q, q, v, 1.0)
    finally:
        testing_fail_allocations(False)
    assert ei.value.status == 3
    gs.gauss_sum(q, q, v, 1.0)
    torch.cuda.synchronize()


def test_stream_ordering_on_side_stream():
    import paper_2609_04910_gb300 as gs
    from paper_2609_04910_gb300.workloads import generate
    w = case(257, 600, 64, 2, "fp16")
    q, k, v = device_inputs(generate(w))
    ref = gs.gauss_sum(q, k, v, w.tau)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        out = gs.gauss_sum(q, k, v, w.tau)
    s.synchronize()
    assert torch.equal(out, ref)


@pytest.mark.parametrize("D,dtype", [(32, "fp32"), (24, "fp32"), (120, "fp16"), (122, "bf16"),
                                     (256, "fp16"), (200, "bf16")])
def test_long_mma_sequences_repeat_bitwise(D, dtype):
    """Long MMA sequences per key tile (3xTF32 at D = 24-32, augmented fp16 /
    bf16 rows of 128 columns with four pipeline stages, q^ in TMEM with one
    S slot at D = 200-256): repeated calls agree bit for bit and sampled rows
    match the oracle.  (An early release of the TMEM S slots once made
    single warps read overwritten S values on the two-slot path,
    nondeterministically.)"""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    from paper_2609_04910_gb300.workloads import generate, sample_rows
    w = case(16384, 16384, D, 1, dtype)
    inp = generate(w)
    q, k, v = device_inputs(inp)
    path = gs.GS_PATH_TENSOR
    outs = [gs.gauss_sum(q, k, v, w.tau, path=path) for _ in range(4)]
    gs.gauss_sum_device_status()
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    rows = sample_rows(16384, 96)
    ref, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows)
    assert rel_err(outs[0].cpu().numpy()[rows], ref, den) <= TOL[dtype]


@pytest.mark.parametrize("M,N,D,C,dtype", [(700, 140000, 256, 3, "fp16"), (300, 200000, 200, 1, "bf16")])
def test_keys_larger_than_l2_banded_order(M, N, D, C, dtype):
    """Key operands above 64 MB take the banded work order of the FMA kernel
    (all CTAs inside a few bands of 64 key tiles, one partial-sum slot per
    band): ragged rows and key tail, every row against the oracle."""
    forward_check(case(M, N, D, C, dtype))


# ---------------------------------------------------------------- exponent bound
@pytest.mark.parametrize("D,C,dtype,path", [
    (64, 1, "fp16", None),      # FMA kernel, augmented operands, value magnitudes folded
    (64, 1, "bf16", None),      # FMA kernel, augmented operands, value records
    (128, 2, "fp16", None),     # FMA kernel, q^ in TMEM, norms from A and B
    (64, 8, "fp16", None),      # two-MMA kernel (P in fp16 with the 2^15 shift)
    (48, 40, "bf16", None),     # two-MMA kernel, plain operands
    (16, 1, "fp32", "tensor"),  # 3xTF32 variant of the FMA kernel
])
def test_self_pairs_never_exceed_one(D, C, dtype, path):
    """The exponent is <= 0 in exact arithmetic (Phi <= 1, proof of Prop. 1);
    for q = k the computed self-pair exponent is only rounding, which can
    be slightly positive.  With tau large enough that every other pair
    underflows to 0, s_m = Phi(x_m, x_m) for unit values: it must lie in
    [1 - tol, 1] (the kernels clamp the exponent at 0), never above 1 --
    except with folded value magnitudes (one fp16 channel on augmented
    operands), where the exponent also carries log2(|v| 2^-16) and cannot
    be clamped at the value's own log: there s_m may exceed 1 by the
    rounding of the exponent, about c |x|^2 2^-22 relative (c = tau log2 e,
    centring off), and no more."""
    import paper_2609_04910_gb300 as gs
    w = case(300, 300, D, C, dtype, tau=200.0 / D)
    inp = generate(w)
    q, k, _ = device_inputs(inp)
    v = torch.ones((300, C), dtype=q.dtype, device="cuda")
    kw = {"path": gs.GS_PATH_TENSOR} if path == "tensor" else {}
    # Centring off: the operands keep the points' full norms, so the
    # rounding of the self-pair exponent is as large as it gets.
    s = gs.gauss_sum(q, q, v, w.tau, center=False, **kw).cpu().numpy()
    gs.gauss_sum_device_status()
    ones = np.ones((300, C))
    ref, den = oracle_sum(inp["q64"], inp["q64"], ones, w.tau)
    assert np.max(np.abs(ref - 1.0)) < 1e-10      # other pairs vanish in float64 too
    if dtype == "fp16" and C == 1 and path is None:
        c = w.tau * np.log2(np.e)
        bound = 4.0 * c * float(np.max(np.sum(inp["q64"] ** 2, axis=1))) * 2.0 ** -22
        assert np.all(s <= 1.0 + bound), f"max {s.max()!r}, bound 1 + {bound:.2e}"
    else:
        assert np.all(s <= 1.0), f"max {s.max()!r}"
    tol = TOL[dtype]
    if path == "tensor":
        # 3xTF32: the exponent carries the tf32 split error, about
        # c |x^|^2 2^-21 (c = tau log2 e); at tau = 200 / D that is above
        # the fp32 tolerance, which holds while c |x^|^2 stays below ~20.
        c = w.tau * np.log2(np.e)
        tol = c * float(np.max(np.sum(inp["q64"] ** 2, axis=1))) * 2.0 ** -20
    assert rel_err(s, ref, den) <= tol


# ---------------------------------------------------------------- FMA-pipe exp2
@pytest.mark.parametrize("share", [1, 2, 3, 4])
@pytest.mark.parametrize("M,N,D,dtype,q_is_k", [
    (300, 1000, 64, "fp16", False), (513, 700, 60, "bf16", False),
    (700, 700, 64, "fp16", True),
])
def test_exp2_on_fma_pipe_parity(share, M, N, D, dtype, q_is_k):
    """exp2_fma = 1..4 computes 1/32 .. 1/4 of the kernel values with the
    Cody-Waite + minimax-polynomial exp2 on the FMA pipe; the sums still
    match the oracle at the fp16/bf16 tolerance."""
    w = case(M, N, D, 1, dtype, kind="mmd" if q_is_k else "normal", q_is_k=q_is_k)
    forward_check(w, exp2_fma=share)


def test_exp2_on_fma_pipe_matches_mufu_closely():
    """The polynomial's relative error (< 3e-6) is far below the fp16
    tolerance: the variant agrees with the MUFU-only sums to 1e-5 of the
    oracle's scale, and far values flush to zero as with ex2.approx.ftz."""
    import paper_2609_04910_gb300 as gs
    w = case(600, 2000, 64, 1, "fp16")
    inp = generate(w)
    q, k, v = device_inputs(inp)
    a = gs.gauss_sum(q, k, v, w.tau)
    b = gs.gauss_sum(q, k, v, w.tau, exp2_fma=4)
    gs.gauss_sum_device_status()
    _, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
    assert rel_err(b.cpu().numpy(), a.cpu().numpy(), den) <= 1e-5


def test_exp2_on_fma_pipe_rejected_outside_its_range():
    import paper_2609_04910_gb300 as gs
    q = torch.randn(200, 64, device="cuda", dtype=torch.float16)
    v2 = torch.randn(200, 2, device="cuda", dtype=torch.float16)
    for args in ((q, q, v2), (q.float(), q.float(), v2[:, :1].float())):
        with pytest.raises(gs.GaussSumError) as ei:
            gs.gauss_sum(*args, 0.1, exp2_fma=2)
        assert ei.value.status == 2
        assert "exp2_fma" in ei.value.message
