"""GPU parity of the batched Gauss sum and of the squared MMD (Sec. 3).

Every problem of a batch is checked against the float64 oracle on its own
points, with the tolerance of the single-problem tests.  The batch covers
the one-launch path (C <= 4 on fp16/bf16, with and without augmented
operands) and the paths that run the problems one after another (C > 4,
fp32).
"""
import numpy as np
import pytest

from tests.gpu_helpers import TOL, case, rel_err

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_04910_gb300.build import build_library
    build_library()
    torch.cuda.set_device(0)


def _stacked(B, M, N, D, C, dtype, q_is_k=False, kind="normal"):
    """B seeded problems (seeds 0..B-1) of the workload recipe, stacked."""
    from paper_2609_04910_gb300.workloads import generate, to_device
    w = case(M, N, D, C, dtype, kind=kind, q_is_k=q_is_k)
    inps = [generate(w, seed=b) for b in range(B)]
    qs = torch.stack([to_device(i["q"], dtype) for i in inps]).contiguous()
    ks = qs if q_is_k else torch.stack([to_device(i["k"], dtype) for i in inps]).contiguous()
    vs = torch.stack([to_device(i["v"], dtype) for i in inps]).contiguous()
    return w, inps, qs, ks, vs


def _check_batched(B, M, N, D, C, dtype, q_is_k=False, kind="normal"):
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_sum
    w, inps, q, k, v = _stacked(B, M, N, D, C, dtype, q_is_k, kind)
    out = gs.gauss_sum_batched(q, k, v, w.tau)
    gs.gauss_sum_device_status()
    got = out.cpu().numpy()
    for b, inp in enumerate(inps):
        ref, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau)
        rel = rel_err(got[b], ref, den)
        assert rel <= TOL[dtype], f"problem {b}: max rel {rel:.3e}"


@pytest.mark.parametrize("B,M,N,D,C,dtype", [
    (3, 200, 333, 64, 2, "fp16"),     # one launch, augmented operands
    (2, 300, 130, 17, 1, "bf16"),     # one launch, ragged sizes
    (2, 70, 400, 200, 3, "fp16"),     # one launch, q^ in TMEM (no augmented operands)
    (2, 150, 260, 32, 8, "fp16"),     # C > 4: one problem after another
    (3, 90, 110, 16, 2, "fp32"),      # small fp32 problems: SIMT, one after another
    (8, 2048, 2100, 16, 1, "fp32"),   # fp32 tensor-core path: one launch for the batch
])
def test_batched_matches_each_problem(B, M, N, D, C, dtype):
    _check_batched(B, M, N, D, C, dtype)


def test_batched_q_is_k():
    # The MMD recipe draws one point set per problem (q = k).
    _check_batched(2, 300, 300, 32, 1, "fp16", q_is_k=True, kind="mmd")


def test_batched_empty_and_no_keys():
    import paper_2609_04910_gb300 as gs
    q = torch.zeros((0, 10, 8), dtype=torch.float16, device="cuda")
    v = torch.zeros((0, 12, 1), dtype=torch.float16, device="cuda")
    k = torch.zeros((0, 12, 8), dtype=torch.float16, device="cuda")
    assert gs.gauss_sum_batched(q, k, v, 1.0).shape == (0, 10, 1)
    q = torch.randn((2, 10, 8), device="cuda").half()
    k = torch.zeros((2, 0, 8), dtype=torch.float16, device="cuda")
    v = torch.zeros((2, 0, 3), dtype=torch.float16, device="cuda")
    out = torch.full((2, 10, 3), float("nan"), device="cuda")
    gs.gauss_sum_batched(q, k, v, 1.0, out=out)
    assert torch.count_nonzero(out).item() == 0


@pytest.mark.parametrize("dtype", ["fp16", "bf16", "fp32"])
def test_mmd2_matches_oracle(dtype):
    """mmd2[b] = v_b^T s_b for the two-sample weights (+1/n, -1/n) of the
    MMD workload; error bound: tolerance x sum_m |v_m| sum_n Phi |v_n|."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_mmd2
    B, N, D = 3, 600, 16
    w, inps, x, _, v = _stacked(B, N, N, D, 1, dtype, q_is_k=True, kind="mmd")
    got = gs.gauss_sum_mmd2(x, v[..., 0].contiguous(), w.tau).cpu().numpy()
    gs.gauss_sum_device_status()
    for b, inp in enumerate(inps):
        ref, den = oracle_mmd2(inp["q64"], inp["v64"][:, 0], w.tau)
        assert abs(got[b] - ref) <= TOL[dtype] * den + 1e-30, (b, got[b], ref, den)


def test_mmd2_of_equal_samples_vanishes():
    """Two equal samples: MMD^2 = 0 up to the computed sums' error."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_mmd2
    rng = np.random.default_rng(9)
    a = rng.standard_normal((300, 24)).astype(np.float16)
    x = np.concatenate([a, a])
    v = np.concatenate([np.full(300, 1 / 300), np.full(300, -1 / 300)]).astype(np.float16)
    got = gs.gauss_sum_mmd2(torch.from_numpy(x).cuda(), torch.from_numpy(v).cuda(), 1 / 24)
    gs.gauss_sum_device_status()
    _, den = oracle_mmd2(x.astype(np.float64), v.astype(np.float64), 1 / 24)
    assert abs(float(got[0])) <= TOL["fp16"] * den


@pytest.mark.parametrize("B,N,D,dtype", [
    (1, 20000, 64, "fp16"),   # one problem, many CTAs per pair of query tiles
    (5, 3000, 32, "fp16"),    # CTA runs crossing pairs and problems, ragged N
    (4, 2100, 100, "bf16"),   # bf16 augmented operands (three norm terms)
    (2, 1000, 125, "fp16"),   # no augmented operands: the full sum K v is used
])
def test_mmd2_upper_triangle(B, N, D, dtype):
    """MMD^2 over the upper triangle of tile pairs (K symmetric, off-diagonal
    tiles counted twice) against the oracle and against v^T (K v) from the
    full Gauss sum."""
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_mmd2
    w, inps, x, _, v = _stacked(B, N, N, D, 1, dtype, q_is_k=True, kind="mmd")
    v1 = v[..., 0].contiguous()
    got = gs.gauss_sum_mmd2(x, v1, w.tau).cpu().numpy().astype(np.float64)
    full = gs.gauss_sum_batched(x, x, v, w.tau)
    gs.gauss_sum_device_status()
    vt_s = (v1.double() * full[..., 0].double()).sum(dim=1).cpu().numpy()
    for b, inp in enumerate(inps):
        ref, den = oracle_mmd2(inp["q64"], inp["v64"][:, 0], w.tau)
        assert abs(got[b] - ref) <= TOL[dtype] * den + 1e-30, (b, got[b], ref, den)
        assert abs(got[b] - vt_s[b]) <= 2 * TOL[dtype] * den + 1e-30, (b, got[b], vt_s[b], den)
