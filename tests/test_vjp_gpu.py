"""GPU parity of the vector-Jacobian product of Eq. 1 (gradients of
L = sum_m g_m . s_m in q, k and v) against the float64 oracle.

Tolerance per output: |x_gpu - x_oracle| / (its error scale + 1e-30) within
the forward tolerance (2e-3 fp16/bf16, 1e-5 fp32), with the error scales of
the oracle (the terms of the per-channel Gauss sums the library evaluates,
shifted by the common mean).  Cases cover the weighted single pass
(2 <= C <= 8 weight channels, D + 1 <= 128, fp16/bf16: pair weights g_m . v_n
folded into the kernel values), its boundaries (C = 9, D = 128), one and
several channel chunks of the per-channel path (C (D + 1) above 256),
ragged row and key tails, q = k, and the degenerate sizes.
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


def _inputs(M, N, D, C, dtype, alias=False, seed=0):
    from paper_2609_04910_gb300.workloads import device_inputs, generate, upstream
    w = case(M, N, D, C, dtype)
    inp = generate(w, seed)
    q, k, v = device_inputs(inp)
    q64, k64 = inp["q64"], inp["k64"]
    if alias:
        q, q64 = k, k64
        M = N
    g = upstream(M, C, seed)
    return w, q, k, v, torch.from_numpy(g).cuda(), q64, k64, inp["v64"], g.astype(np.float64)


def _check(M, N, D, C, dtype, alias=False):
    import paper_2609_04910_gb300 as gs
    from oracle import oracle_vjp
    w, q, k, v, g, q64, k64, v64, g64 = _inputs(M, N, D, C, dtype, alias)
    gq, gk, gv = gs.gauss_sum_vjp(q, k, v, g, w.tau)
    gs.gauss_sum_device_status()
    ref = oracle_vjp(q64, k64, v64, g64, w.tau)
    tol = TOL[dtype]
    for name, got, want, den in (("grad_q", gq, ref["gq"], ref["dq"]),
                                 ("grad_k", gk, ref["gk"], ref["dk"]),
                                 ("grad_v", gv, ref["gv"], ref["dv"])):
        rel = rel_err(got.cpu().numpy(), want, den)
        assert rel <= tol, f"{name}: max rel {rel:.3e} > {tol:.1e}"


VJP_CASES = [
    # M, N, D, C, dtype
    (300, 257, 32, 1, "fp16"),     # one chunk of 33 channels
    (129, 200, 17, 3, "fp16"),     # 54 channels
    (200, 150, 64, 5, "fp16"),     # 325 channels: two chunks of 163
    (90, 130, 256, 1, "fp16"),     # 257 channels: two chunks
    (70, 300, 8, 40, "fp16"),      # 360 channels: groups split across chunks
    (150, 260, 48, 2, "bf16"),
    (64, 100, 100, 3, "bf16"),     # 303 channels: two chunks
    (100, 130, 16, 1, "fp32"),
    (70, 90, 33, 3, "fp32"),
    # weighted single pass: several row and key tiles, ragged tails
    (400, 700, 64, 4, "fp16"),     # four weight channels
    (300, 520, 32, 8, "bf16"),     # eight
    (260, 390, 127, 6, "fp16"),    # D + 1 = 128 value channels, six weights padded to eight
    (333, 300, 40, 9, "fp16"),     # nine weights: per-channel path
    (200, 300, 128, 2, "fp16"),    # D + 1 = 129: per-channel path
]


@pytest.mark.parametrize("M,N,D,C,dtype", VJP_CASES)
def test_vjp_parity(M, N, D, C, dtype):
    _check(M, N, D, C, dtype)


@pytest.mark.parametrize("dtype", ["fp16", "bf16", "fp32"])
def test_vjp_q_aliases_k(dtype):
    _check(0, 260, 24, 2, dtype, alias=True)


@pytest.mark.parametrize("dtype", ["fp16", "fp32"])
def test_vjp_q_gradient_matches_grad_q(dtype):
    """C = 1 with g = 1 is the q-gradient of Sec. 3: the same launches, so
    the results agree bit for bit."""
    import paper_2609_04910_gb300 as gs
    w, q, k, v, _, *_ = _inputs(200, 333, 20, 1, dtype)
    ones = torch.ones((200, 1), dtype=torch.float32, device="cuda")
    gq, _, _ = gs.gauss_sum_vjp(q, k, v, ones, w.tau, want=("q",))
    ref, _ = gs.gauss_sum_grad_q(q, k, v, w.tau, want_s=False)
    gs.gauss_sum_device_status()
    assert torch.equal(gq, ref)


def test_vjp_selected_outputs_match_full():
    import paper_2609_04910_gb300 as gs
    w, q, k, v, g, *_ = _inputs(150, 170, 12, 2, "fp16")
    full = gs.gauss_sum_vjp(q, k, v, g, w.tau)
    only_v = gs.gauss_sum_vjp(q, k, v, g, w.tau, want=("v",))
    only_q = gs.gauss_sum_vjp(q, k, v, g, w.tau, want=("q",))
    gs.gauss_sum_device_status()
    assert only_v[0] is None and only_v[1] is None
    assert torch.equal(only_v[2], full[2])
    assert torch.equal(only_q[0], full[0])


@pytest.mark.parametrize("dtype", ["fp16", "fp32"])
def test_vjp_degenerate_sizes(dtype):
    """D = 0 (Phi = 1: grad_v[n] = sum_m g_m), C = 0 (L = 0), N = 0 and M = 0."""
    import paper_2609_04910_gb300 as gs
    tdt = {"fp16": torch.float16, "fp32": torch.float32}[dtype]
    dev = "cuda"
    g = torch.randn(6, 3, device=dev)
    q = torch.zeros((6, 0), dtype=tdt, device=dev)
    k = torch.zeros((5, 0), dtype=tdt, device=dev)
    v = torch.randn(5, 3, device=dev).to(tdt)
    gq, gk, gv = gs.gauss_sum_vjp(q, k, v, g, 0.5)
    gs.gauss_sum_device_status()
    assert gq.shape == (6, 0) and gk.shape == (5, 0)
    want = g.double().sum(0).cpu().numpy()
    got = gv.cpu().numpy()
    scale = g.abs().double().sum(0).cpu().numpy()
    assert np.all(np.abs(got - want) <= TOL[dtype] * scale)

    q = torch.randn(6, 4, device=dev).to(tdt)
    k = torch.randn(5, 4, device=dev).to(tdt)
    gq = torch.full((6, 4), 7.0, device=dev)
    gk = torch.full((5, 4), 7.0, device=dev)
    v0 = torch.zeros((5, 0), dtype=tdt, device=dev)
    g0 = torch.zeros((6, 0), device=dev)
    gs.gauss_sum_vjp(q, k, v0, g0, 0.5, grad_q=gq, grad_k=gk)
    gs.gauss_sum_device_status()
    assert torch.count_nonzero(gq).item() == 0 and torch.count_nonzero(gk).item() == 0

    kN = torch.zeros((0, 4), dtype=tdt, device=dev)
    vN = torch.zeros((0, 2), dtype=tdt, device=dev)
    gq = torch.full((6, 4), 7.0, device=dev)
    out = gs.gauss_sum_vjp(q, kN, vN, torch.randn(6, 2, device=dev), 0.5, grad_q=gq)
    gs.gauss_sum_device_status()
    assert torch.count_nonzero(gq).item() == 0 and out[1].shape == (0, 4)

    qM = torch.zeros((0, 4), dtype=tdt, device=dev)
    gk = torch.full((5, 4), 7.0, device=dev)
    gv = torch.full((5, 2), 7.0, device=dev)
    gs.gauss_sum_vjp(qM, k, torch.randn(5, 2, device=dev).to(tdt), torch.zeros((0, 2), device=dev),
                     0.5, grad_k=gk, grad_v=gv)
    gs.gauss_sum_device_status()
    assert torch.count_nonzero(gk).item() == 0 and torch.count_nonzero(gv).item() == 0
