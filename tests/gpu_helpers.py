"""Shared helpers of the GPU parity tests: move seeded inputs to the device,
call the library through its C ABI, and compare with the float64 oracle."""
import numpy as np

from oracle import oracle_grad_q, oracle_sum
from paper_2609_04910_gb300.workloads import Workload, device_inputs, generate, to_device  # noqa: F401

TOL = {"fp32": 1e-5, "fp16": 2e-3, "bf16": 2e-3}


def rel_err(got, ref, den):
    return float(np.max(np.abs(got - ref) / (den + 1e-30))) if got.size else 0.0


def case(M, N, D, C, dtype, tau=None, kind="normal", q_is_k=False):
    return Workload(f"case_{M}x{N}x{D}x{C}_{dtype}", M, N, D, C, dtype,
                    tau if tau is not None else 1.0 / max(D, 1), kind, q_is_k=q_is_k)


def forward_check(w, seed=0, rows=None, tol=None, **kw):
    import paper_2609_04910_gb300 as gs
    inp = generate(w, seed)
    q, k, v = device_inputs(inp)
    s = gs.gauss_sum(q, k, v, w.tau, **kw)
    gs.gauss_sum_device_status()
    got = s.cpu().numpy()
    ref, den = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows)
    if rows is not None:
        got = got[rows]
    rel = rel_err(got, ref, den)
    limit = TOL[w.dtype] if tol is None else tol
    assert rel <= limit, f"{w.name}: max rel {rel:.3e} > {limit:.1e}"
    return rel, got, ref, den


def grad_check(w, seed=0, rows=None, tol=None, **kw):
    import paper_2609_04910_gb300 as gs
    inp = generate(w, seed)
    q, k, v = device_inputs(inp)
    g, s = gs.gauss_sum_grad_q(q, k, v, w.tau, **kw)
    gs.gauss_sum_device_status()
    g = g.cpu().numpy()
    s = s.cpu().numpy()
    gref, sref, gden, _ = oracle_grad_q(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows)
    _, sden = oracle_sum(inp["q64"], inp["k64"], inp["v64"], w.tau, rows=rows)
    if rows is not None:
        g = g[rows]
        s = s[rows]
    limit = TOL[w.dtype] if tol is None else tol
    relg = rel_err(g, gref, gden)
    rels = rel_err(s, sref, sden[:, 0])
    assert relg <= limit, f"{w.name}: grad max rel {relg:.3e} > {limit:.1e}"
    assert rels <= limit, f"{w.name}: s max rel {rels:.3e} > {limit:.1e}"
    return relg, rels
