"""The oracle's pins are strong enough to catch plausible mistakes.

Each case plants one mistake in a temporary copy of ``oracle/gauss_oracle.c``
(a dropped factor, a flipped sign, a dropped term, a wrong index or stride),
compiles it on the CPU, and checks that at least one pin rejects it.  The
committed oracle is never modified.
"""
import math
import os

import numpy as np
import pytest

from oracle import build_oracle, oracle_grad_q, oracle_sum, oracle_vjp
from tests.paper_forms import prescale

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle",
                   "gauss_oracle.c")

MUTANTS = {
    "dropped_half": ("exp(-0.5 * tau * sq_dist(a, b, D))", "exp(-tau * sq_dist(a, b, D))"),
    "sign_of_difference": ("double t = a[d] - b[d];", "double t = a[d] + b[d];"),
    "dropped_coordinate": ("for (int64_t d = 0; d < D; ++d) {\n        double t",
                           "for (int64_t d = 0; d < D - 1; ++d) {\n        double t"),
    "channel_index": ("sr[c] += phi * vn[c];", "sr[c] += phi * vn[0];"),
    "value_stride": ("D, tau);\n            const double* vn = v + n * C;",
                     "D, tau);\n            const double* vn = v + n;"),
    "row_index": ("const double* qm = q + m * D;\n        double* sr",
                  "const double* qm = q + r * D;\n        double* sr"),
    "grad_sign": ("gr[d] += w * (kn[d] - qm[d]);", "gr[d] += w * (qm[d] - kn[d]);"),
    "grad_factor": ("gr[d] *= tau;", "gr[d] *= 0.5 * tau;"),
    "transposed_key": ("double phi = gauss_kernel(qm, k + n * D, D, tau);",
                       "double phi = gauss_kernel(qm, k + n, D, tau);"),
    "vjp_k_sign": ("outk[d] += phi * w * (qm[d] - kn[d]);", "outk[d] += phi * w * (kn[d] - qm[d]);"),
    "vjp_v_upstream": ("if (outv) outv[c] += phi * gm[c];", "if (outv) outv[c] += phi * vn[c];"),
    "vjp_q_contraction": ("w += gm[c] * vn[c];", "w += gm[0] * vn[c];"),
    "vjp_k_contraction": ("w += vn[c] * gm[c];", "w += vn[c] * gm[c] * (c == 0);"),
    "vjp_q_factor": ("if (out) out[d] *= tau;", "if (out) out[d] *= 0.5 * tau;"),
    # The error scales of the VJP (the denominators of its parity bar).
    "vjp_dq_signed_upstream": (
        "e += fabs(gm[c]) * (a[c * Dm + d] + fabs(qm[d] - mu[d]) * b[c]);",
        "e += gm[c] * (a[c * Dm + d] + fabs(qm[d] - mu[d]) * b[c]);"),
    "vjp_dq_first_channel": (
        "e += fabs(gm[c]) * (a[c * Dm + d] + fabs(qm[d] - mu[d]) * b[c]);",
        "e += fabs(gm[0]) * (a[c * Dm + d] + fabs(qm[d] - mu[d]) * b[c]);"),
    "vjp_dk_dropped_shift_term": (
        "e += fabs(vn[c]) * (a[c * Dm + d] + fabs(kn[d] - mu[d]) * b[c]);",
        "e += fabs(vn[c]) * a[c * Dm + d];"),
    "vjp_dk_unweighted_abs": (
        "a[c * Dm + d] += pg * fabs(qm[d] - mu[d]);",
        "a[c * Dm + d] += pg * (qm[d] - mu[d]);"),
    "vjp_dv_signed_accumulation": ("const double pg = phi * fabs(gm[c]);",
                                   "const double pg = phi * gm[c];"),
    "vjp_dv_channel": ("dv[r * C + c] = b[c];", "dv[r * C + c] = b[0];"),
    "vjp_dq_value_magnitude": ("const double pv = phi * fabs(vn[c]);",
                               "const double pv = phi * vn[c];"),
}


def _pin_failures(lib):
    """Run a fast subset of the pins against the library at ``lib``."""
    fails = []
    rng = np.random.default_rng(0)
    # single key closed form, D=3, C=2
    q = rng.standard_normal((3, 3))
    k = rng.standard_normal((1, 3))
    v = rng.standard_normal((1, 2))
    s, _ = oracle_sum(q, k, v, 0.7, lib_path=lib)
    for m in range(3):
        want = math.exp(-0.35 * math.fsum((q[m] - k[0]) ** 2)) * v[0]
        if not np.allclose(s[m], want, rtol=1e-12, atol=0):
            fails.append("single_key")
            break
    # Alg. 1 route, multi-channel
    q = rng.standard_normal((6, 4))
    k = rng.standard_normal((9, 4))
    v = rng.standard_normal((9, 3))
    s, den = oracle_sum(q, k, v, 0.5, lib_path=lib)
    if np.max(np.abs(prescale(q, k, v, 0.5) - s) / den) > 1e-10:
        fails.append("alg1")
    # row subset equals full evaluation
    sub, _ = oracle_sum(q, k, v, 0.5, rows=[5, 1], lib_path=lib)
    if not np.array_equal(sub, s[[5, 1]]):
        fails.append("row_subset")
    # gradient vs finite differences
    q = rng.standard_normal((2, 3))
    k = rng.standard_normal((8, 3))
    v = rng.standard_normal(8)
    g, _, _, _ = oracle_grad_q(q, k, v, 0.9, lib_path=lib)
    h = 1e-6
    for d in range(3):
        qp = q[:1].copy(); qp[0, d] += h
        qm = q[:1].copy(); qm[0, d] -= h
        fd = (oracle_sum(qp, k, v[:, None], 0.9, lib_path=lib)[0][0, 0]
              - oracle_sum(qm, k, v[:, None], 0.9, lib_path=lib)[0][0, 0]) / (2 * h)
        if abs(fd - g[0, d]) > 1e-6 * (1 + abs(fd)):
            fails.append("grad_fd")
            break
    # vector-Jacobian product vs finite differences of sum_m g_m . s_m
    q = rng.standard_normal((3, 2))
    k = rng.standard_normal((4, 2))
    v = rng.standard_normal((4, 2))
    up = rng.standard_normal((3, 2))
    r = oracle_vjp(q, k, v, up, 0.8, lib_path=lib)

    def loss(qq, kk, vv):
        return float(np.sum(up * oracle_sum(qq, kk, vv, 0.8, lib_path=lib)[0]))

    for arr, got, which in ((q, r["gq"], 0), (k, r["gk"], 1), (v, r["gv"], 2)):
        for idx in np.ndindex(arr.shape):
            args_p = [q.copy(), k.copy(), v.copy()]
            args_m = [q.copy(), k.copy(), v.copy()]
            args_p[which][idx] += h
            args_m[which][idx] -= h
            fd = (loss(*args_p) - loss(*args_m)) / (2 * h)
            if abs(fd - got[idx]) > 1e-6 * (1 + abs(fd)):
                fails.append(f"vjp_fd_{which}")
                break
    # VJP error scales (C = 2, signed non-unit upstream g) against the
    # scales of the q-gradient and forward oracles, contracted per channel.
    q = rng.standard_normal((3, 2)) + 1.0
    k = rng.standard_normal((4, 2)) - 0.5
    v = rng.standard_normal((4, 2)) * np.array([1.0, -2.0])
    up = rng.standard_normal((3, 2)) * np.array([-1.5, 0.5])
    r = oracle_vjp(q, k, v, up, 0.8, lib_path=lib)
    dq = sum(np.abs(up[:, c:c + 1]) * oracle_grad_q(q, k, v[:, c], 0.8, lib_path=lib)[2]
             for c in range(2))
    dk = sum(np.abs(v[:, c:c + 1]) * oracle_grad_q(k, q, up[:, c], 0.8, lib_path=lib)[2]
             for c in range(2))
    dv = oracle_sum(k, q, up, 0.8, lib_path=lib)[1]
    for name, got, want in (("dq", r["dq"], dq), ("dk", r["dk"], dk), ("dv", r["dv"], dv)):
        if not np.allclose(got, want, rtol=1e-12, atol=0):
            fails.append(f"vjp_scale_{name}")
    return fails


def test_committed_oracle_passes_fast_pins():
    assert _pin_failures(None) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique"
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    lib = build_oracle(src=str(mutated), out=str(tmp_path / "libmutant.so"), force=True)
    assert _pin_failures(lib), f"no pin caught the planted mistake {name}"
