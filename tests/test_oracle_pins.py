"""Pins of the float64 oracle against facts fixed by the paper and by mathematics.

None of these checks re-evaluates the oracle's own formula: each compares it
with a closed form, a symmetry, an independent algebraic route (Alg. 1,
Alg. 2), finite differences, a Monte-Carlo expectation or brute force.
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import oracle_grad_q, oracle_sum
from tests.paper_forms import prescale, reweight

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rel(a, b, den):
    return float(np.max(np.abs(a - b) / (den + 1e-300)))


# ---------------------------------------------------------------- closed forms
def test_worked_example_d1():
    """D=1, q=0, k=1, tau=2: Phi = exp(-1) (Sec. 1 definition)."""
    s, den = oracle_sum(np.zeros((1, 1)), np.ones((1, 1)), np.ones((1, 1)), 2.0)
    assert s[0, 0] == pytest.approx(math.exp(-1.0), rel=1e-15)
    assert den[0, 0] == pytest.approx(math.exp(-1.0), rel=1e-15)


def test_single_key_closed_form():
    """N=1: s_m = exp(-tau/2 ||q_m - k||^2) v (Eq. 1 with one term)."""
    rng = np.random.default_rng(3)
    q = rng.standard_normal((5, 7))
    k = rng.standard_normal((1, 7))
    v = rng.standard_normal((1, 3))
    tau = 0.37
    s, _ = oracle_sum(q, k, v, tau)
    for m in range(5):
        d2 = math.fsum((q[m, d] - k[0, d]) ** 2 for d in range(7))
        want = math.exp(-tau * d2 / 2.0) * v[0]
        np.testing.assert_allclose(s[m], want, rtol=1e-14, atol=0)


def test_tau_to_zero_gives_plain_sum():
    """tau -> 0: Phi -> 1, so s_m = sum_n v_n for every m."""
    rng = np.random.default_rng(4)
    q = rng.standard_normal((6, 4))
    k = rng.standard_normal((50, 4))
    v = rng.standard_normal((50, 2))
    s, den = oracle_sum(q, k, v, 1e-30)
    want = np.array([math.fsum(v[:, c]) for c in range(2)])
    np.testing.assert_allclose(s, np.broadcast_to(want, s.shape), rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(den, np.broadcast_to(np.abs(v).sum(0), den.shape), rtol=1e-13)


def test_identical_keys():
    """k_n = k for all n: s_m = Phi(q_m, k) sum_n v_n."""
    rng = np.random.default_rng(5)
    q = rng.standard_normal((4, 3))
    k1 = rng.standard_normal(3)
    k = np.tile(k1, (9, 1))
    v = rng.standard_normal((9, 1))
    tau = 1.3
    s, _ = oracle_sum(q, k, v, tau)
    for m in range(4):
        phi = math.exp(-tau / 2 * math.fsum((q[m] - k1) ** 2))
        assert s[m, 0] == pytest.approx(phi * math.fsum(v[:, 0]), rel=1e-13)


def test_separable_lattice_factorises():
    """Keys on a product grid G^D with unit weights: the Gauss kernel
    factorises over coordinates, so s(q) = prod_d sum_{g in G} exp(-tau/2 (q_d - g)^2).
    A dropped coordinate, a wrong index or a wrong factor breaks the product."""
    G = np.array([-1.5, -0.2, 0.4, 1.1])
    D = 3
    grid = np.array(np.meshgrid(*([G] * D), indexing="ij")).reshape(D, -1).T
    rng = np.random.default_rng(6)
    q = rng.standard_normal((5, D))
    tau = 0.8
    s, _ = oracle_sum(q, grid, np.ones((grid.shape[0], 1)), tau)
    for m in range(5):
        want = 1.0
        for d in range(D):
            want *= math.fsum(math.exp(-tau / 2 * (q[m, d] - g) ** 2) for g in G)
        assert s[m, 0] == pytest.approx(want, rel=1e-13)


# ---------------------------------------------------------------- symmetry
def test_kernel_matrix_symmetry():
    """Phi(q,k) = Phi(k,q): with one-hot values the oracle returns the kernel
    matrix, and swapping the roles of q and k transposes it."""
    rng = np.random.default_rng(7)
    q = rng.standard_normal((6, 4))
    k = rng.standard_normal((9, 4))
    Kqk, _ = oracle_sum(q, k, np.eye(9), 0.6)
    Kkq, _ = oracle_sum(k, q, np.eye(6), 0.6)
    np.testing.assert_allclose(Kqk, Kkq.T, rtol=1e-14, atol=0)
    assert np.all(Kqk > 0) and np.all(Kqk <= 1.0)


def test_unit_weight_total_symmetry():
    """M = N, C = 1, unit weights: 1^T s(q,k) = 1^T s(k,q)."""
    rng = np.random.default_rng(8)
    q = rng.standard_normal((40, 5))
    k = rng.standard_normal((40, 5))
    a, _ = oracle_sum(q, k, np.ones((40, 1)), 0.9)
    b, _ = oracle_sum(k, q, np.ones((40, 1)), 0.9)
    assert math.fsum(a[:, 0]) == pytest.approx(math.fsum(b[:, 0]), rel=1e-13)


# ---------------------------------------------------------------- algebraic routes
@pytest.mark.parametrize("M,N,D,C,tau", [(7, 11, 3, 1, 1.0), (16, 40, 8, 5, 0.25),
                                         (5, 64, 32, 3, 1.0 / 32), (9, 13, 1, 2, 3.0)])
def test_alg1_prescale_matches(M, N, D, C, tau):
    """Alg. 1: Att(q,k,v~) exp(lse) exp(-tau/2||q||^2) with v~ = v exp(-tau/2||k||^2)."""
    rng = np.random.default_rng(M * 1000 + N)
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, C))
    s, den = oracle_sum(q, k, v, tau)
    assert _rel(prescale(q, k, v, tau), s, den) < 1e-10


@pytest.mark.parametrize("M,N,D,C,tau", [(7, 11, 3, 1, 1.0), (16, 40, 8, 5, 0.25),
                                         (5, 64, 32, 3, 1.0 / 32), (9, 13, 1, 2, 3.0)])
def test_alg2_reweight_and_prop1(M, N, D, C, tau):
    """Alg. 2 reproduces the sum, and Prop. 1's bounds hold:
    kappa/(N+1) <= beta_m <= kappa and ||alpha_m||_inf <= max_n ||v_n||_inf."""
    rng = np.random.default_rng(M * 7 + N)
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, C))
    s_rw, alpha, beta, kappa = reweight(q, k, v, tau, return_parts=True)
    s, den = oracle_sum(q, k, v, tau)
    assert _rel(s_rw, s, den) < 1e-10
    assert np.all(beta <= kappa * (1 + 1e-14))
    assert np.all(beta >= kappa / (N + 1) * (1 - 1e-14))
    assert np.max(np.abs(alpha)) <= np.max(np.abs(v)) * (1 + 1e-14)
    # The proof's closed form: beta_m = kappa / (1 + sum_n Phi(q_m, k_n)).
    ones, _ = oracle_sum(q, k, np.ones((N, 1)), tau)
    np.testing.assert_allclose(beta, kappa / (1.0 + ones[:, 0]), rtol=1e-12)


# ---------------------------------------------------------------- gradient
def test_gradient_matches_finite_differences():
    """Sec. 3 q-gradient vs central differences of the oracle's own s."""
    rng = np.random.default_rng(9)
    M, N, D = 4, 30, 5
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, 1))
    tau = 0.7
    g, s, den, dsh = oracle_grad_q(q, k, v, tau)
    s_ref, _ = oracle_sum(q, k, v, tau)
    np.testing.assert_allclose(s, s_ref[:, 0], rtol=1e-14)
    h = 1e-6
    for m in range(M):
        for d in range(D):
            qp = q.copy(); qp[m, d] += h
            qm = q.copy(); qm[m, d] -= h
            sp, _ = oracle_sum(qp[m:m + 1], k, v, tau)
            sm, _ = oracle_sum(qm[m:m + 1], k, v, tau)
            fd = (sp[0, 0] - sm[0, 0]) / (2 * h)
            assert abs(fd - g[m, d]) <= 1e-7 * (1 + abs(g[m, d]))
    assert np.all(dsh >= np.abs(g) * (1 - 1e-12))


def test_gradient_error_scale_definition():
    """den of the gradient is tau(sum Phi|v||k_d-mu_d| + |q_d-mu_d| sum Phi|v|)
    with mu the mean of all points; checked by brute force."""
    rng = np.random.default_rng(10)
    q = rng.standard_normal((3, 2)) + 2.0
    k = rng.standard_normal((4, 2)) - 1.0
    v = rng.standard_normal(4)
    tau = 0.5
    g, s, den, dsh = oracle_grad_q(q, k, v, tau)
    mu = np.concatenate([q, k]).mean(0)
    for m in range(3):
        phi = [math.exp(-tau / 2 * math.fsum((q[m] - k[n]) ** 2)) for n in range(4)]
        absw = math.fsum(phi[n] * abs(v[n]) for n in range(4))
        for d in range(2):
            want = tau * (math.fsum(phi[n] * abs(v[n]) * abs(k[n, d] - mu[d]) for n in range(4))
                          + abs(q[m, d] - mu[d]) * absw)
            assert den[m, d] == pytest.approx(want, rel=1e-13)
            gw = tau * math.fsum(phi[n] * v[n] * (k[n, d] - q[m, d]) for n in range(4))
            assert g[m, d] == pytest.approx(gw, rel=1e-12, abs=1e-15)


def test_gradient_as_augmented_gauss_sum():
    """Sec. 3: the gradient is one Gauss sum with values (v_n k_n, v_n):
    g = tau (S[:D] - q_m S[D])."""
    rng = np.random.default_rng(11)
    q = rng.standard_normal((5, 3))
    k = rng.standard_normal((20, 3))
    v = rng.standard_normal(20)
    tau = 1.1
    g, s, _, _ = oracle_grad_q(q, k, v, tau)
    aug = np.concatenate([v[:, None] * k, v[:, None]], axis=1)
    S, _ = oracle_sum(q, k, aug, tau)
    want = tau * (S[:, :3] - q * S[:, 3:4])
    np.testing.assert_allclose(g, want, rtol=1e-10, atol=1e-13)


# ---------------------------------------------------------------- MMD invariants
def test_mmd_nonnegative_and_zero_for_equal_samples():
    """Sec. 3: MMD^2 = sum_m v_m s_m with q = k is >= 0 (positive-definite
    kernel) and is 0 when the two signed halves sit on the same points."""
    rng = np.random.default_rng(12)
    X = rng.standard_normal((30, 4))
    v = np.concatenate([np.full(15, 1 / 15), np.full(15, -1 / 15)])[:, None]
    s, _ = oracle_sum(X, X, v, 0.5)
    assert float(v[:, 0] @ s[:, 0]) > 0
    Y = np.concatenate([X[:15], X[:15]])
    s2, den2 = oracle_sum(Y, Y, v, 0.5)
    assert abs(float(v[:, 0] @ s2[:, 0])) < 1e-15
    assert np.max(np.abs(s2)) < 1e-15


# ---------------------------------------------------------------- statistics
def test_gaussian_expectation_monte_carlo():
    """For k ~ N(0, sigma^2 I_D): E Phi(q, k) = (1+tau sigma^2)^(-D/2)
    exp(-tau ||q||^2 / (2 (1 + tau sigma^2))).  The oracle's mean over many
    keys must agree within Monte-Carlo error."""
    rng = np.random.default_rng(13)
    D, N, sigma, tau = 3, 200000, 0.8, 1.2
    q = np.array([[0.3, -0.5, 0.9], [0.0, 0.0, 0.0]])
    k = sigma * rng.standard_normal((N, D))
    ones = np.ones((N, 1))
    s, _ = oracle_sum(q, k, ones, tau, nthreads=2)
    a = 1.0 + tau * sigma ** 2
    for m in range(2):
        want = a ** (-D / 2) * math.exp(-tau * float(q[m] @ q[m]) / (2 * a))
        # Phi in (0, 1]; its standard deviation is below 0.5.
        assert abs(s[m, 0] / N - want) < 5 * 0.5 / math.sqrt(N)


# ---------------------------------------------------------------- brute force
def test_brute_force_tiny():
    """Tiny inputs expanded by hand with math.exp / math.fsum."""
    rng = np.random.default_rng(14)
    for M, N, D, C in [(1, 1, 1, 1), (2, 3, 2, 1), (4, 4, 3, 2), (3, 2, 1, 3)]:
        q = rng.standard_normal((M, D))
        k = rng.standard_normal((N, D))
        v = rng.standard_normal((N, C))
        tau = float(rng.uniform(0.1, 2.0))
        s, den = oracle_sum(q, k, v, tau)
        for m in range(M):
            for c in range(C):
                terms = []
                absterms = []
                for n in range(N):
                    if D == 1:
                        d2 = (q[m, 0] - k[n, 0]) ** 2
                    elif D == 2:
                        d2 = (q[m, 0] - k[n, 0]) ** 2 + (q[m, 1] - k[n, 1]) ** 2
                    else:
                        d2 = ((q[m, 0] - k[n, 0]) ** 2 + (q[m, 1] - k[n, 1]) ** 2
                              + (q[m, 2] - k[n, 2]) ** 2)
                    terms.append(math.exp(-0.5 * tau * d2) * v[n, c])
                    absterms.append(math.exp(-0.5 * tau * d2) * abs(v[n, c]))
                assert abs(s[m, c] - math.fsum(terms)) <= 1e-14 * (1 + math.fsum(absterms))
                assert den[m, c] == pytest.approx(math.fsum(absterms), rel=1e-14)


# ---------------------------------------------------------------- golden values
def test_golden_fixtures():
    """Small hand-checkable fixtures stored under tests/golden/, each with the
    passage it follows; expected values are closed forms written out there."""
    with open(os.path.join(GOLDEN, "closed_forms.json")) as f:
        cases = json.load(f)
    assert len(cases) >= 3
    for case in cases:
        q = np.array(case["q"], dtype=np.float64)
        k = np.array(case["k"], dtype=np.float64)
        v = np.array(case["v"], dtype=np.float64)
        s, _ = oracle_sum(q, k, v, case["tau"])
        np.testing.assert_allclose(s, np.array(case["s"]), rtol=1e-13, atol=1e-300,
                                   err_msg=case["cite"])


# ---------------------------------------------------------------- plumbing
def test_row_subset_and_thread_count_invariance():
    rng = np.random.default_rng(15)
    q = rng.standard_normal((50, 6))
    k = rng.standard_normal((70, 6))
    v = rng.standard_normal((70, 2))
    full, fden = oracle_sum(q, k, v, 0.4, nthreads=1)
    rows = np.array([49, 0, 17, 17, 3])
    sub, sden = oracle_sum(q, k, v, 0.4, rows=rows, nthreads=3)
    np.testing.assert_array_equal(sub, full[rows])
    np.testing.assert_array_equal(sden, fden[rows])
    full4, _ = oracle_sum(q, k, v, 0.4, nthreads=4)
    np.testing.assert_array_equal(full4, full)


def test_empty_and_rejected_inputs():
    s, den = oracle_sum(np.zeros((3, 2)), np.zeros((0, 2)), np.zeros((0, 1)), 1.0)
    assert np.all(s == 0) and s.shape == (3, 1)
    with pytest.raises(ValueError):
        oracle_sum(np.zeros((3, 2)), np.zeros((4, 2)), np.zeros((4, 1)), 1.0, rows=[3])


# ---------------------------------------------------------------- MMD^2 (Sec. 3)
def test_mmd2_brute_force_double_sum():
    """oracle_mmd2 equals sum_{m,n} v_m exp(-tau/2 ||x_m - x_n||^2) v_n
    written out with math.exp and math.fsum on a tiny case."""
    from oracle import oracle_mmd2
    rng = np.random.default_rng(21)
    x = rng.standard_normal((5, 3))
    v = np.array([0.4, -0.1, 0.3, -0.35, -0.25])
    tau = 0.7
    terms = []
    for m in range(5):
        for n in range(5):
            d2 = sum((x[m, d] - x[n, d]) ** 2 for d in range(3))
            terms.append(v[m] * math.exp(-tau / 2 * d2) * v[n])
    got, den = oracle_mmd2(x, v, tau)
    assert got == pytest.approx(math.fsum(terms), rel=1e-13, abs=1e-15)
    assert den >= abs(got)


def test_mmd2_zero_for_equal_samples_and_positive_otherwise():
    """MMD^2 of two equal samples (weights +1/n on one copy, -1/n on the
    other) is 0; for different samples it is > 0 (positive definite kernel)."""
    from oracle import oracle_mmd2
    rng = np.random.default_rng(22)
    a = rng.standard_normal((40, 4))
    v = np.concatenate([np.full(40, 1 / 40), np.full(40, -1 / 40)])
    same, den = oracle_mmd2(np.concatenate([a, a]), v, 0.5)
    assert abs(same) <= 1e-14 * den
    b = rng.standard_normal((40, 4)) + 0.5
    diff, _ = oracle_mmd2(np.concatenate([a, b]), v, 0.5)
    assert diff > 0


# ---------------------------------------------------------------- VJP of Eq. 1
def _loss(q, k, v, g, tau):
    """L = sum_m g_m . s_m through the (separately pinned) forward oracle."""
    s, _ = oracle_sum(q, k, v, tau)
    return math.fsum((g * s).ravel())


def test_vjp_matches_finite_differences():
    """Central differences of L = sum_m g_m . s_m in every coordinate of q,
    k and v (chain rule on Eq. 1): catches a dropped term, a wrong sign or a
    transposed contraction in any of the three outputs."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(21)
    M, N, D, C, tau = 4, 5, 3, 2, 0.8
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, C))
    g = rng.standard_normal((M, C))
    r = oracle_vjp(q, k, v, g, tau)
    h = 1e-6

    def fd(arr, idx):
        a = arr.copy()
        a[idx] += h
        args_p = [a if x is arr else x for x in (q, k, v)]
        a2 = arr.copy()
        a2[idx] -= h
        args_m = [a2 if x is arr else x for x in (q, k, v)]
        return (_loss(*args_p, g, tau) - _loss(*args_m, g, tau)) / (2 * h)

    for name, arr, got in (("q", q, r["gq"]), ("k", k, r["gk"]), ("v", v, r["gv"])):
        want = np.array([[fd(arr, (i, j)) for j in range(arr.shape[1])]
                         for i in range(arr.shape[0])])
        np.testing.assert_allclose(got, want, rtol=1e-7, atol=1e-8, err_msg=name)


def test_vjp_reduces_to_q_gradient_for_unit_upstream():
    """C = 1, g = 1: dL/dq_m is the q-gradient of Sec. 3 (the other oracle
    function, written separately)."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(22)
    q = rng.standard_normal((9, 6))
    k = rng.standard_normal((13, 6))
    v = rng.standard_normal((13, 1))
    r = oracle_vjp(q, k, v, np.ones((9, 1)), 0.45)
    gq, _, den, _ = oracle_grad_q(q, k, v, 0.45)
    np.testing.assert_allclose(r["gq"], gq, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(r["dq"], den, rtol=1e-13, atol=1e-15)


def test_vjp_pairwise_antisymmetry_and_translation():
    """Each pair contributes opposite forces to q_m and k_n, so
    sum_m dL/dq_m + sum_n dL/dk_n = 0 (L is invariant under moving every
    point by the same vector); a common shift of all points changes no
    output."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(23)
    M, N, D, C, tau = 11, 7, 4, 3, 0.3
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, C))
    g = rng.standard_normal((M, C))
    r = oracle_vjp(q, k, v, g, tau)
    total = r["gq"].sum(0) + r["gk"].sum(0)
    scale = np.abs(r["gq"]).sum(0) + np.abs(r["gk"]).sum(0)
    assert np.all(np.abs(total) <= 1e-13 * scale)
    t = rng.standard_normal(D) * 3.0
    r2 = oracle_vjp(q + t, k + t, v, g, tau)
    for key in ("gq", "gk", "gv"):
        np.testing.assert_allclose(r2[key], r[key], rtol=1e-9, atol=1e-12, err_msg=key)


def test_vjp_brute_force_tiny():
    """Pure-Python double loop over pairs on a 2 x 3 problem."""
    from oracle import oracle_vjp
    q = [[0.5, -1.0], [0.0, 0.25]]
    k = [[1.0, 0.0], [-0.5, 0.5], [0.25, -0.75]]
    v = [[1.0, -2.0], [0.5, 0.0], [-1.5, 1.0]]
    g = [[2.0, 1.0], [-1.0, 0.5]]
    tau = 1.3
    gq = [[0.0, 0.0] for _ in q]
    gk = [[0.0, 0.0] for _ in k]
    gv = [[0.0, 0.0] for _ in k]
    for m in range(2):
        for n in range(3):
            phi = math.exp(-tau / 2 * sum((q[m][d] - k[n][d]) ** 2 for d in range(2)))
            w = sum(g[m][c] * v[n][c] for c in range(2))
            for d in range(2):
                gq[m][d] += tau * phi * w * (k[n][d] - q[m][d])
                gk[n][d] += tau * phi * w * (q[m][d] - k[n][d])
            for c in range(2):
                gv[n][c] += phi * g[m][c]
    r = oracle_vjp(np.array(q), np.array(k), np.array(v), np.array(g), tau)
    np.testing.assert_allclose(r["gq"], gq, rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(r["gk"], gk, rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(r["gv"], gv, rtol=1e-14, atol=1e-15)


def test_vjp_row_subsets_and_scales():
    """Row subsets return the selected rows of the full result; the error
    scales bound the outputs they belong to (|x| <= its scale, since both
    are sums of the same terms before and after taking magnitudes)."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(24)
    M, N, D, C = 17, 12, 5, 2
    q = rng.standard_normal((M, D))
    k = rng.standard_normal((N, D))
    v = rng.standard_normal((N, C))
    g = rng.standard_normal((M, C))
    full = oracle_vjp(q, k, v, g, 0.6)
    rq, rk = [16, 0, 5], [3, 11]
    sub = oracle_vjp(q, k, v, g, 0.6, rows_q=rq, rows_k=rk, nthreads=1)
    for key, rows in (("gq", rq), ("dq", rq), ("gk", rk), ("dk", rk), ("gv", rk), ("dv", rk)):
        np.testing.assert_array_equal(sub[key], full[key][rows], err_msg=key)
    for key, den in (("gq", "dq"), ("gk", "dk"), ("gv", "dv")):
        assert np.all(np.abs(full[key]) <= full[den] * (1 + 1e-12))
    with pytest.raises(ValueError):
        oracle_vjp(q, k, v, g, 0.6, rows_q=[M])


def test_vjp_error_scales_brute_force_signed_upstream():
    """The three error scales of the vector-Jacobian product for C = 2 and a
    signed, non-unit upstream g, recomputed by a pure-Python double loop
    (math.fsum) from their definitions: the terms of the per-channel Gauss
    sums with values (w x^, w) in coordinates shifted by the common mean mu,
    contracted with the magnitudes of the other side's weights (chain rule on
    Eq. 1, the gradient flows of Sec. 3)."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(25)
    M, N, D, C, tau = 4, 5, 3, 2, 0.7
    q = rng.standard_normal((M, D)) + 1.5
    k = rng.standard_normal((N, D)) - 0.5
    v = rng.standard_normal((N, C)) * np.array([1.0, -3.0])
    g = rng.standard_normal((M, C)) * np.array([-2.5, 0.4])
    r = oracle_vjp(q, k, v, g, tau)
    mu = np.concatenate([q, k]).mean(0)
    phi = [[math.exp(-tau / 2 * math.fsum((q[m] - k[n]) ** 2)) for n in range(N)]
           for m in range(M)]
    for m in range(M):
        for d in range(D):
            want = tau * math.fsum(
                abs(g[m, c]) * (math.fsum(phi[m][n] * abs(v[n, c]) * abs(k[n, d] - mu[d])
                                          for n in range(N))
                                + abs(q[m, d] - mu[d]) * math.fsum(phi[m][n] * abs(v[n, c])
                                                                    for n in range(N)))
                for c in range(C))
            assert r["dq"][m, d] == pytest.approx(want, rel=1e-13)
    for n in range(N):
        for d in range(D):
            want = tau * math.fsum(
                abs(v[n, c]) * (math.fsum(phi[m][n] * abs(g[m, c]) * abs(q[m, d] - mu[d])
                                          for m in range(M))
                                + abs(k[n, d] - mu[d]) * math.fsum(phi[m][n] * abs(g[m, c])
                                                                    for m in range(M)))
                for c in range(C))
            assert r["dk"][n, d] == pytest.approx(want, rel=1e-13)
        for c in range(C):
            want = math.fsum(phi[m][n] * abs(g[m, c]) for m in range(M))
            assert r["dv"][n, c] == pytest.approx(want, rel=1e-13)


def test_vjp_error_scales_from_the_other_oracle_functions():
    """Each VJP scale is a contraction of scales that the separately written
    (and separately pinned) oracle functions return: dq = sum_c |g_c| times
    the q-gradient scale of channel c, dk = sum_c |v_c| times the q-gradient
    scale with queries and keys exchanged and weights g_c, dv = the forward
    denominator sum_m Phi |g_mc| with queries and keys exchanged."""
    from oracle import oracle_vjp
    rng = np.random.default_rng(26)
    M, N, D, C, tau = 7, 6, 4, 3, 0.45
    q = rng.standard_normal((M, D)) * 0.8 + 0.3
    k = rng.standard_normal((N, D)) * 1.2
    v = rng.standard_normal((N, C))
    g = rng.standard_normal((M, C)) * 2.0
    r = oracle_vjp(q, k, v, g, tau)
    dq = np.zeros((M, D))
    dk = np.zeros((N, D))
    for c in range(C):
        _, _, den_q, _ = oracle_grad_q(q, k, v[:, c], tau)
        dq += np.abs(g[:, c:c + 1]) * den_q
        _, _, den_k, _ = oracle_grad_q(k, q, g[:, c], tau)
        dk += np.abs(v[:, c:c + 1]) * den_k
    _, dv = oracle_sum(k, q, g, tau)
    np.testing.assert_allclose(r["dq"], dq, rtol=1e-12)
    np.testing.assert_allclose(r["dk"], dk, rtol=1e-12)
    np.testing.assert_allclose(r["dv"], dv, rtol=1e-12)
