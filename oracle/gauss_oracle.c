/*
 * Gauss-sum oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, float64 CPU evaluation of the Gauss kernel sum and of its
 * gradient with respect to the query points, written straight from the
 * problem statement of "Fast Gauss Sums via Flash Attention" (arXiv
 * 2609.04910):
 *
 *   Phi_tau(q, k) = exp(-tau/2 * ||q - k||^2)                  (Sec. 1)
 *   s_m           = sum_n Phi_tau(q_m, k_n) v_n   in R^C          (Eq. 1)
 *   grad_{q_m} s_m = tau * sum_n Phi_tau(q_m, k_n) v_n (k_n - q_m) (Sec. 3,
 *                    MMD flows / SVGD, scalar weights v_n)
 *
 * and the vector-Jacobian product of Eq. 1 for an upstream g (M x C),
 * i.e. the gradients of L = sum_m g_m . s_m with respect to q, k and v
 * (chain rule on Eq. 1, the building block of the flows of Sec. 3):
 *
 *   dL/dq_m = tau * sum_n Phi(q_m, k_n) (g_m . v_n) (k_n - q_m)
 *   dL/dk_n = tau * sum_m Phi(q_m, k_n) (g_m . v_n) (q_m - k_n)
 *   dL/dv_n =       sum_m Phi(q_m, k_n) g_m
 *
 * Nothing of the fast method is used here: no Gram identity, no centering,
 * no log2/exp2, no tiling.  The squared distance is the direct difference
 * form, the exponential is libm exp(), and the sum over n is sequential in
 * n.  Rows are independent and are spread over OpenMP threads; each row is
 * computed by one thread in a fixed order, so results do not depend on the
 * thread count.
 *
 * Only the test suite, the package smoke check and the benchmark's CPU
 * baseline call this file.  The CUDA library never links or loads it.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* Squared Euclidean distance ||a - b||^2, direct difference form. */
static double sq_dist(const double* a, const double* b, int64_t D)
{
    double acc = 0.0;
    for (int64_t d = 0; d < D; ++d) {
        double t = a[d] - b[d];
        acc += t * t;
    }
    return acc;
}

/* Phi_tau(q, k) = exp(-tau/2 ||q-k||^2)  (Sec. 1). */
static double gauss_kernel(const double* a, const double* b, int64_t D, double tau)
{
    return exp(-0.5 * tau * sq_dist(a, b, D));
}

/*
 * Eq. 1 for the rows listed in `rows` (or rows 0..R-1 when rows == NULL).
 *
 *   q    : M x D row-major, k : N x D, v : N x C  (float64)
 *   s    : R x C output,  s[r, c]   = sum_n Phi(q_m, k_n) v[n, c]
 *   den  : R x C output,  den[r, c] = sum_n Phi(q_m, k_n) |v[n, c]|
 *          (the scale of the sum before signed cancellation; may be NULL)
 *
 * Returns 0, or -1 on a bad argument.
 */
int gs_oracle_sum(const double* q, const double* k, const double* v,
                  double tau, int64_t M, int64_t N, int64_t D, int64_t C,
                  const int64_t* rows, int64_t R,
                  double* s, double* den, int nthreads)
{
    if (M < 0 || N < 0 || D < 0 || C < 0 || R < 0) return -1;
    if (R > 0 && (!q || !s)) return -1;
    if (N > 0 && (!k || !v)) return -1;
    if (nthreads < 1) nthreads = 1;
    for (int64_t r = 0; r < R; ++r) {
        int64_t m = rows ? rows[r] : r;
        if (m < 0 || m >= M) return -1;
    }

#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads)
    for (int64_t r = 0; r < R; ++r) {
        int64_t m = rows ? rows[r] : r;
        const double* qm = q + m * D;
        double* sr = s + r * C;
        double* dr = den ? den + r * C : NULL;
        for (int64_t c = 0; c < C; ++c) {
            sr[c] = 0.0;
            if (dr) dr[c] = 0.0;
        }
        for (int64_t n = 0; n < N; ++n) {
            double phi = gauss_kernel(qm, k + n * D, D, tau);
            const double* vn = v + n * C;
            for (int64_t c = 0; c < C; ++c) {
                sr[c] += phi * vn[c];
                if (dr) dr[c] += phi * fabs(vn[c]);
            }
        }
    }
    return 0;
}

/*
 * Gradient of Eq. 1 with respect to q_m for scalar weights (C = 1), as in
 * Sec. 3 (MMD flows and SVGD):
 *
 *   g[r, d] = tau * sum_n Phi(q_m, k_n) v_n (k[n, d] - q[m, d])
 *   s[r]    = sum_n Phi(q_m, k_n) v_n
 *
 * Error scales reported beside g (either may be NULL):
 *   den[r, d]       = tau * ( sum_n Phi |v_n| |k[n,d] - mu[d]|
 *                             + |q[m,d] - mu[d]| * sum_n Phi |v_n| )
 *       with mu the float64 mean of all M + N points.  This is the size of
 *       the two terms the sum splits into when the gradient is evaluated as
 *       one Gauss sum with values (v_n k_n, v_n) in coordinates shifted by
 *       the common mean.
 *   den_shift[r, d] = tau * sum_n Phi |v_n| |k[n,d] - q[m,d]|
 *       (shift invariant; a diagnostic only).
 */
int gs_oracle_grad_q(const double* q, const double* k, const double* v,
                     double tau, int64_t M, int64_t N, int64_t D,
                     const int64_t* rows, int64_t R,
                     double* g, double* s, double* den, double* den_shift,
                     int nthreads)
{
    if (M < 0 || N < 0 || D < 0 || R < 0) return -1;
    if (R > 0 && (!q || !g)) return -1;
    if (N > 0 && (!k || !v)) return -1;
    if (nthreads < 1) nthreads = 1;
    for (int64_t r = 0; r < R; ++r) {
        int64_t m = rows ? rows[r] : r;
        if (m < 0 || m >= M) return -1;
    }

    double* mu = (double*)calloc((size_t)(D > 0 ? D : 1), sizeof(double));
    if (!mu) return -1;
    if (M + N > 0) {
        for (int64_t m = 0; m < M; ++m)
            for (int64_t d = 0; d < D; ++d) mu[d] += q[m * D + d];
        for (int64_t n = 0; n < N; ++n)
            for (int64_t d = 0; d < D; ++d) mu[d] += k[n * D + d];
        for (int64_t d = 0; d < D; ++d) mu[d] /= (double)(M + N);
    }

    int bad = 0;
#pragma omp parallel num_threads(nthreads)
    {
        double* kshift = (double*)malloc((size_t)(D > 0 ? D : 1) * 3 * sizeof(double));
        if (!kshift) {
#pragma omp atomic write
            bad = 1;
        } else {
            double* acc_den = kshift + (D > 0 ? D : 1);
            double* acc_dsh = acc_den + (D > 0 ? D : 1);
#pragma omp for schedule(dynamic, 1)
            for (int64_t r = 0; r < R; ++r) {
                int64_t m = rows ? rows[r] : r;
                const double* qm = q + m * D;
                double* gr = g + r * D;
                double sum_w = 0.0, sum_absw = 0.0;
                for (int64_t d = 0; d < D; ++d) {
                    gr[d] = 0.0;
                    acc_den[d] = 0.0;
                    acc_dsh[d] = 0.0;
                }
                for (int64_t n = 0; n < N; ++n) {
                    const double* kn = k + n * D;
                    double phi = gauss_kernel(qm, kn, D, tau);
                    double w = phi * v[n];
                    double aw = phi * fabs(v[n]);
                    sum_w += w;
                    sum_absw += aw;
                    for (int64_t d = 0; d < D; ++d) {
                        gr[d] += w * (kn[d] - qm[d]);
                        acc_den[d] += aw * fabs(kn[d] - mu[d]);
                        acc_dsh[d] += aw * fabs(kn[d] - qm[d]);
                    }
                }
                for (int64_t d = 0; d < D; ++d) {
                    gr[d] *= tau;
                    if (den) den[r * D + d] = tau * (acc_den[d] + fabs(qm[d] - mu[d]) * sum_absw);
                    if (den_shift) den_shift[r * D + d] = tau * acc_dsh[d];
                }
                if (s) s[r] = sum_w;
            }
            free(kshift);
        }
    }
    free(mu);
    return bad ? -1 : 0;
}

/*
 * Vector-Jacobian product of Eq. 1: the gradients of L = sum_m g_m . s_m
 * with respect to q, k and v, for rows rows_q (R_q entries) of dL/dq and
 * rows rows_k (R_k entries) of dL/dk and dL/dv (NULL: all rows).
 *
 *   q : M x D, k : N x D, v : N x C, g : M x C  (float64)
 *   gq[r, d] = tau * sum_n Phi(q_m, k_n) w_mn (k[n, d] - q[m, d])
 *   gk[r, d] = tau * sum_m Phi(q_m, k_n) w_mn (q[m, d] - k[n, d])
 *   gv[r, c] =       sum_m Phi(q_m, k_n) g[m, c]
 *   with w_mn = sum_c g[m, c] v[n, c].
 *
 * Error scales beside each output (any may be NULL), with mu the float64
 * mean of all M + N points: the size of the terms of the evaluation as
 * per-channel Gauss sums with values (w k^, w) in coordinates shifted by mu,
 * contracted with the other side's weights:
 *   dq[r, d] = tau sum_c |g[m,c]| ( sum_n Phi |v[n,c]| |k[n,d] - mu_d|
 *                                   + |q[m,d] - mu_d| sum_n Phi |v[n,c]| )
 *   dk[r, d] = tau sum_c |v[n,c]| ( sum_m Phi |g[m,c]| |q[m,d] - mu_d|
 *                                   + |k[n,d] - mu_d| sum_m Phi |g[m,c]| )
 *   dv[r, c] = sum_m Phi |g[m, c]|
 * Any of gq, gk, gv may be NULL (that output is skipped).
 */
int gs_oracle_vjp(const double* q, const double* k, const double* v, const double* g,
                  double tau, int64_t M, int64_t N, int64_t D, int64_t C,
                  const int64_t* rows_q, int64_t Rq, const int64_t* rows_k, int64_t Rk,
                  double* gq, double* gk, double* gv, double* dq, double* dk, double* dv,
                  int nthreads)
{
    if (M < 0 || N < 0 || D < 0 || C < 0 || Rq < 0 || Rk < 0) return -1;
    if ((M > 0 && (!q || !g)) || (N > 0 && (!k || !v))) return -1;
    if (nthreads < 1) nthreads = 1;
    for (int64_t r = 0; r < Rq; ++r) {
        int64_t m = rows_q ? rows_q[r] : r;
        if (m < 0 || m >= M) return -1;
    }
    for (int64_t r = 0; r < Rk; ++r) {
        int64_t n = rows_k ? rows_k[r] : r;
        if (n < 0 || n >= N) return -1;
    }

    const int64_t Dm = D > 0 ? D : 1, Cm = C > 0 ? C : 1;
    double* mu = (double*)calloc((size_t)Dm, sizeof(double));
    if (!mu) return -1;
    if (M + N > 0) {
        for (int64_t m = 0; m < M; ++m)
            for (int64_t d = 0; d < D; ++d) mu[d] += q[m * D + d];
        for (int64_t n = 0; n < N; ++n)
            for (int64_t d = 0; d < D; ++d) mu[d] += k[n * D + d];
        for (int64_t d = 0; d < D; ++d) mu[d] /= (double)(M + N);
    }

    int bad = 0;
#pragma omp parallel num_threads(nthreads)
    {
        /* per thread: sum_n Phi |v_nc| |x_d - mu_d| (C x D) and sum Phi |v_nc| (C) */
        double* a = (double*)malloc((size_t)(Cm * Dm + Cm) * sizeof(double));
        if (!a) {
#pragma omp atomic write
            bad = 1;
        } else {
            double* b = a + Cm * Dm;
            /* dL/dq: one query row at a time, keys in order. */
#pragma omp for schedule(dynamic, 1)
            for (int64_t r = 0; r < Rq; ++r) {
                const int64_t m = rows_q ? rows_q[r] : r;
                const double* qm = q + m * D;
                const double* gm = g + m * C;
                for (int64_t i = 0; i < Cm * Dm + Cm; ++i) a[i] = 0.0;
                double* out = gq ? gq + r * D : NULL;
                if (out)
                    for (int64_t d = 0; d < D; ++d) out[d] = 0.0;
                for (int64_t n = 0; n < N; ++n) {
                    const double* kn = k + n * D;
                    const double* vn = v + n * C;
                    const double phi = gauss_kernel(qm, kn, D, tau);
                    double w = 0.0;
                    for (int64_t c = 0; c < C; ++c) w += gm[c] * vn[c];
                    if (out)
                        for (int64_t d = 0; d < D; ++d) out[d] += phi * w * (kn[d] - qm[d]);
                    for (int64_t c = 0; c < C; ++c) {
                        const double pv = phi * fabs(vn[c]);
                        b[c] += pv;
                        for (int64_t d = 0; d < D; ++d) a[c * Dm + d] += pv * fabs(kn[d] - mu[d]);
                    }
                }
                for (int64_t d = 0; d < D; ++d) {
                    if (out) out[d] *= tau;
                    if (dq) {
                        double e = 0.0;
                        for (int64_t c = 0; c < C; ++c)
                            e += fabs(gm[c]) * (a[c * Dm + d] + fabs(qm[d] - mu[d]) * b[c]);
                        dq[r * D + d] = tau * e;
                    }
                }
            }
            /* dL/dk and dL/dv: one key row at a time, queries in order. */
#pragma omp for schedule(dynamic, 1)
            for (int64_t r = 0; r < Rk; ++r) {
                const int64_t n = rows_k ? rows_k[r] : r;
                const double* kn = k + n * D;
                const double* vn = v + n * C;
                for (int64_t i = 0; i < Cm * Dm + Cm; ++i) a[i] = 0.0;
                double* outk = gk ? gk + r * D : NULL;
                double* outv = gv ? gv + r * C : NULL;
                if (outk)
                    for (int64_t d = 0; d < D; ++d) outk[d] = 0.0;
                if (outv)
                    for (int64_t c = 0; c < C; ++c) outv[c] = 0.0;
                for (int64_t m = 0; m < M; ++m) {
                    const double* qm = q + m * D;
                    const double* gm = g + m * C;
                    const double phi = gauss_kernel(qm, kn, D, tau);
                    double w = 0.0;
                    for (int64_t c = 0; c < C; ++c) w += vn[c] * gm[c];
                    if (outk)
                        for (int64_t d = 0; d < D; ++d) outk[d] += phi * w * (qm[d] - kn[d]);
                    for (int64_t c = 0; c < C; ++c) {
                        if (outv) outv[c] += phi * gm[c];
                        const double pg = phi * fabs(gm[c]);
                        b[c] += pg;
                        for (int64_t d = 0; d < D; ++d) a[c * Dm + d] += pg * fabs(qm[d] - mu[d]);
                    }
                }
                for (int64_t d = 0; d < D; ++d) {
                    if (outk) outk[d] *= tau;
                    if (dk) {
                        double e = 0.0;
                        for (int64_t c = 0; c < C; ++c)
                            e += fabs(vn[c]) * (a[c * Dm + d] + fabs(kn[d] - mu[d]) * b[c]);
                        dk[r * D + d] = tau * e;
                    }
                }
                if (dv)
                    for (int64_t c = 0; c < C; ++c) dv[r * C + c] = b[c];
            }
            free(a);
        }
    }
    free(mu);
    return bad ? -1 : 0;
}

/* Threads OpenMP would use by default (1 when built without OpenMP). */
int gs_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
