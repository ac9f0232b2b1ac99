"""Fits the polynomial behind the FMA-pipe exp2 of tc_gauss_fma.cu.

2^x = 2^j * 2^f with j = round(x) and f = x - j in [-1/2, 1/2] (Cody-Waite
range reduction with a single constant, exact here because the reduction
is by an integer).  2^f is replaced by the polynomial p of degree n that
minimises max |p(f) / 2^f - 1| on [-1/2, 1/2], found by the Remez exchange
algorithm (equioscillation of the weighted error at n + 2 points).  The
coefficients are then rounded to float32 and the relative error of the
float32 Horner evaluation is measured on a dense grid.

Run: python fit_exp2_poly.py [degree]   (prints the coefficients, c0 first)
"""
import sys

import numpy as np


def remez(deg, lo=-0.5, hi=0.5, iters=30):
    n = deg + 2
    # Chebyshev extrema as the first reference.
    x = 0.5 * (lo + hi) + 0.5 * (hi - lo) * np.cos(np.pi * np.arange(n)[::-1] / (n - 1))
    grid = np.linspace(lo, hi, 200001)
    for _ in range(iters):
        # p(x_i) - 2^x_i = (-1)^i E 2^x_i  ->  unknowns c_0..c_deg, E
        A = np.zeros((n, n))
        for i in range(n):
            A[i, :deg + 1] = x[i] ** np.arange(deg + 1)
            A[i, deg + 1] = -((-1) ** i) * 2.0 ** x[i]
        sol = np.linalg.solve(A, 2.0 ** x)
        c = sol[:deg + 1]
        err = np.polyval(c[::-1], grid) / 2.0 ** grid - 1.0
        # New reference: the extremum of each run of constant error sign.
        sign = np.sign(err)
        cuts = np.flatnonzero(np.diff(sign)) + 1
        runs = np.split(np.arange(grid.size), cuts)
        ext = [r[np.argmax(np.abs(err[r]))] for r in runs]
        if len(ext) < n:
            break
        # keep the n consecutive extrema with the largest minimum magnitude
        best, best_k = -1.0, 0
        for k in range(len(ext) - n + 1):
            m = np.min(np.abs(err[ext[k:k + n]]))
            if m > best:
                best, best_k = m, k
        x = grid[ext[best_k:best_k + n]]
    return c, float(np.max(np.abs(err)))


def f32_horner_error(c32, lo=-0.5, hi=0.5, count=2000001):
    f = np.linspace(lo, hi, count).astype(np.float32)
    p = np.full_like(f, c32[-1])
    for a in c32[-2::-1]:
        # fma in float32: the product of two float32 is exact in float64
        p = (p.astype(np.float64) * f.astype(np.float64) + np.float64(a)).astype(np.float32)
    return float(np.max(np.abs(p.astype(np.float64) / 2.0 ** f.astype(np.float64) - 1.0)))


if __name__ == "__main__":
    deg = int(sys.argv[1]) if len(sys.argv) > 1 else 5
    c, e = remez(deg)
    c32 = c.astype(np.float32)
    print(f"degree {deg}: minimax relative error {e:.3e} (float64 coefficients), "
          f"{f32_horner_error(c32):.3e} (float32 Horner)")
    for i, a in enumerate(c32):
        print(f"c{i} = {float(a):.9e}f  /* 0x{np.float32(a).view(np.uint32):08x} */")
