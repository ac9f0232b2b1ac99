"""The FMA-pipe exp2 of the fused kernel (exp2_fma_x2 in ptx.cuh), emulated
step by step in float32 on the CPU with the coefficients read from the
source: relative error against 2^x within the fitted bound where 2^x is a
normal float, and results that flush to zero (or stay below 2^-126) where
ex2.approx.ftz flushes.  Also re-derives the fit: the Remez exchange in
csrc/fit_exp2_poly.py must reproduce the committed coefficients."""
import os
import re

import numpy as np

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2609_04910_gb300", "csrc")


def _coefficients():
    src = open(os.path.join(CSRC, "ptx.cuh")).read()
    body = src[src.index("exp2_fma_x2"):]
    vals = [float(x) for x in re.findall(r"f32x2_pack\(([0-9.e+-]+)f, \1f\)", body)[:5]]
    # Horner order in the source: c4, c3, c2, c1, c0
    return np.array(vals[::-1], dtype=np.float32)


def _f32(x):
    return np.asarray(x, dtype=np.float64).astype(np.float32)


def _fma32(a, b, c):
    # float32 fma: the product of two float32 values is exact in float64
    return _f32(a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64))


def _exp2_fma(s, c):
    s = _f32(s)
    c = np.float32(c)
    s_min = np.float32(-127.0) / c
    s = np.maximum(s, s_min)
    magic = np.float32(12582912.0)
    cc = np.full_like(s, c)
    t = _fma32(s, cc, np.full_like(s, magic))
    f = _fma32(s, cc, _f32(magic - t))
    k = _coefficients()
    p = _fma32(f, np.full_like(f, k[4]), np.full_like(f, k[3]))
    for a in (k[2], k[1], k[0]):
        p = _fma32(p, f, np.full_like(f, a))
    bits = (t.view(np.uint32).astype(np.uint64) * (1 << 23) + 0x3F800000) & 0xFFFFFFFF
    e = bits.astype(np.uint32).view(np.float32)
    r = _f32(p.astype(np.float64) * e.astype(np.float64))
    r[np.abs(r) < np.float32(2.0 ** -126)] = 0.0          # mul.ftz
    return r


def test_relative_error_in_normal_range():
    for c in (1.4426950408889634 / 64, 1.0, 0.37, 9.5):
        x = np.linspace(-125.9, 0.3, 400001)
        s = _f32(x / c)
        xe = s.astype(np.float64) * np.float64(np.float32(c))
        got = _exp2_fma(s, c).astype(np.float64)
        rel = np.abs(got / np.exp2(xe) - 1.0)
        assert rel.max() < 3e-6, (c, rel.max())


def test_flush_below_the_normal_range():
    c = 0.7
    s = _f32(np.linspace(-1e6, -127.0 / c, 10001))
    got = _exp2_fma(s, c)
    assert np.all(got == 0.0)
    s = _f32(np.linspace(-127.0 / c, -126.0 / c, 1001))
    got = _exp2_fma(s, c)
    assert np.all((got >= 0.0) & (got <= 2.0 ** -125))


def test_exact_at_integers():
    c = 1.0
    s = _f32(np.arange(-120, 1))
    got = _exp2_fma(s, c).astype(np.float64)
    assert np.all(np.abs(got / np.exp2(s.astype(np.float64)) - 1.0) < 1e-6)


def test_fit_reproduces_coefficients():
    import importlib.util
    spec = importlib.util.spec_from_file_location("fit", os.path.join(CSRC, "fit_exp2_poly.py"))
    fit = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(fit)
    c, err = fit.remez(4)
    assert err < 3e-6
    np.testing.assert_allclose(c.astype(np.float32), _coefficients(), rtol=0, atol=0)
