"""The C-ABI library loads, exports every declared symbol, and rejects bad
arguments on the host (no GPU needed: these calls return before any CUDA
work is issued)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_04910_gb300.build import build_library
    from paper_2609_04910_gb300._binding import load_library
    build_library()
    return load_library()


def _declared_functions(header="gauss_sum.h"):
    src = open(os.path.join(ROOT, "include", header)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(gauss_sum\w*)\s*\(", src)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    from paper_2609_04910_gb300._binding import EXPORTS, TESTING_EXPORTS
    declared = _declared_functions()
    assert len(declared) == 16
    assert sorted(EXPORTS) == declared
    testing = _declared_functions("gauss_sum_testing.h")
    assert sorted(TESTING_EXPORTS) == testing
    headers = sorted(f for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h"))
    assert headers == ["gauss_sum.h", "gauss_sum_testing.h"]
    for name in declared + testing:
        assert hasattr(lib, name), name


def test_launch_counter_starts_without_gpu_work(lib):
    # Argument errors return before any launch, so the count does not move.
    n0 = lib.gauss_sum_kernel_launches()
    st = lib.gauss_sum(None, None, None, 1.0, 1, 1, 1, 1, 1, None, None)
    assert st == 1
    assert lib.gauss_sum_kernel_launches() == n0


def test_status_strings(lib):
    assert lib.gauss_sum_status_string(0) == b"GS_OK"
    assert lib.gauss_sum_status_string(5) == b"GS_ERR_DEVICE_TIMEOUT"


def test_default_options(lib):
    from paper_2609_04910_gb300._binding import GsOptions
    o = GsOptions()
    o.center = 7
    lib.gauss_sum_default_options(ctypes.byref(o))
    assert (o.center, o.split_n, o.workspace, o.workspace_bytes, o.path) == (1, 0, None, 0, 0)
    assert list(o.main_events) == [None, None]
    assert o.exp2_fma == 0


@pytest.mark.parametrize("bad", [-1, 5])
def test_exp2_fma_range_checked(lib, bad):
    from paper_2609_04910_gb300._binding import GsOptions
    o = GsOptions()
    lib.gauss_sum_default_options(ctypes.byref(o))
    o.exp2_fma = bad
    st = lib.gauss_sum_ex(ALIGNED, ALIGNED, ALIGNED, 1.0, 4, 4, 3, 1, 1, ALIGNED, None,
                          ctypes.byref(o))
    assert st == 1
    assert b"exp2_fma" in lib.gauss_sum_last_error()


ALIGNED = 4096  # a fake 16-byte-aligned address; never dereferenced


@pytest.mark.parametrize("case,expect", [
    (dict(tau=0.0), 1), (dict(tau=-1.0), 1), (dict(tau=float("nan")), 1),
    (dict(tau=float("inf")), 1), (dict(M=-1), 1), (dict(D=-3), 1), (dict(dtype=9), 1),
    (dict(q=None), 1), (dict(k=None), 1), (dict(v=None), 1), (dict(out=None), 1),
    (dict(q=ALIGNED + 4), 1), (dict(out=ALIGNED + 8), 1),
])
def test_argument_errors(lib, case, expect):
    a = dict(q=ALIGNED, k=ALIGNED, v=ALIGNED, tau=1.0, M=4, N=4, D=3, C=2, dtype=1, out=ALIGNED)
    a.update(case)
    st = lib.gauss_sum(a["q"], a["k"], a["v"], a["tau"], a["M"], a["N"], a["D"], a["C"],
                       a["dtype"], a["out"], None)
    assert st == expect
    assert lib.gauss_sum_last_error()


def test_grad_requires_scalar_weights(lib):
    from paper_2609_04910_gb300._binding import GsOptions
    st = lib.gauss_sum_grad_q(ALIGNED, ALIGNED, ALIGNED, 0.0, 4, 4, 3, 1, ALIGNED, None, None)
    assert st == 1


@pytest.mark.parametrize("case", [
    dict(g=None), dict(g=ALIGNED + 4), dict(C=-1), dict(tau=0.0), dict(dtype=7), dict(v=None),
    dict(gq=ALIGNED + 8),
])
def test_vjp_argument_errors(lib, case):
    a = dict(q=ALIGNED, k=ALIGNED, v=ALIGNED, g=ALIGNED, tau=1.0, M=4, N=5, D=3, C=2, dtype=1,
             gq=ALIGNED, gk=ALIGNED, gv=ALIGNED)
    a.update(case)
    n0 = lib.gauss_sum_kernel_launches()
    st = lib.gauss_sum_vjp(a["q"], a["k"], a["v"], a["g"], a["tau"], a["M"], a["N"], a["D"],
                           a["C"], a["dtype"], a["gq"], a["gk"], a["gv"], None)
    assert st == 1
    assert lib.gauss_sum_last_error()
    assert lib.gauss_sum_kernel_launches() == n0


def test_vjp_without_outputs_is_a_noop(lib):
    assert lib.gauss_sum_vjp(ALIGNED, ALIGNED, ALIGNED, ALIGNED, 1.0, 4, 5, 3, 2, 1,
                             None, None, None, None) == 0


def test_path_dtype_mismatch_is_unsupported(lib):
    from paper_2609_04910_gb300._binding import GS_PATH_SIMT, GS_PATH_TENSOR, options
    o = options(path=GS_PATH_TENSOR)
    # fp32 on the tensor cores: forward sums with C <= 4 and D <= 32 only.
    st = lib.gauss_sum_ex(ALIGNED, ALIGNED, ALIGNED, 1.0, 4, 4, 40, 1, 0, ALIGNED, None, ctypes.byref(o))
    assert st == 2
    st = lib.gauss_sum_ex(ALIGNED, ALIGNED, ALIGNED, 1.0, 4, 4, 3, 5, 0, ALIGNED, None, ctypes.byref(o))
    assert st == 2
    o = options(path=GS_PATH_SIMT)
    st = lib.gauss_sum_ex(ALIGNED, ALIGNED, ALIGNED, 1.0, 4, 4, 3, 1, 1, ALIGNED, None, ctypes.byref(o))
    assert st == 2


def test_noop_calls_succeed_without_gpu(lib):
    # M = 0 returns before any CUDA call.
    assert lib.gauss_sum(None, ALIGNED, ALIGNED, 1.0, 0, 5, 3, 1, 1, None, None) == 0


def test_workspace_size_plans(lib):
    from paper_2609_04910_gb300._binding import options
    o = options()
    f = lib.gauss_sum_workspace_size
    assert f(0, 10, 3, 1, 1, 0, ctypes.byref(o)) == 0
    big = f(65536, 65536, 64, 1, 1, 0, ctypes.byref(o))
    assert big > 2 * 65536 * 64 * 2
    assert f(10, 10, 300, 1, 1, 0, ctypes.byref(o)) == ctypes.c_size_t(-1).value  # D > 256 fp16
    # Gradient with D + 1 > 256 channels: evaluated in two channel chunks.
    assert 0 < f(10, 10, 256, 1, 1, 1, ctypes.byref(o)) < ctypes.c_size_t(-1).value
    assert f(10, 10, 200, 1, 0, 0, ctypes.byref(o)) == ctypes.c_size_t(-1).value  # fp32 D > 128
    assert f(1000, 1000, 16, 3, 0, 0, ctypes.byref(o)) > 0


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2609_04910_gb300._binding import load_library
    with pytest.raises(RuntimeError):
        load_library(str(tmp_path / "missing.so"))
