"""Seeded synthetic inputs for the Gauss-sum workloads.

This module only draws random numbers and rounds them to the storage dtype;
it contains none of the Gauss-sum arithmetic.  The same arrays feed the CUDA
library and the float64 oracle, so both see bit-identical inputs.

Recipe (all draws from ``numpy.random.default_rng(seed)``, PCG64, in float64,
in the order listed, row blocks of ``_BLOCK`` rows drawn one after another;
then rounded to the dtype: float32/float16 by ``numpy.astype`` (round to
nearest even), bfloat16 by float64 -> float32 -> bfloat16 with round to
nearest even).  The clouds follow the benchmark of Sec. 4 of the paper
(standard Gaussian point clouds; the paper scales the points by D^-1/2 at
tau = 1, which is the same kernel as unscaled points at tau = 1/D).

  fp32_d16     M=N=4096,   D=16,  C=1,  fp32: q, k, v ~ N(0,1); tau = 1/16
  mmd_d64      M=N=65536,  D=64,  C=1,  fp16: q ~ N(0,1) and k ~ N(0,1) drawn
               independently (q first); v = +1/N for the first N/2 keys,
               -1/N for the rest; tau = 1/64
  mmd_d64_qk   the same sizes in the MMD form q = k = X of Sec. 3 (one cloud
               X ~ N(0,1) carrying both signed halves)
  multi_c64    M=N=262144, D=128, C=64, bf16: q, k ~ 0.5 N(0,1); v ~ N(0,1);
               tau = 2/128
  svgd_d32     M=N=131072, D=32,  C=1,  fp16: 4-component Gaussian mixture
               (component means ~ N(0, 4 I), unit covariance, labels drawn
               uniformly); q = k = X; v = +1/N first half, -1/N second half;
               tau = 1/32; forward sum and q-gradient
  offset_d256  M=16384, N=1048576, D=256, C=4, fp16: shared offset
               u = 50 w/||w||, w ~ N(0, I) drawn first; q = u + 0.1 N(0,I),
               k = u + 0.1 N(0,I); v ~ U[-1, 1]; tau = 10/256
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

_BLOCK = 65536


@dataclass(frozen=True)
class Workload:
    name: str
    M: int
    N: int
    D: int
    C: int
    dtype: str          # "fp32", "fp16" or "bf16"
    tau: float
    kind: str           # generator recipe, see module docstring
    grad: bool = False  # also evaluate the q-gradient (C must be 1)
    q_is_k: bool = False
    note: str = field(default="", compare=False)

    @property
    def pairs(self) -> int:
        return self.M * self.N

    def resized(self, M=None, N=None, D=None, C=None) -> "Workload":
        """The same recipe at other sizes (tau keeps its 1/D-type law)."""
        D2 = self.D if D is None else D
        tau = self.tau * self.D / D2
        M2 = self.M if M is None else M
        N2 = self.N if N is None else N
        if self.q_is_k:
            M2 = N2 = N if N is not None else M2
        return replace(self, M=M2, N=N2, D=D2, C=self.C if C is None else C, tau=tau)


WORKLOADS = {
    "fp32_d16": Workload("fp32_d16", 4096, 4096, 16, 1, "fp32", 1.0 / 16, "normal",
                         note="forward Gauss sum in fp32"),
    "mmd_d64": Workload("mmd_d64", 65536, 65536, 64, 1, "fp16", 1.0 / 64, "independent_mmd",
                        note="MMD-style forward in fp16, fp32 accumulation"),
    "mmd_d64_qk": Workload("mmd_d64_qk", 65536, 65536, 64, 1, "fp16", 1.0 / 64, "mmd",
                           q_is_k=True, note="MMD-style forward, q = k form"),
    "multi_c64": Workload("multi_c64", 262144, 262144, 128, 64, "bf16", 2.0 / 128, "half_normal",
                          note="multi-channel forward in bf16"),
    "svgd_d32": Workload("svgd_d32", 131072, 131072, 32, 1, "fp16", 1.0 / 32, "gmm", grad=True,
                         q_is_k=True, note="SVGD/MMD flow step: forward sum and q-gradient"),
    "offset_d256": Workload("offset_d256", 16384, 1048576, 256, 4, "fp16", 10.0 / 256, "offset",
                            note="fp16 cancellation stress: common offset of norm 50"),
}


def _normal_rows(rng, rows, cols, scale=1.0):
    out = np.empty((rows, cols), dtype=np.float64)
    for r0 in range(0, rows, _BLOCK):
        r1 = min(rows, r0 + _BLOCK)
        out[r0:r1] = rng.standard_normal((r1 - r0, cols))
    if scale != 1.0:
        out *= scale
    return out


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 draws to the storage dtype.

    Returns float32 / float16 numpy arrays, or for bf16 a uint16 array of
    the raw bfloat16 bit patterns (numpy has no bfloat16 type).
    """
    if dtype == "fp32":
        return np.ascontiguousarray(x.astype(np.float32))
    if dtype == "fp16":
        return np.ascontiguousarray(x.astype(np.float16))
    if dtype == "bf16":
        import torch
        t = torch.from_numpy(np.ascontiguousarray(x.astype(np.float32))).to(torch.bfloat16)
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    raise ValueError(f"unknown dtype {dtype!r}")


def to_float64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 value of an array produced by ``round_to``."""
    if dtype == "bf16":
        bits = np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16
        return bits.view(np.float32).astype(np.float64)
    return np.asarray(a, dtype=np.float64)


def _signed_halves(N):
    v = np.full((N, 1), 1.0 / N, dtype=np.float64)
    v[N // 2:] = -1.0 / N
    return v


def generate(w: Workload, seed: int = 0) -> dict:
    """Draw the inputs of workload ``w``.

    Returns a dict with ``q``, ``k``, ``v`` (rounded, see ``round_to``),
    their float64 values ``q64``, ``k64``, ``v64``, and the workload.
    When ``w.q_is_k`` the ``q`` entry is the same array object as ``k``.
    """
    rng = np.random.default_rng(seed)
    M, N, D, C = w.M, w.N, w.D, w.C
    if w.kind == "normal":
        q = _normal_rows(rng, M, D)
        k = _normal_rows(rng, N, D)
        v = _normal_rows(rng, N, C)
    elif w.kind == "half_normal":
        q = _normal_rows(rng, M, D, 0.5)
        k = _normal_rows(rng, N, D, 0.5)
        v = _normal_rows(rng, N, C)
    elif w.kind == "mmd":
        k = _normal_rows(rng, N, D)
        q = k
        v = _signed_halves(N)
        if C != 1:
            v = np.repeat(v, C, axis=1)
    elif w.kind == "gmm":
        means = rng.standard_normal((4, D)) * 2.0
        labels = rng.integers(0, 4, size=N)
        k = _normal_rows(rng, N, D)
        k += means[labels]
        q = k
        v = _signed_halves(N)
    elif w.kind == "offset":
        wv = rng.standard_normal(D)
        u = 50.0 * wv / np.linalg.norm(wv)
        q = _normal_rows(rng, M, D, 0.1)
        q += u
        k = _normal_rows(rng, N, D, 0.1)
        k += u
        v = np.empty((N, C), dtype=np.float64)
        for r0 in range(0, N, _BLOCK):
            r1 = min(N, r0 + _BLOCK)
            v[r0:r1] = rng.uniform(-1.0, 1.0, size=(r1 - r0, C))
    elif w.kind == "independent_mmd":
        q = _normal_rows(rng, M, D)
        k = _normal_rows(rng, N, D)
        v = _signed_halves(N)
    else:
        raise ValueError(f"unknown workload kind {w.kind!r}")

    kr = round_to(k, w.dtype)
    qr = kr if q is k else round_to(q, w.dtype)
    vr = round_to(v, w.dtype)
    return {
        "q": qr, "k": kr, "v": vr,
        "q64": to_float64(qr, w.dtype), "k64": to_float64(kr, w.dtype),
        "v64": to_float64(vr, w.dtype),
        "workload": w,
    }


def batched_clouds(B: int, n: int, D: int, dtype: str = "fp16", seed: int = 0) -> dict:
    """B independent problems of the Sec. 4 benchmark shape: per problem n
    query and n key points ~ N(0, I_D) and weights v ~ N(0, 1) (C = 1),
    tau = 1/D.  Drawn q (B n rows), then k, then v, as in ``generate``;
    returns ``q`` and ``k`` of shape (B, n, D), ``v`` of shape (B, n, 1)
    (rounded, see ``round_to``) and ``tau``."""
    rng = np.random.default_rng(seed)
    q = round_to(_normal_rows(rng, B * n, D), dtype).reshape(B, n, D)
    k = round_to(_normal_rows(rng, B * n, D), dtype).reshape(B, n, D)
    v = round_to(_normal_rows(rng, B * n, 1), dtype).reshape(B, n, 1)
    return {"q": q, "k": k, "v": v, "tau": 1.0 / D, "dtype": dtype}


def to_device(a: np.ndarray, dtype: str, dev="cuda:0"):
    """Copy a ``round_to`` array to a torch device tensor of the storage dtype."""
    import torch
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def device_inputs(inp: dict, dev="cuda:0"):
    """(q, k, v) device tensors of a ``generate`` result; q is k when aliased."""
    w = inp["workload"]
    k = to_device(inp["k"], w.dtype, dev)
    q = k if inp["q"] is inp["k"] else to_device(inp["q"], w.dtype, dev)
    v = to_device(inp["v"], w.dtype, dev)
    return q, k, v


def sample_rows(M: int, count: int, seed: int = 1) -> np.ndarray:
    """Seeded, sorted subset of row indices for checks on large M."""
    if count >= M:
        return np.arange(M, dtype=np.int64)
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(M, size=count, replace=False)).astype(np.int64)


def upstream(M: int, C: int, seed: int = 0) -> np.ndarray:
    """Seeded float32 upstream gradient g (M x C) of a vector-Jacobian
    product: standard normal entries, drawn from a stream separate from the
    points' (seed offset 7919)."""
    rng = np.random.default_rng(seed + 7919)
    return np.ascontiguousarray(rng.standard_normal((M, C)).astype(np.float32))
