"""Seeded synthetic inputs for the SFC GEMM (shared by tests and the benchmark).

This module only draws random numbers; it holds none of the method's
arithmetic.  Every generator is a CPU ``torch.Generator`` seeded explicitly, so
the same call gives the same bf16 bits on any machine.  Values are drawn in
fp32 and rounded to bf16 with round-to-nearest-even (``Tensor.to``).

Workload recipes (the paper's shapes, Sec. IV-A and IV-D):
  * ``uniform``  -- entries uniform in [-1, 1]           (square / irregular / high-K sweeps)
  * ``prefill``  -- A (activations) ~ N(0, 1), B (weights, stored K x N) ~ N(0, 0.02)
  * ``int``      -- integers in {-2, ..., 2} (exact in fp32 accumulation for K < 2^21)
For a pair (A, B) one generator draws A first, then B.  ``gemm_inputs_f8``
draws the same distributions and rounds them to an 8-bit float format.
"""
from __future__ import annotations

import torch


def _gen(seed: int) -> torch.Generator:
    return torch.Generator(device="cpu").manual_seed(int(seed))


def _uniform(shape, g) -> torch.Tensor:
    return (torch.rand(shape, generator=g, dtype=torch.float32) * 2.0 - 1.0).to(torch.bfloat16)


def _normal(shape, g, std: float) -> torch.Tensor:
    return (torch.randn(shape, generator=g, dtype=torch.float32) * std).to(torch.bfloat16)


def _small_int(shape, g) -> torch.Tensor:
    return torch.randint(-2, 3, shape, generator=g, dtype=torch.int32).to(torch.bfloat16)


def uniform_bf16(shape, seed: int = 0) -> torch.Tensor:
    return _uniform(shape, _gen(seed))


def normal_bf16(shape, seed: int = 0, std: float = 1.0) -> torch.Tensor:
    return _normal(shape, _gen(seed), std)


def small_int_bf16(shape, seed: int = 0) -> torch.Tensor:
    return _small_int(shape, _gen(seed))


def gemm_inputs(M: int, N: int, K: int, kind: str = "uniform", seed: int = 0,
                lda: int | None = None, ldb: int | None = None):
    """Return (A, B) as CPU bf16 tensors, A is M x K, B is K x N, row-major.

    With ``lda`` / ``ldb`` larger than K / N the matrices are views into padded
    row-major buffers (padding filled with zeros), for shapes whose rows are
    not a multiple of 16 bytes.
    """
    g = _gen(seed)
    if kind == "uniform":
        A = _uniform((M, K), g)
        B = _uniform((K, N), g)
    elif kind == "prefill":
        A = _normal((M, K), g, 1.0)
        B = _normal((K, N), g, 0.02)
    elif kind == "int":
        A = _small_int((M, K), g)
        B = _small_int((K, N), g)
    else:
        raise ValueError("unknown input kind %r" % kind)
    if lda is not None and lda != K:
        buf = torch.zeros((M, lda), dtype=torch.bfloat16)
        buf[:, :K] = A
        A = buf[:, :K]
    if ldb is not None and ldb != N:
        buf = torch.zeros((K, ldb), dtype=torch.bfloat16)
        buf[:, :N] = B
        B = buf[:, :N]
    return A, B


def f8_dtype(fmt: str):
    """torch dtype of an 8-bit float format ("e4m3" or "e5m2")."""
    return {"e4m3": torch.float8_e4m3fn, "e5m2": torch.float8_e5m2}[fmt]


def gemm_inputs_f8(M: int, N: int, K: int, fmt: str = "e4m3", kind: str = "uniform", seed: int = 0):
    """(A, B) as CPU 8-bit float tensors of format ``fmt``: A is M x K, B is
    K x N.  Values are drawn in fp32 with the distributions of ``gemm_inputs``
    (uniform in [-1, 1]; prefill N(0, 1) x N(0, 0.02); integers in {-2, ..., 2})
    and rounded to the format by torch."""
    g = _gen(seed)
    if kind == "uniform":
        A = torch.rand((M, K), generator=g, dtype=torch.float32) * 2.0 - 1.0
        B = torch.rand((K, N), generator=g, dtype=torch.float32) * 2.0 - 1.0
    elif kind == "prefill":
        A = torch.randn((M, K), generator=g, dtype=torch.float32)
        B = torch.randn((K, N), generator=g, dtype=torch.float32) * 0.02
    elif kind == "int":
        A = torch.randint(-2, 3, (M, K), generator=g, dtype=torch.int32).float()
        B = torch.randint(-2, 3, (K, N), generator=g, dtype=torch.int32).float()
    else:
        raise ValueError("unknown input kind %r" % kind)
    dt = f8_dtype(fmt)
    return A.to(dt), B.to(dt)


def uniform_f8(shape, fmt: str = "e4m3", seed: int = 0) -> torch.Tensor:
    return (torch.rand(shape, generator=_gen(seed), dtype=torch.float32) * 2.0 - 1.0).to(f8_dtype(fmt))


def pad8(n: int) -> int:
    """Smallest multiple of 8 elements >= n (16-byte rows for bf16)."""
    return (int(n) + 7) // 8 * 8
