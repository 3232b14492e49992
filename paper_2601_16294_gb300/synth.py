"""Seeded synthetic inputs for the SFC GEMM (shared by tests and the benchmark).

This module only draws random numbers; it holds none of the method's
arithmetic.  Values are drawn in fp32 and rounded to bf16 with
round-to-nearest-even (a copy into a bf16 tensor).

Workload recipes (the paper's shapes, Sec. IV-A and IV-D):
  * ``uniform``  -- entries uniform in [-1, 1]           (square / irregular / high-K sweeps)
  * ``prefill``  -- A (activations) ~ N(0, 1), B (weights, stored K x N) ~ N(0, 0.02)
  * ``int``      -- integers in {-2, ..., 2} (exact in fp32 accumulation for K < 2^21)

Streams.  An operand (A is operand 0, B operand 1 of a pair; a lone matrix is
operand 0) is drawn in row-major order in blocks of BLOCK = 2^22 elements;
block b is drawn by its own CPU ``torch.Generator`` seeded with
``block_seed(seed, operand, b) = ((seed * 1000003 + operand) * 1000003 + b)
mod 2^63``, so the same call gives the same bits on any machine and with any
number of threads, and the blocks are drawn in parallel (the largest
operands of the workloads hold half a billion values).
``gemm_inputs_f8`` draws the same distributions and rounds them to an 8-bit
float format.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import torch

BLOCK = 1 << 22
_PRIME = 1000003


def block_seed(seed: int, operand: int, block: int) -> int:
    return ((int(seed) * _PRIME + int(operand)) * _PRIME + int(block)) % (1 << 63)


def _sample(kind: str, n: int, g: torch.Generator, std: float = 1.0) -> torch.Tensor:
    if kind == "uniform":
        return torch.rand(n, generator=g, dtype=torch.float32).mul_(2.0).sub_(1.0)
    if kind == "normal":
        return torch.randn(n, generator=g, dtype=torch.float32).mul_(std)
    if kind == "int":
        return torch.randint(-2, 3, (n,), generator=g, dtype=torch.int32).float()
    raise ValueError("unknown input kind %r" % kind)


def draw(shape, seed: int, operand: int, kind: str, std: float = 1.0, dtype=torch.bfloat16,
         threads: int | None = None) -> torch.Tensor:
    """A row-major CPU tensor of `shape` and `dtype` drawn block by block (see
    the module's description); `kind` is "uniform", "normal" (times `std`) or
    "int".  The result does not depend on `threads`."""
    out = torch.empty(tuple(shape), dtype=dtype)
    flat = out.view(-1)
    n = flat.numel()
    nb = (n + BLOCK - 1) // BLOCK

    def job(b):
        lo, hi = b * BLOCK, min(n, (b + 1) * BLOCK)
        g = torch.Generator(device="cpu").manual_seed(block_seed(seed, operand, b))
        flat[lo:hi].copy_(_sample(kind, hi - lo, g, std))

    workers = min(nb, threads or os.cpu_count() or 1)
    if workers <= 1:
        for b in range(nb):
            job(b)
    else:
        with ThreadPoolExecutor(workers) as ex:
            list(ex.map(job, range(nb)))
    return out


def uniform_bf16(shape, seed: int = 0) -> torch.Tensor:
    return draw(shape, seed, 0, "uniform")


def normal_bf16(shape, seed: int = 0, std: float = 1.0) -> torch.Tensor:
    return draw(shape, seed, 0, "normal", std)


def small_int_bf16(shape, seed: int = 0) -> torch.Tensor:
    return draw(shape, seed, 0, "int")


_KINDS = {"uniform": (("uniform", 1.0), ("uniform", 1.0)),
          "prefill": (("normal", 1.0), ("normal", 0.02)),
          "int": (("int", 1.0), ("int", 1.0))}


def gemm_inputs(M: int, N: int, K: int, kind: str = "uniform", seed: int = 0,
                lda: int | None = None, ldb: int | None = None):
    """Return (A, B) as CPU bf16 tensors, A is M x K (operand 0), B is K x N
    (operand 1), row-major.

    With ``lda`` / ``ldb`` larger than K / N the matrices are views into padded
    row-major buffers (padding filled with zeros), for shapes whose rows are
    not a multiple of 16 bytes.
    """
    if kind not in _KINDS:
        raise ValueError("unknown input kind %r" % kind)
    (ka, sa), (kb, sb) = _KINDS[kind]
    A = draw((M, K), seed, 0, ka, sa)
    B = draw((K, N), seed, 1, kb, sb)
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
    K x N.  The fp32 values of ``gemm_inputs`` with the same seed (uniform in
    [-1, 1]; prefill N(0, 1) x N(0, 0.02); integers in {-2, ..., 2}), rounded to
    the format by torch."""
    if kind not in _KINDS:
        raise ValueError("unknown input kind %r" % kind)
    (ka, sa), (kb, sb) = _KINDS[kind]
    dt = f8_dtype(fmt)
    return draw((M, K), seed, 0, ka, sa, dtype=dt), draw((K, N), seed, 1, kb, sb, dtype=dt)


def uniform_f8(shape, fmt: str = "e4m3", seed: int = 0) -> torch.Tensor:
    return draw(shape, seed, 0, "uniform", dtype=f8_dtype(fmt))


def pad8(n: int) -> int:
    """Smallest multiple of 8 elements >= n (16-byte rows for bf16)."""
    return (int(n) + 7) // 8 * 8
