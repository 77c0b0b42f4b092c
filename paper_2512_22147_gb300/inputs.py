"""Seeded synthetic inputs for the dual matrix-vector product.

This module holds no arithmetic of the method: it only draws random operands
and names the workloads.  Both the CUDA path (tests, benchmark) and the CPU
oracle take their inputs from here, so both sides see the same numbers.

Recipe: one ``torch.Generator`` on the target device, seeded with the
workload's seed, fills A, then p, then r, in that order.  Floats are drawn
with ``uniform_(-1, 1)`` (half-open [-1, 1)) or ``normal_(0, 1)``; integers
with ``randint(-8, 9)`` (inclusive [-8, 8]).  Batched workloads draw each
operand for the whole batch in one call.  Padding columns (``lda > N``) are
filled with a sentinel the kernels must never read: NaN for floats,
INT32_MIN for integers.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import torch

DTYPES = {"f32": torch.float32, "f64": torch.float64, "i32": torch.int32}
OUT_DTYPES = {"f32": torch.float32, "f64": torch.float64, "i32": torch.int64}
ELEM_BYTES = {"f32": 4, "f64": 8, "i32": 4}
OUT_BYTES = {"f32": 4, "f64": 8, "i32": 8}


@dataclass(frozen=True)
class Workload:
    """One synthetic problem (or strided batch of problems)."""

    name: str
    dtype: str          # "f32" | "f64" | "i32"
    M: int
    N: int
    lda: int
    dist: str           # "uniform" | "normal" | "int8"
    seed: int
    batch: int = 0      # 0 = single problem; >= 1 = strided batch
    op: str = "bicg"    # "bicg" (dual product) | "gesummv" | "atax" | "gemver"
    update_a: bool = False  # gemver: A_hat written over A

    @property
    def batched(self) -> bool:
        return self.batch > 0

    @property
    def nbatch(self) -> int:
        return max(1, self.batch)

    def bytes_counted(self) -> int:
        """Bytes of the logical matrices (padding excluded) read once, of the
        input vectors and of the outputs: the numerator of the
        effective-bandwidth metric.  Dual product: A, p, r, q, s.  GESUMMV:
        A, B, x, y.  ATAX: A (once: the least any algorithm must move), x, y.
        GEMVER: A (and, with update_a, A_hat written), the six input vectors,
        x and w read and written."""
        e, o = ELEM_BYTES[self.dtype], OUT_BYTES[self.dtype]
        if self.op == "gesummv":
            return 2 * self.M * self.N * e + self.N * e + self.M * o
        if self.op == "atax":
            return self.M * self.N * e + self.N * e + self.N * o
        if self.op == "gemver":   # A once (and A_hat written); u1 v1 u2 v2 y z read; x w in and out
            mat = (2 if self.update_a else 1) * self.M * self.N * e
            return mat + 3 * (self.M + self.N) * e + (self.M + self.N) * o
        per = (self.M * self.N * e + (self.M + self.N) * e
               + (self.M + self.N) * o)
        return per * self.nbatch

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads: a small square problem, a 1 GiB square fp32 matrix, a
# 2 GiB tall-skinny fp64 matrix, a wide int32 matrix with a padded, ragged
# row, and a strided batch of 256 square fp32 problems (4 GiB).
WORKLOADS = {
    w.name: w for w in (
        Workload("f32_1024x1024", "f32", 1024, 1024, 1024, "uniform", 0),
        Workload("f32_16384x16384", "f32", 16384, 16384, 16384, "uniform", 1),
        Workload("f64_65536x4096", "f64", 65536, 4096, 4096, "normal", 2),
        Workload("i32_4001x100003_lda100008", "i32", 4001, 100003, 100008,
                 "int8", 3),
        Workload("f32_batch256_2048x2048", "f32", 2048, 2048, 2048, "uniform",
                 4, batch=256),
    )
}


# Workloads of the further PolyBench kernels built on the same products
# (GESUMMV, ATAX and GEMVER, Table 1), sized like the dual product's square
# fp32 workload so that every matrix is far larger than L2.
OP_WORKLOADS = {
    w.name: w for w in (
        Workload("gesummv_f32_16384x16384", "f32", 16384, 16384, 16384, "uniform", 5,
                 op="gesummv"),
        Workload("gesummv_f64_8192x8192", "f64", 8192, 8192, 8192, "normal", 6, op="gesummv"),
        Workload("atax_f32_16384x16384", "f32", 16384, 16384, 16384, "uniform", 7, op="atax"),
        Workload("atax_f64_16384x8192", "f64", 16384, 8192, 8192, "normal", 8, op="atax"),
        Workload("gemver_f32_16384x16384", "f32", 16384, 16384, 16384, "uniform", 9,
                 op="gemver"),
        Workload("gemver_f64_8192x8192", "f64", 8192, 8192, 8192, "normal", 10, op="gemver"),
        Workload("gemver_update_f64_8192x8192", "f64", 8192, 8192, 8192, "normal", 11,
                 op="gemver", update_a=True),
        Workload("gemver_update_f32_16384x16384", "f32", 16384, 16384, 16384, "uniform", 12,
                 op="gemver", update_a=True),
    )
}


def _sentinel(dtype: str):
    return float("nan") if dtype != "i32" else -(2 ** 31)


def _fill(t: torch.Tensor, dist: str, g: torch.Generator) -> None:
    if dist == "uniform":
        t.uniform_(-1.0, 1.0, generator=g)
    elif dist == "normal":
        t.normal_(0.0, 1.0, generator=g)
    elif dist == "int8":
        t.copy_(torch.randint(-8, 9, t.shape, generator=g, device=t.device,
                              dtype=t.dtype))
    else:
        raise ValueError(f"unknown distribution {dist!r}")


def generate(w: Workload, device: str | torch.device = "cpu"):
    """Return ``(A, p, r)`` on ``device``.

    ``A`` has shape ``(M, lda)`` (or ``(batch, M, lda)``) and holds the
    matrix in its first N columns and the padding sentinel after them.
    ``p`` is ``(N,)`` / ``(batch, N)`` and ``r`` is ``(M,)`` /
    ``(batch, M)``.
    """
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed)
    t = DTYPES[w.dtype]
    lead = (w.batch,) if w.batched else ()
    A = torch.empty(lead + (w.M, w.lda), dtype=t, device=dev)
    if w.lda > w.N:
        A[..., w.N:] = _sentinel(w.dtype)
    view = A[..., : w.N]
    if view.numel():
        if view.is_contiguous():
            _fill(view, w.dist, g)
        else:
            tmp = torch.empty(view.shape, dtype=t, device=dev)
            _fill(tmp, w.dist, g)
            view.copy_(tmp)
            del tmp
    p = torch.empty(lead + (w.N,), dtype=t, device=dev)
    r = torch.empty(lead + (w.M,), dtype=t, device=dev)
    if p.numel():
        _fill(p, w.dist, g)
    if r.numel():
        _fill(r, w.dist, g)
    return A, p, r


def empty_outputs(w: Workload, device: str | torch.device = "cpu"):
    """Output buffers ``(q, s)`` of the right dtype and shape."""
    t = OUT_DTYPES[w.dtype]
    lead = (w.batch,) if w.batched else ()
    q = torch.empty(lead + (w.M,), dtype=t, device=device)
    s = torch.empty(lead + (w.N,), dtype=t, device=device)
    return q, s


def _matrix(w: Workload, g: torch.Generator, dev) -> torch.Tensor:
    A = torch.empty((w.M, w.lda), dtype=DTYPES[w.dtype], device=dev)
    if w.lda > w.N:
        A[:, w.N:] = _sentinel(w.dtype)
    view = A[:, : w.N]
    if view.numel():
        if view.is_contiguous():
            _fill(view, w.dist, g)
        else:
            tmp = torch.empty(view.shape, dtype=A.dtype, device=dev)
            _fill(tmp, w.dist, g)
            view.copy_(tmp)
    return A


def _vector(n: int, w: Workload, g: torch.Generator, dev) -> torch.Tensor:
    v = torch.empty(n, dtype=DTYPES[w.dtype], device=dev)
    if n:
        _fill(v, w.dist, g)
    return v


def generate_gesummv(w: Workload, device: str | torch.device = "cpu"):
    """``(A, B, x)`` for GESUMMV: one generator fills A, then B, then x."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed)
    A = _matrix(w, g, dev)
    B = _matrix(w, g, dev)
    return A, B, _vector(w.N, w, g, dev)


def generate_atax(w: Workload, device: str | torch.device = "cpu"):
    """``(A, x)`` for ATAX: one generator fills A, then x."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed)
    A = _matrix(w, g, dev)
    return A, _vector(w.N, w, g, dev)


def generate_gemver(w: Workload, device: str | torch.device = "cpu"):
    """``(A, u1, v1, u2, v2, w, x, y, z)`` for GEMVER: one generator fills A,
    then the vectors in that order (u's, w, y of length M; v's, x, z of
    length N)."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed)
    A = _matrix(w, g, dev)
    u1 = _vector(w.M, w, g, dev)
    v1 = _vector(w.N, w, g, dev)
    u2 = _vector(w.M, w, g, dev)
    v2 = _vector(w.N, w, g, dev)
    wv = _vector(w.M, w, g, dev)
    x = _vector(w.N, w, g, dev)
    y = _vector(w.M, w, g, dev)
    z = _vector(w.N, w, g, dev)
    return A, u1, v1, u2, v2, wv, x, y, z
