"""Tensor-level entry point: ``dualmv(A, p, r)`` on CUDA torch tensors.

PyTorch only provides device memory and the current stream; the work runs
in the CUDA library through the C ABI (``_binding``).

Shapes (BICG, Tables 1-2 of the paper: q = A p, s = A^T r):
  single:  A (M, N) with A.stride(1) == 1 and leading dimension A.stride(0);
           p (N,), r (M,)  ->  q (M,), s (N,)
  batched: A (B, M, N) with A.stride(2) == 1; lda = A.stride(1),
           strideA = A.stride(0); p (B, N) or (N,) (shared), r (B, M) or
           (M,) (shared)  ->  q (B, M), s (B, N)
dtype float32 -> float32 outputs, float64 -> float64, int32 -> int64
(exact modulo 2^64).  A may be a column slice of a wider buffer (its row
stride is the leading dimension).
"""
from __future__ import annotations

import torch

from . import _binding as B

B_ = B  # the binding, where a parameter is named B

_OUT = {torch.float32: torch.float32, torch.float64: torch.float64,
        torch.int32: torch.int64}
_TAG = {torch.float32: "f32", torch.float64: "f64", torch.int32: "i32"}


def _vec_stride(v: torch.Tensor, length: int, batch: int, name: str) -> int:
    """Element stride between problems for a per-problem vector (0 = shared)."""
    if v.dim() == 1:
        if v.shape[0] != length or (length > 1 and v.stride(0) != 1):
            raise ValueError(f"{name} must be a contiguous vector of length {length}")
        return 0
    if v.dim() != 2 or v.shape[0] != batch or v.shape[1] != length:
        raise ValueError(f"{name} must have shape ({batch}, {length})")
    if length > 1 and v.stride(1) != 1:
        raise ValueError(f"{name} rows must be contiguous")
    return v.stride(0)


# Per input dtype: (output dtype, single-problem entry, batched entry, tag).
_ENTRY: dict = {}

# The current device and the raw handle of its current stream, as plain
# integers when torch has these bindings (building a torch.cuda.Stream
# object costs microseconds a call); else through the public API.
_get_device = getattr(torch._C, "_cuda_getDevice", None) or torch.cuda.current_device
_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _current_stream_handle(dev_idx: int) -> int:
    if _raw_stream is not None:
        return _raw_stream(dev_idx)
    return torch.cuda.current_stream(dev_idx).cuda_stream


def _call_on(dev_idx: int, stream, fn, *args):
    """fn(*args, stream handle) with device dev_idx current (switched to only
    when it is not); stream None means that device's current stream."""
    ctx = torch.cuda.device(dev_idx) if dev_idx != _get_device() else None
    if ctx is not None:
        ctx.__enter__()
    try:
        h = _current_stream_handle(dev_idx) if stream is None else stream.cuda_stream
        return fn(*args, h)
    finally:
        if ctx is not None:
            ctx.__exit__(None, None, None)


def _entry(dtype):
    e = _ENTRY.get(dtype)
    if e is None:
        tag = _TAG.get(dtype)
        if tag is None:
            raise TypeError(f"unsupported dtype {dtype}; use float32, float64 or int32")
        e = (_OUT[dtype], getattr(B, f"dualmv_{tag}"),
             getattr(B, f"dualmv_{tag}_strided_batched"), tag)
        _ENTRY[dtype] = e
    return e


def dualmv(A: torch.Tensor, p: torch.Tensor, r: torch.Tensor,
           q: torch.Tensor | None = None, s: torch.Tensor | None = None,
           stream: torch.cuda.Stream | None = None):
    """Compute ``q = A p`` and ``s = A^T r`` (per problem when batched).

    Returns ``(q, s)``; pass ``q``/``s`` to write into existing buffers.
    Runs asynchronously on ``stream`` (default: the current stream of A's
    device).
    """
    dt = A.dtype
    out_t, fn_single, fn_batched, tag = _entry(dt)
    if not A.is_cuda:
        raise ValueError("A must be a CUDA tensor (the library has no CPU path)")
    dev_idx = A.get_device()
    for t, n in ((p, "p"), (r, "r")):
        if t.dtype != dt or t.get_device() != dev_idx:
            raise ValueError(f"{n} must match A's dtype and device")
    nd = A.dim()
    if nd not in (2, 3):
        raise ValueError("A must be 2-D (M, N) or 3-D (B, M, N)")
    batched = nd == 3
    shape, strides = A.shape, A.stride()
    Bn = shape[0] if batched else 1
    M, N = shape[-2], shape[-1]
    if N > 1 and strides[-1] != 1:
        raise ValueError("A's last dimension must be contiguous")
    if M > 1 and strides[-2] < N:
        raise ValueError("A's rows overlap (row stride smaller than N)")
    lda = max(strides[-2], N, 1) if M > 1 else max(N, 1)
    shape_q = (Bn, M) if batched else (M,)
    shape_s = (Bn, N) if batched else (N,)
    if q is None:
        q = torch.empty(shape_q, dtype=out_t, device=A.device)
    elif q.dtype != out_t or tuple(q.shape) != shape_q:
        raise ValueError(f"q must be {out_t} of shape {shape_q}")
    if s is None:
        s = torch.empty(shape_s, dtype=out_t, device=A.device)
    elif s.dtype != out_t or tuple(s.shape) != shape_s:
        raise ValueError(f"s must be {out_t} of shape {shape_s}")
    if batched:
        sP = _vec_stride(p, N, Bn, "p")
        sR = _vec_stride(r, M, Bn, "r")
        sQ = _vec_stride(q, M, Bn, "q") if q.dim() == 2 else M
        sS = _vec_stride(s, N, Bn, "s") if s.dim() == 2 else N
        rc = _call_on(dev_idx, stream, fn_batched, M, N, A.data_ptr(), lda, strides[0],
                      p.data_ptr(), sP, r.data_ptr(), sR, q.data_ptr(), sQ, s.data_ptr(), sS,
                      Bn)
    else:
        if p.dim() != 1 or r.dim() != 1 or p.shape[0] != N or r.shape[0] != M or \
                not (p.is_contiguous() and r.is_contiguous()):
            raise ValueError(f"p and r must be contiguous vectors of lengths {N} and {M}")
        if not (q.is_contiguous() and s.is_contiguous()):
            raise ValueError("q and s must be contiguous")
        rc = _call_on(dev_idx, stream, fn_single, M, N, A.data_ptr(), lda, p.data_ptr(),
                      r.data_ptr(), q.data_ptr(), s.data_ptr())
    if rc != B.DUALMV_SUCCESS:
        raise B.DualmvError(rc, f"dualmv_{tag}")
    return q, s


def device_fault(stream: torch.cuda.Stream | None = None) -> int:
    """Synchronise ``stream`` and return (and clear) the device fault status."""
    h = _current_stream_handle(_get_device()) if stream is None else stream.cuda_stream
    return B.dualmv_device_fault(h)


def _matrix(A: torch.Tensor, name: str):
    if A.dim() != 2:
        raise ValueError(f"{name} must be 2-D")
    M, N = A.shape
    if N > 1 and A.stride(1) != 1:
        raise ValueError(f"{name}'s last dimension must be contiguous")
    if M > 1 and A.stride(0) < N:
        raise ValueError(f"{name}'s rows overlap")
    return M, N, (max(A.stride(0), N, 1) if M > 1 else max(N, 1))


def _vector(v: torch.Tensor, n: int, like: torch.Tensor, name: str):
    if v.dtype != like.dtype or v.device != like.device or v.dim() != 1 or v.shape[0] != n:
        raise ValueError(f"{name} must be a {like.dtype} vector of length {n} on {like.device}")
    if n > 1 and v.stride(0) != 1:
        raise ValueError(f"{name} must be contiguous")


def gesummv(A: torch.Tensor, B: torch.Tensor, x: torch.Tensor, alpha: float = 1.0,
            beta: float = 1.0, y: torch.Tensor | None = None,
            stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """GESUMMV (Table 1 / Table 2): ``y = alpha * (A x) + beta * (B x)``.

    A and B are M x N float32/float64 CUDA tensors (unit column stride)."""
    tag = {torch.float32: "f32", torch.float64: "f64"}.get(A.dtype)
    if tag is None or not A.is_cuda:
        raise TypeError("A must be a float32 or float64 CUDA tensor")
    M, N, lda = _matrix(A, "A")
    MB, NB, ldb = _matrix(B, "B")
    if (MB, NB) != (M, N) or B.dtype != A.dtype or B.device != A.device:
        raise ValueError("B must match A's shape, dtype and device")
    _vector(x, N, A, "x")
    if y is None:
        y = torch.empty(M, dtype=A.dtype, device=A.device)
    _vector(y, M, A, "y")
    rc = _call_on(A.get_device(), stream, getattr(B_, f"dualmv_gesummv_{tag}"), M, N, alpha,
                  A.data_ptr(), lda, beta, B.data_ptr(), ldb, x.data_ptr(), y.data_ptr())
    if rc != B_.DUALMV_SUCCESS:
        raise B_.DualmvError(rc, f"dualmv_gesummv_{tag}")
    return y


def atax(A: torch.Tensor, x: torch.Tensor, y: torch.Tensor | None = None,
         stream: torch.cuda.Stream | None = None) -> torch.Tensor:
    """ATAX (Table 1): ``y = A^T (A x)`` for an M x N float32/float64 A."""
    tag = {torch.float32: "f32", torch.float64: "f64"}.get(A.dtype)
    if tag is None or not A.is_cuda:
        raise TypeError("A must be a float32 or float64 CUDA tensor")
    M, N, lda = _matrix(A, "A")
    _vector(x, N, A, "x")
    if y is None:
        y = torch.empty(N, dtype=A.dtype, device=A.device)
    _vector(y, N, A, "y")
    rc = _call_on(A.get_device(), stream, getattr(B_, f"dualmv_atax_{tag}"), M, N,
                  A.data_ptr(), lda, x.data_ptr(), y.data_ptr())
    if rc != B_.DUALMV_SUCCESS:
        raise B_.DualmvError(rc, f"dualmv_atax_{tag}")
    return y


def gemver(A: torch.Tensor, u1: torch.Tensor, v1: torch.Tensor, u2: torch.Tensor,
           v2: torch.Tensor, w: torch.Tensor, x: torch.Tensor, y: torch.Tensor,
           z: torch.Tensor, alpha: float = 1.0, beta: float = 1.0, update_A: bool = False,
           stream: torch.cuda.Stream | None = None):
    """GEMVER (Table 1 / Table 2): A_hat = A + u1 v1^T + u2 v2^T;
    x = x + beta A_hat^T y + z;  w = w + alpha A_hat x.

    x and w are updated in place (and A too when ``update_A``); returns
    ``(w, x)``.  A is M x N; u1, u2, w, y have M elements; v1, v2, x, z N."""
    tag = {torch.float32: "f32", torch.float64: "f64"}.get(A.dtype)
    if tag is None or not A.is_cuda:
        raise TypeError("A must be a float32 or float64 CUDA tensor")
    M, N, lda = _matrix(A, "A")
    for v, n, name in ((u1, M, "u1"), (u2, M, "u2"), (w, M, "w"), (y, M, "y"),
                       (v1, N, "v1"), (v2, N, "v2"), (x, N, "x"), (z, N, "z")):
        _vector(v, n, A, name)
    rc = _call_on(A.get_device(), stream, getattr(B_, f"dualmv_gemver_{tag}"), M, N, alpha,
                  beta, A.data_ptr(), lda, int(bool(update_A)), u1.data_ptr(), v1.data_ptr(),
                  u2.data_ptr(), v2.data_ptr(), w.data_ptr(), x.data_ptr(), y.data_ptr(),
                  z.data_ptr())
    if rc != B_.DUALMV_SUCCESS:
        raise B_.DualmvError(rc, f"dualmv_gemver_{tag}")
    return w, x


_DTYPE_CODE = {torch.float32: B.DUALMV_DTYPE_F32, torch.float64: B.DUALMV_DTYPE_F64,
               torch.int32: B.DUALMV_DTYPE_I32}


def variants(dtype: torch.dtype) -> list[dict]:
    """The compiled kernel variants for ``dtype`` (entry 0 is the default)."""
    code = _DTYPE_CODE[dtype]
    out = []
    for i in range(B.dualmv_variant_count(code)):
        v = B.dualmv_variant_info(code, i)
        out.append({f: getattr(v, f) for f, _ in v._fields_})
    return out


def tune(A: torch.Tensor, p: torch.Tensor, r: torch.Tensor, q: torch.Tensor | None = None,
         s: torch.Tensor | None = None, repeats: int = 30, trim: int = 3, max_rounds: int = 4,
         candidates: int = 4, min_gain: float = 0.01, flush_l2: bool = True,
         stream: torch.cuda.Stream | None = None) -> dict:
    """Tune the kernel variant for this problem's shape (Section 3.2: Eq. 3
    scores, the Eq. 4 equivalence gate, the Eq. 5 choice); later ``dualmv``
    calls of the same shape use the result.  A is one (M, N) problem or a
    strided batch (B, M, N) with p (B, N) and r (B, M), as ``dualmv`` takes
    them.  Blocks until done.  Returns the tuner's report; q and s hold the
    chosen variant's outputs."""
    if A.dtype not in _TAG or A.dim() not in (2, 3):
        raise ValueError("tune takes a 2-D (or 3-D batched) float32, float64 or int32 A")
    batched = A.dim() == 3
    Bn = A.shape[0] if batched else 1
    M, N = A.shape[-2], A.shape[-1]
    if N > 1 and A.stride(-1) != 1:
        raise ValueError("A's last dimension must be contiguous")
    lda = max(A.stride(-2), N, 1) if M > 1 else max(N, 1)
    out_t = _OUT[A.dtype]
    if q is None:
        q = torch.empty((Bn, M) if batched else M, dtype=out_t, device=A.device)
    if s is None:
        s = torch.empty((Bn, N) if batched else N, dtype=out_t, device=A.device)
    for t_, n in ((p, "p"), (r, "r"), (q, "q"), (s, "s")):
        dt = A.dtype if n in ("p", "r") else out_t
        if t_.dtype != dt or t_.device != A.device:
            raise ValueError(f"{n} must be of dtype {dt} on A's device")
    if batched:   # per-problem vectors (B, n), or p, r shared by every problem
        sP, sR = _vec_stride(p, N, Bn, "p"), _vec_stride(r, M, Bn, "r")
        if q.dim() != 2 or s.dim() != 2:
            raise ValueError(f"q and s must have shapes ({Bn}, {M}) and ({Bn}, {N})")
        sQ, sS = _vec_stride(q, M, Bn, "q"), _vec_stride(s, N, Bn, "s")
    elif not all(t_.dim() == 1 and t_.is_contiguous() for t_ in (p, r, q, s)):
        raise ValueError("p, r, q and s must be contiguous vectors")
    cfg = B.TuneConfig(repeats, trim, max_rounds, candidates, min_gain, int(flush_l2))
    res = B.TuneResult()
    strm = stream if stream is not None else torch.cuda.current_stream(A.device)
    if batched:
        fn = getattr(B, f"dualmv_tune_{_TAG[A.dtype]}_strided_batched")
        rc = fn(M, N, A.data_ptr(), lda, A.stride(0), p.data_ptr(), sP, r.data_ptr(), sR,
                q.data_ptr(), sQ, s.data_ptr(), sS, Bn, cfg, res, strm.cuda_stream)
    else:
        fn = getattr(B, f"dualmv_tune_{_TAG[A.dtype]}")
        rc = fn(M, N, A.data_ptr(), lda, p.data_ptr(), r.data_ptr(), q.data_ptr(),
                s.data_ptr(), cfg, res, strm.cuda_stream)
    if rc != B.DUALMV_SUCCESS:
        raise B.DualmvError(rc, "dualmv_tune")
    rep = {f: getattr(res, f) for f, _ in res._fields_
           if f not in ("trace", "trace_len")}
    rep["trace"] = [{"index": st.index, "round": st.round, "feasible": bool(st.feasible),
                     "ms": st.ms, "fe": st.fe} for st in res.trace[:res.trace_len]]
    rep["q"], rep["s"] = q, s
    return rep


def tune_pass(A: torch.Tensor, x: torch.Tensor, pass_: str = "rows",
              out: torch.Tensor | None = None, repeats: int = 30, trim: int = 3,
              max_rounds: int = 4, candidates: int = 4, min_gain: float = 0.01,
              flush_l2: bool = True, stream: torch.cuda.Stream | None = None) -> dict:
    """Tune one single-sided pass for A's shape: ``pass_="rows"`` computes
    ``out = A x`` (the passes of GESUMMV and GEMVER's rows side),
    ``pass_="cols"`` computes ``out = A^T x`` (GEMVER's columns pass); later
    forward passes of the same shape use the result.  A is one float32 or
    float64 (M, N) problem.  Blocks until done.  Returns the tuner's report;
    ``out`` holds the chosen variant's result."""
    if A.dtype not in (torch.float32, torch.float64) or A.dim() != 2:
        raise ValueError("tune_pass takes a 2-D float32 or float64 A")
    if pass_ not in ("rows", "cols"):
        raise ValueError('pass_ must be "rows" or "cols"')
    M, N, lda = _matrix(A, "A")
    rows = pass_ == "rows"
    nx, nout = (N, M) if rows else (M, N)
    if out is None:
        out = torch.empty(nout, dtype=A.dtype, device=A.device)
    for t_, n, ln in ((x, "x", nx), (out, "out", nout)):
        if t_.dtype != A.dtype or t_.device != A.device or t_.dim() != 1 or \
                not t_.is_contiguous() or t_.numel() != ln:
            raise ValueError(f"{n} must be a contiguous {A.dtype} vector of length {ln} "
                             "on A's device")
    cfg = B.TuneConfig(repeats, trim, max_rounds, candidates, min_gain, int(flush_l2))
    res = B.TuneResult()
    strm = stream if stream is not None else torch.cuda.current_stream(A.device)
    fn = getattr(B, f"dualmv_tune_pass_{_TAG[A.dtype]}")
    rc = fn(M, N, A.data_ptr(), lda, B.DUALMV_PASS_ROWS if rows else B.DUALMV_PASS_COLS,
            x.data_ptr(), out.data_ptr(), cfg, res, strm.cuda_stream)
    if rc != B.DUALMV_SUCCESS:
        raise B.DualmvError(rc, "dualmv_tune_pass")
    rep = {f: getattr(res, f) for f, _ in res._fields_
           if f not in ("trace", "trace_len")}
    rep["trace"] = [{"index": st.index, "round": st.round, "feasible": bool(st.feasible),
                     "ms": st.ms, "fe": st.fe} for st in res.trace[:res.trace_len]]
    rep["out"] = out
    return rep
