"""PyTorch-facing wrapper of the C ABI: CSR matrices in torch device memory.

PyTorch provides device memory and the current stream; the product itself is
computed entirely by libws_spgemm.so through the four ABI calls:

    ws_csr_create(A), ws_csr_create(B), ws_csr_create(C)    -- borrow arrays
    nnz = ws_spgemm_symbolic(A, B, C)   -- C.rowptr + nnz(C) (the declare step)
    allocate C.colidx[nnz], C.vals[nnz] with torch
    ws_spgemm_numeric(A, B, C, ...)     -- fill C (the update step)
    ws_csr_destroy(...)
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

from . import _abi


_DTYPES = {torch.float32: _abi.WS_F32, torch.float64: _abi.WS_F64}


def _stream_handle(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


@dataclass
class DeviceCSR:
    """CSR matrix whose arrays live in torch CUDA tensors."""

    nrows: int
    ncols: int
    rowptr: torch.Tensor  # int64 [nrows + 1]
    colidx: torch.Tensor  # int32 [nnz]
    vals: torch.Tensor  # float32 / float64 [nnz]

    @property
    def nnz(self) -> int:
        return int(self.colidx.numel())

    @property
    def dtype(self) -> torch.dtype:
        return self.vals.dtype

    @classmethod
    def from_host(cls, M, device="cuda", non_blocking: bool = False) -> "DeviceCSR":
        """Copies a host CSR (numpy arrays rowptr/colidx/vals) to the device."""
        def put(a, dt):
            t = torch.from_numpy(np.ascontiguousarray(a)).to(dt)
            return t.to(device, non_blocking=non_blocking)
        return cls(int(M.nrows), int(M.ncols), put(M.rowptr, torch.int64), put(M.colidx, torch.int32),
                   put(M.vals, torch.float32 if np.dtype(M.vals.dtype) == np.float32 else torch.float64))

    def to_host(self):
        return (self.rowptr.cpu().numpy(), self.colidx.cpu().numpy(), self.vals.cpu().numpy())

    def _handle(self, validate: bool, stream: int) -> int:
        if self.dtype not in _DTYPES:
            raise TypeError(f"values must be float32 or float64, got {self.dtype}")
        for t, dt in ((self.rowptr, torch.int64), (self.colidx, torch.int32)):
            if t.dtype != dt or not t.is_cuda or not t.is_contiguous():
                raise TypeError("rowptr/colidx must be contiguous CUDA int64/int32 tensors")
        if self.rowptr.numel() != self.nrows + 1:
            raise ValueError("rowptr must have nrows + 1 entries")
        nnz = self.nnz
        return _abi.ws_csr_create(self.nrows, self.ncols, nnz, self.rowptr.data_ptr(),
                                  self.colidx.data_ptr() if nnz else 0, self.vals.data_ptr() if nnz else 0,
                                  _DTYPES[self.dtype], validate, stream)


class SpGEMM:
    """A reusable product C = A*B: handles and the row plan persist across calls.

    ``symbolic()`` returns nnz(C) (and synchronises the stream), ``numeric()``
    queues the value pass and returns C as a :class:`DeviceCSR`.
    """

    def __init__(self, A: DeviceCSR, B: DeviceCSR, validate: bool = False, stream=None):
        if A.dtype != B.dtype:
            raise TypeError("A and B must have the same value dtype")
        self.A, self.B = A, B
        s = _stream_handle(stream)
        self._hA = self._hB = self._hC = None
        self.device = A.rowptr.device
        self._hA = A._handle(validate, s)
        self._hB = B._handle(validate, s)
        self.c_rowptr = torch.empty(A.nrows + 1, dtype=torch.int64, device=self.device)
        self._hC = _abi.ws_csr_create(A.nrows, B.ncols, 0, self.c_rowptr.data_ptr(), 0, 0,
                                      _DTYPES[A.dtype], False, s)
        self.nnz = None

    def symbolic(self, stream=None) -> int:
        self.nnz = _abi.ws_spgemm_symbolic(self._hA, self._hB, self._hC, _stream_handle(stream))
        return self.nnz

    def numeric(self, out: DeviceCSR | None = None, stream=None) -> DeviceCSR:
        if self.nnz is None:
            raise RuntimeError("symbolic() must run before numeric()")
        if out is None or out.nnz != self.nnz:
            colidx = torch.empty(self.nnz, dtype=torch.int32, device=self.device)
            vals = torch.empty(self.nnz, dtype=self.A.dtype, device=self.device)
            out = DeviceCSR(self.A.nrows, self.B.ncols, self.c_rowptr, colidx, vals)
        _abi.ws_spgemm_numeric(self._hA, self._hB, self._hC, out.colidx.data_ptr() if self.nnz else 0,
                               out.vals.data_ptr() if self.nnz else 0, _stream_handle(stream))
        return out

    def wait(self, stream=None) -> None:
        _abi.ws_spgemm_wait(self._hC, _stream_handle(stream))

    def plan_info(self) -> dict:
        return _abi.ws_spgemm_plan_info(self._hC)

    def close(self) -> None:
        for name in ("_hC", "_hB", "_hA"):
            h = getattr(self, name, None)
            if h:
                _abi.ws_csr_destroy(h)
                setattr(self, name, None)

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Ewise:
    """A reusable elementwise operation C = A op B (op "add": SpAdd on the
    union of the patterns; op "mul": Hadamard product on their intersection).

    ``symbolic()`` returns nnz(C) (and synchronises the stream), ``numeric()``
    queues the value pass and returns C as a :class:`DeviceCSR`.
    """

    def __init__(self, A: DeviceCSR, B: DeviceCSR, op: str = "add", validate: bool = False, stream=None):
        if A.dtype != B.dtype:
            raise TypeError("A and B must have the same value dtype")
        if op not in _abi.EWISE_OPS:
            raise ValueError(f"op must be one of {tuple(_abi.EWISE_OPS)}, got {op!r}")
        self.A, self.B, self.op = A, B, op
        s = _stream_handle(stream)
        self._hA = self._hB = self._hC = None
        self.device = A.rowptr.device
        self._hA = A._handle(validate, s)
        self._hB = B._handle(validate, s)
        self.c_rowptr = torch.empty(A.nrows + 1, dtype=torch.int64, device=self.device)
        self._hC = _abi.ws_csr_create(A.nrows, A.ncols, 0, self.c_rowptr.data_ptr(), 0, 0,
                                      _DTYPES[A.dtype], False, s)
        self.nnz = None

    def symbolic(self, stream=None) -> int:
        self.nnz = _abi.ws_ewise_symbolic(self._hA, self._hB, self._hC, self.op, _stream_handle(stream))
        return self.nnz

    def numeric(self, out: DeviceCSR | None = None, stream=None) -> DeviceCSR:
        if self.nnz is None:
            raise RuntimeError("symbolic() must run before numeric()")
        if out is None or out.nnz != self.nnz:
            colidx = torch.empty(self.nnz, dtype=torch.int32, device=self.device)
            vals = torch.empty(self.nnz, dtype=self.A.dtype, device=self.device)
            out = DeviceCSR(self.A.nrows, self.A.ncols, self.c_rowptr, colidx, vals)
        _abi.ws_ewise_numeric(self._hA, self._hB, self._hC, out.colidx.data_ptr() if self.nnz else 0,
                              out.vals.data_ptr() if self.nnz else 0, _stream_handle(stream))
        return out

    wait = SpGEMM.wait
    plan_info = SpGEMM.plan_info
    close = SpGEMM.close
    __enter__ = SpGEMM.__enter__
    __exit__ = SpGEMM.__exit__
    __del__ = SpGEMM.__del__


def ewise(A: DeviceCSR, B: DeviceCSR, op: str = "add", validate: bool = False, stream=None) -> DeviceCSR:
    """C = A + B (op "add") or C = A .* B (op "mul") for CSR matrices of one shape on the GPU."""
    with Ewise(A, B, op, validate=validate, stream=stream) as e:
        e.symbolic(stream)
        C = e.numeric(stream=stream)
        e.wait(stream)
    return C


class SpMSpV:
    """A reusable sparse matrix - sparse vector product y = A x, with A given by
    columns: ``At`` is the DeviceCSR of A^T (row j of ``At`` = column j of A).

    ``__call__(x_idx, x_vals)`` returns (y_idx, y_vals) as CUDA tensors (views
    of capacity-m buffers kept by the object); it synchronises the stream.
    """

    def __init__(self, At: DeviceCSR, validate: bool = False, stream=None):
        self.At = At
        self._h = None
        self._h = At._handle(validate, _stream_handle(stream))
        dev = At.rowptr.device
        self._y_idx = torch.empty(At.ncols, dtype=torch.int32, device=dev)
        self._y_vals = torch.empty(At.ncols, dtype=At.dtype, device=dev)

    def __call__(self, x_idx: torch.Tensor, x_vals: torch.Tensor, stream=None):
        if x_idx.dtype != torch.int32 or x_vals.dtype != self.At.dtype or not x_idx.is_cuda or not x_vals.is_cuda:
            raise TypeError("x_idx must be a CUDA int32 tensor and x_vals a CUDA tensor of A's dtype")
        if x_idx.numel() != x_vals.numel():
            raise ValueError("x_idx and x_vals differ in length")
        x_idx, x_vals = x_idx.contiguous(), x_vals.contiguous()
        nx = x_idx.numel()
        nnz = _abi.ws_spmspv(self._h, nx, x_idx.data_ptr() if nx else 0, x_vals.data_ptr() if nx else 0,
                             self._y_idx.data_ptr(), self._y_vals.data_ptr(), _stream_handle(stream))
        return self._y_idx[:nnz], self._y_vals[:nnz]

    def plan_info(self) -> dict:
        return _abi.ws_spgemm_plan_info(self._h)

    def close(self) -> None:
        if self._h:
            _abi.ws_csr_destroy(self._h)
            self._h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def spmspv(At: DeviceCSR, x_idx: torch.Tensor, x_vals: torch.Tensor, stream=None):
    """y = A x for a sparse x (A given by columns: At = A^T in CSR); returns (y_idx, y_vals)."""
    with SpMSpV(At, stream=stream) as op:
        yi, yv = op(x_idx, x_vals, stream)
        return yi.clone(), yv.clone()


def submatrix(A: DeviceCSR, r0: int, r1: int, c0: int, c1: int, stream=None, stats: dict | None = None) -> DeviceCSR:
    """S = A[r0:r1, c0:c1] as a DeviceCSR with columns shifted by -c0 (CUDA kernels).
    `stats["launches"]`, when given, is increased by the kernel launches queued."""
    s = _stream_handle(stream)
    hA = hS = None
    try:
        hA = A._handle(False, s)
        rowptr = torch.empty(max(r1 - r0, 0) + 1, dtype=torch.int64, device=A.rowptr.device)
        hS = _abi.ws_csr_create(r1 - r0, c1 - c0, 0, rowptr.data_ptr(), 0, 0, _DTYPES[A.dtype], False, s)
        nnz = _abi.ws_csr_submatrix_symbolic(hA, r0, r1, c0, c1, hS, s)
        colidx = torch.empty(nnz, dtype=torch.int32, device=A.rowptr.device)
        vals = torch.empty(nnz, dtype=A.dtype, device=A.rowptr.device)
        _abi.ws_csr_submatrix_numeric(hA, hS, colidx.data_ptr() if nnz else 0, vals.data_ptr() if nnz else 0, s)
        _abi.ws_spgemm_wait(hS, s)
        if stats is not None:
            info = _abi.ws_spgemm_plan_info(hS)
            stats["launches"] = stats.get("launches", 0) + info["symbolic_launches"] + info["numeric_launches"]
        return DeviceCSR(r1 - r0, c1 - c0, rowptr, colidx, vals)
    finally:
        for h in (hS, hA):
            if h:
                _abi.ws_csr_destroy(h)


class SpGEMMOuter(SpGEMM):
    """A reusable outer-product product C = A*B (ws_spgemm_outer_symbolic /
    ws_spgemm_outer_numeric): the k range is split into `parts` blocks, each
    block's partial product is a worker's own copy of C and the copies are
    coalesced by sparse additions, all inside the library.  Same interface as
    :class:`SpGEMM`."""

    def __init__(self, A: DeviceCSR, B: DeviceCSR, parts: int = 4, validate: bool = False, stream=None):
        super().__init__(A, B, validate=validate, stream=stream)
        self.parts = int(parts)

    def symbolic(self, stream=None) -> int:
        self.nnz = _abi.ws_spgemm_outer_symbolic(self._hA, self._hB, self._hC, self.parts, _stream_handle(stream))
        return self.nnz

    def numeric(self, out: DeviceCSR | None = None, stream=None) -> DeviceCSR:
        if self.nnz is None:
            raise RuntimeError("symbolic() must run before numeric()")
        if out is None or out.nnz != self.nnz:
            colidx = torch.empty(self.nnz, dtype=torch.int32, device=self.device)
            vals = torch.empty(self.nnz, dtype=self.A.dtype, device=self.device)
            out = DeviceCSR(self.A.nrows, self.B.ncols, self.c_rowptr, colidx, vals)
        _abi.ws_spgemm_outer_numeric(self._hA, self._hB, self._hC, out.colidx.data_ptr() if self.nnz else 0,
                                     out.vals.data_ptr() if self.nnz else 0, _stream_handle(stream))
        return out


def spgemm_outer(A: DeviceCSR, B: DeviceCSR, parts: int = 4, stream=None, stats: dict | None = None) -> DeviceCSR:
    """C = A*B as the outer-product SpGEMM of Sec. 5.1 (see :class:`SpGEMMOuter`).
    `stats["launches"]`, when given, is increased by the kernel launches queued."""
    if A.ncols != B.nrows:
        raise ValueError(f"shape mismatch: A is {A.nrows}x{A.ncols}, B is {B.nrows}x{B.ncols}")
    with SpGEMMOuter(A, B, parts, stream=stream) as op:
        op.symbolic(stream)
        C = op.numeric(stream=stream)
        op.wait(stream)
        if stats is not None:
            info = op.plan_info()
            stats["launches"] = stats.get("launches", 0) + info["symbolic_launches"] + info["numeric_launches"]
    return C


def spgemm(A: DeviceCSR, B: DeviceCSR, validate: bool = False, stream=None) -> DeviceCSR:
    """C = A*B for CSR matrices on the GPU (sorted columns, structural zeros kept)."""
    with SpGEMM(A, B, validate=validate, stream=stream) as op:
        op.symbolic(stream)
        C = op.numeric(stream=stream)
        op.wait(stream)
    return C
