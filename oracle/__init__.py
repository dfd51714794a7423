"""CPU oracles for C = A*B and for C = A op B (elementwise) on CSR matrices -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline leg use this
package.  The CUDA library never imports or links it, and it imports nothing
from the CUDA library.

``oracle_spgemm(A, B, rows=None, threads=1)`` returns the rows ``rows`` of
C (all rows when ``rows`` is None) as numpy arrays computed by
``spgemm_oracle.cpp`` (Gustavson's row-wise algorithm with an ordered map per
row, Sec. 5.1), with values accumulated in float64, plus
absmass = sum |a*b| per output entry.  ``oracle_ewise(A, B, op)`` (ewise.py)
is the elementwise SpAdd / Hadamard oracle, ``oracle_spmspv(A, x_idx, x_vals)``
(spmspv.py) the sparse matrix - sparse vector product.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

from .build import LIB, build

_lib = None


def _load():
    global _lib
    if _lib is None:
        path = build()
        lib = ctypes.CDLL(path)
        i64, p = ctypes.c_int64, ctypes.c_void_p
        lib.oracle_spgemm.restype = p
        lib.oracle_spgemm.argtypes = [i64, i64, i64, p, p, p, p, p, p, p, i64, ctypes.c_int,
                                      ctypes.POINTER(i64)]
        lib.oracle_result_copy.restype = ctypes.c_int
        lib.oracle_result_copy.argtypes = [p, p, p, p, p]
        lib.oracle_result_free.restype = None
        lib.oracle_result_free.argtypes = [p]
        _lib = lib
    return _lib


@dataclass
class OracleCSR:
    """Rows of C as computed by the oracle (float64 values)."""

    nrows: int
    ncols: int
    rowptr: np.ndarray  # int64[nrows + 1]
    colidx: np.ndarray  # int32[nnz]
    vals: np.ndarray  # float64[nnz]
    absmass: np.ndarray  # float64[nnz]

    @property
    def nnz(self) -> int:
        return int(self.rowptr[-1])


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p) if a.size else None


def oracle_spgemm(A, B, rows=None, threads: int = 1) -> OracleCSR:
    """C[rows, :] = A[rows, :] * B.  A, B: objects with nrows, ncols, rowptr, colidx, vals."""
    if A.ncols != B.nrows:
        raise ValueError(f"shape mismatch: A is {A.nrows}x{A.ncols}, B is {B.nrows}x{B.ncols}")
    lib = _load()
    rpA = np.ascontiguousarray(A.rowptr, dtype=np.int64)
    ciA = np.ascontiguousarray(A.colidx, dtype=np.int32)
    vA = np.ascontiguousarray(A.vals, dtype=np.float64)
    rpB = np.ascontiguousarray(B.rowptr, dtype=np.int64)
    ciB = np.ascontiguousarray(B.colidx, dtype=np.int32)
    vB = np.ascontiguousarray(B.vals, dtype=np.float64)
    if rows is not None:
        sel = np.ascontiguousarray(rows, dtype=np.int64)
        if sel.size and (sel.min() < 0 or sel.max() >= A.nrows):
            raise IndexError("row selection out of range")
        nsel = sel.size
    else:
        sel = None
        nsel = A.nrows
    nnz = ctypes.c_int64(0)
    handle = lib.oracle_spgemm(A.nrows, A.ncols, B.ncols, rpA.ctypes.data_as(ctypes.c_void_p),
                               _ptr(ciA), _ptr(vA), rpB.ctypes.data_as(ctypes.c_void_p), _ptr(ciB),
                               _ptr(vB), None if sel is None else sel.ctypes.data_as(ctypes.c_void_p),
                               nsel, int(threads), ctypes.byref(nnz))
    if not handle:
        raise MemoryError("oracle_spgemm: allocation failed")
    try:
        n = nnz.value
        rowptr = np.empty(nsel + 1, dtype=np.int64)
        colidx = np.empty(n, dtype=np.int32)
        vals = np.empty(n, dtype=np.float64)
        absmass = np.empty(n, dtype=np.float64)
        lib.oracle_result_copy(handle, rowptr.ctypes.data_as(ctypes.c_void_p), _ptr(colidx), _ptr(vals),
                               _ptr(absmass))
    finally:
        lib.oracle_result_free(handle)
    return OracleCSR(nsel, B.ncols, rowptr, colidx, vals, absmass)


from .ewise import oracle_ewise  # noqa: E402  (needs OracleCSR above)
from .spmspv import OracleSparseVector, oracle_spmspv  # noqa: E402

__all__ = ["oracle_spgemm", "oracle_ewise", "oracle_spmspv", "OracleCSR", "OracleSparseVector", "build", "LIB"]
