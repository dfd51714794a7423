"""Shared test helpers: golden-file reading, CSR invariant checks and the value tolerance.

Value tolerance (the summation-order bound).  The oracle accumulates in
float64 in ascending (p, q) order; the CUDA path accumulates in the value
type in an unspecified order.  For an entry with terms x_1..x_t the rounding
error of any summation order is bounded by gamma_t * sum |x_i|, so the error
is measured against absmass = sum |A[i,k] B[k,j]| (which is >= |C[i,j]|, and
equals it when no cancellation occurs):
    err = max |c - c_ref| / absmass      (entries with absmass == 0 must be exactly 0)
Bars: 1e-12 for float64 and 1e-5 for float32.
"""
from __future__ import annotations

import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
TOL = {np.dtype(np.float64): 1e-12, np.dtype(np.float32): 1e-5}


def read_golden(name: str) -> dict:
    out = {}
    with open(os.path.join(GOLDEN, name)) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, *vals = line.split()
            out[key] = vals
    return out


def golden_csr(g: dict, prefix: str):
    from synth import HostCSR

    m, n = (int(x) for x in g[f"{prefix}.shape"])
    rowptr = np.array([int(x) for x in g[f"{prefix}.rowptr"]], dtype=np.int64)
    colidx = np.array([int(x) for x in g.get(f"{prefix}.colidx", [])], dtype=np.int32)
    vals = np.array([float(x) for x in g.get(f"{prefix}.vals", [])], dtype=np.float64)
    return HostCSR(m, n, rowptr, colidx, vals)


def value_error(c, c_ref, absmass) -> float:
    """max |c - c_ref| / absmass; inf if an entry with absmass 0 is not exactly c_ref."""
    c = np.asarray(c, dtype=np.float64)
    c_ref = np.asarray(c_ref, dtype=np.float64)
    absmass = np.asarray(absmass, dtype=np.float64)
    if c.size == 0:
        return 0.0
    diff = np.abs(c - c_ref)
    zero = absmass == 0
    if np.any(diff[zero] != 0):
        return float("inf")
    nz = ~zero
    return float(np.max(diff[nz] / absmass[nz])) if nz.any() else 0.0


def check_csr_invariants(nrows, ncols, rowptr, colidx) -> None:
    """CSR invariants: rowptr[0] = 0, non-decreasing, rowptr[m] = nnz;
    columns strictly increasing within each row and in [0, ncols)."""
    rowptr = np.asarray(rowptr)
    colidx = np.asarray(colidx)
    assert rowptr.shape == (nrows + 1,)
    assert rowptr[0] == 0
    assert np.all(np.diff(rowptr) >= 0)
    assert rowptr[-1] == colidx.size
    if colidx.size:
        assert colidx.min() >= 0 and colidx.max() < ncols
        d = np.diff(colidx.astype(np.int64))
        row_start = np.zeros(colidx.size, dtype=bool)
        starts = rowptr[:-1][np.diff(rowptr) > 0]
        row_start[starts] = True
        assert np.all(d[~row_start[1:]] > 0), "columns not strictly increasing within a row"


def products_per_row(A, B) -> np.ndarray:
    lenB = np.diff(B.rowptr)
    ub = np.zeros(A.nrows, dtype=np.int64)
    if A.nnz:
        np.add.at(ub, np.repeat(np.arange(A.nrows), np.diff(A.rowptr)), lenB[A.colidx])
    return ub


def dense(M) -> np.ndarray:
    D = np.zeros((M.nrows, M.ncols), dtype=np.float64)
    rows = np.repeat(np.arange(M.nrows), np.diff(M.rowptr))
    D[rows, M.colidx] = M.vals
    return D


def pattern(M) -> np.ndarray:
    P = np.zeros((M.nrows, M.ncols), dtype=np.int64)
    rows = np.repeat(np.arange(M.nrows), np.diff(M.rowptr))
    P[rows, M.colidx] = 1
    return P
