"""CPU oracle for the sparse matrix - sparse vector product y = A x -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline leg use this
module.  The CUDA library never imports it, and it imports nothing from the
CUDA library.

What it computes (Sec. 5.2, "Sparse Linear Algebra": SpMSpV, y = A x with a
sparse x):

  y[i] = sum over stored A[i,j] with j stored in x of A[i,j] * x[j]

with the structural pattern {i : some stored A[i,j] meets a stored x[j]}; a
sum that is exactly 0.0 is kept and stored zeros count, as for the matrix
product.  A is m x n in CSR, x is given by strictly increasing indices in
[0, n) and their values; y is returned as strictly increasing indices and
values (float64).  Besides y the oracle returns absmass[i] = sum |A[i,j] x[j]|,
the magnitude against which summation-order differences are judged.

How: x is spread into a dense value array and a dense membership mask of
length n; every stored entry (i, j) of A, in CSR order (row by row, columns
ascending), with mask[j] set adds A[i,j] * x[j] to y[i] (numpy.add.at, which
applies the additions in that order).  Rows hit at least once form the
pattern.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass
class OracleSparseVector:
    """A sparse vector as computed by the oracle (float64 values)."""

    n: int
    idx: np.ndarray  # int32, strictly increasing
    vals: np.ndarray  # float64
    absmass: np.ndarray  # float64

    @property
    def nnz(self) -> int:
        return int(self.idx.size)


def oracle_spmspv(A, x_idx, x_vals) -> OracleSparseVector:
    """y = A x.  A: object with nrows, ncols, rowptr, colidx, vals (valid CSR);
    x_idx: strictly increasing indices in [0, A.ncols); x_vals: their values."""
    m, n = int(A.nrows), int(A.ncols)
    x_idx = np.asarray(x_idx, dtype=np.int64)
    x_vals = np.asarray(x_vals, dtype=np.float64)
    if x_idx.shape != x_vals.shape:
        raise ValueError("x indices and values differ in length")
    if x_idx.size and (x_idx.min() < 0 or x_idx.max() >= n or np.any(np.diff(x_idx) <= 0)):
        raise ValueError("x indices must be strictly increasing in [0, ncols)")
    mask = np.zeros(n, dtype=bool)
    xd = np.zeros(n, dtype=np.float64)
    mask[x_idx] = True
    xd[x_idx] = x_vals
    rows = np.repeat(np.arange(m, dtype=np.int64), np.diff(np.asarray(A.rowptr, dtype=np.int64)))
    cols = np.asarray(A.colidx, dtype=np.int64)
    hit = mask[cols]
    terms = np.asarray(A.vals, dtype=np.float64)[hit] * xd[cols[hit]]
    y = np.zeros(m, dtype=np.float64)
    np.add.at(y, rows[hit], terms)
    absmass = np.zeros(m, dtype=np.float64)
    np.add.at(absmass, rows[hit], np.abs(terms))
    touched = np.zeros(m, dtype=bool)
    touched[rows[hit]] = True
    idx = np.flatnonzero(touched)
    return OracleSparseVector(m, idx.astype(np.int32), y[idx], absmass[idx])
