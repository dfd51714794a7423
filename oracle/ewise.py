"""CPU oracle for elementwise sparse operations on CSR matrices -- TEST INFRASTRUCTURE.

Only the tests, the smoke check and the benchmark's CPU-baseline leg use this
module.  The CUDA library never imports it, and it imports nothing from the
CUDA library.

What it computes (Sec. 5.2, "Sparse Linear Algebra": C = A op B with
op in {+, elementwise product}, A and B of the same shape):

  SpAdd     (op "add"): pattern(C) = pattern(A) union pattern(B);
                        C[i,j] = A[i,j] + B[i,j], a missing operand entry
                        contributing nothing.  A sum that is exactly 0.0 is
                        kept (structural result, as for the product).
  Hadamard  (op "mul"): pattern(C) = pattern(A) intersect pattern(B);
                        C[i,j] = A[i,j] * B[i,j].

Stored zeros in A or B are entries.  Values are widened to float64 and
combined in float64; for an entry in both operands of SpAdd the sum is
A[i,j] + B[i,j] in that order.  Besides C the oracle returns, per entry,
absmass = |A[i,j]| + |B[i,j]| (SpAdd) or |A[i,j] * B[i,j]| (Hadamard), the
magnitude against which rounding differences are judged.

How: every stored entry gets the key i * ncols + j (int64), which orders
entries exactly as CSR does (row-major, columns ascending).  SpAdd takes the
sorted set of keys of both operands (numpy.unique) and adds each operand's
values at its keys; the Hadamard product takes the keys common to both
(numpy.intersect1d) and multiplies the two values at each.  Row pointers are
the prefix sums of the entry counts per row.
"""
from __future__ import annotations

import numpy as np

from . import OracleCSR

OPS = ("add", "mul")


def _keys(M) -> tuple[np.ndarray, np.ndarray]:
    rp = np.asarray(M.rowptr, dtype=np.int64)
    rows = np.repeat(np.arange(M.nrows, dtype=np.int64), np.diff(rp))
    keys = rows * max(int(M.ncols), 1) + np.asarray(M.colidx, dtype=np.int64)
    return keys, np.asarray(M.vals, dtype=np.float64)


def oracle_ewise(A, B, op: str) -> OracleCSR:
    """C = A op B with op "add" (SpAdd) or "mul" (Hadamard).

    A, B: objects with nrows, ncols, rowptr, colidx, vals (valid CSR with
    strictly increasing columns per row).
    """
    if op not in OPS:
        raise ValueError(f"op must be one of {OPS}, got {op!r}")
    if (A.nrows, A.ncols) != (B.nrows, B.ncols):
        raise ValueError(f"shape mismatch: A is {A.nrows}x{A.ncols}, B is {B.nrows}x{B.ncols}")
    m, n = int(A.nrows), int(A.ncols)
    kA, vA = _keys(A)
    kB, vB = _keys(B)
    if op == "add":
        keys, inv = np.unique(np.concatenate([kA, kB]), return_inverse=True)
        both = np.concatenate([vA, vB])
        vals = np.zeros(keys.size, dtype=np.float64)
        np.add.at(vals, inv, both)  # unbuffered, in index order: 0 + A[i,j] (exact), then + B[i,j]
        absmass = np.zeros(keys.size, dtype=np.float64)
        np.add.at(absmass, inv, np.abs(both))
    else:
        keys, ia, ib = np.intersect1d(kA, kB, assume_unique=True, return_indices=True)
        vals = vA[ia] * vB[ib]
        absmass = np.abs(vals)
    width = max(n, 1)
    rows = keys // width
    rowptr = np.zeros(m + 1, dtype=np.int64)
    if m:
        np.cumsum(np.bincount(rows, minlength=m), out=rowptr[1:])
    return OracleCSR(m, n, rowptr, (keys % width).astype(np.int32), vals, absmass)
