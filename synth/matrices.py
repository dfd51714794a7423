"""Seeded synthetic CSR matrices for the SpGEMM workloads.

This module only *draws inputs*.  It contains no part of the product
C = A*B: both the CPU oracle and the CUDA path receive the arrays built here
and nothing else.  Every matrix is returned as a :class:`HostCSR` with
``rowptr`` int64[m+1], ``colidx`` int32[nnz] (0-based, strictly increasing
within a row) and ``vals`` float32 or float64.

Generators
----------
* :func:`uniform_csr` -- exactly ``r`` nonzeros per row, columns drawn
  uniformly *without replacement* per row (rejection of rows that drew a
  repeated column, which leaves every r-subset equally likely).
* :func:`laplacian_2d` -- the 5-point Laplacian of a g x g grid with
  Dirichlet boundaries, lexicographic numbering ``r*g + c``:
  kron(I, T) + kron(T, I) with T = tridiag(-1, 2, -1), so 4.0 on the
  diagonal and -1.0 for each grid neighbour.
* :func:`rmat_pattern` -- recursive-matrix (R-MAT) edge sampling: each edge
  picks one of four quadrants per bit level, most significant bit first,
  with probabilities (a, b, c, d) for (row 0, col 0), (row 0, col 1),
  (row 1, col 0), (row 1, col 1).  No noise, no vertex relabelling,
  duplicate edges merged, self-loops kept.
* :func:`workload` -- the five named workloads (uniform 2048^2 8/row;
  Laplacian 512^2 grid; R-MAT 2^16 edge factor 16; uniform 2^20 x 2^16
  16/row times 2^16 x 2^16 32/row in fp32; R-MAT 2^20 edge factor 8 times
  uniform 4/row).

Randomness: ``numpy.random.default_rng(seed)`` (PCG64), one generator per
workload, drawn in a fixed order (A's columns, A's values, then B's columns,
B's values).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

__all__ = [
    "HostCSR",
    "uniform_csr",
    "laplacian_2d",
    "rmat_pattern",
    "csr_from_coo_unique",
    "random_csr",
    "workload",
    "WORKLOADS",
    "permute_symmetric",
    "ewise_workload",
    "EWISE_WORKLOADS",
    "transpose_csr",
    "sparse_vector",
    "spmspv_workload",
    "SPMSPV_WORKLOADS",
]


@dataclass
class HostCSR:
    """A CSR matrix in host memory (numpy arrays)."""

    nrows: int
    ncols: int
    rowptr: np.ndarray  # int64[nrows + 1]
    colidx: np.ndarray  # int32[nnz]
    vals: np.ndarray  # float32 / float64 [nnz]

    @property
    def nnz(self) -> int:
        return int(self.rowptr[-1]) if self.rowptr.size else 0

    @property
    def dtype(self):
        return self.vals.dtype

    def row_lengths(self) -> np.ndarray:
        return np.diff(self.rowptr)


def _check_dtype(dtype) -> np.dtype:
    dt = np.dtype(dtype)
    if dt not in (np.dtype(np.float32), np.dtype(np.float64)):
        raise ValueError(f"value dtype must be float32 or float64, got {dt}")
    return dt


def _sorted_distinct_rows(rng: np.random.Generator, m: int, n: int, r: int) -> np.ndarray:
    """m rows of r distinct sorted integers in [0, n), each r-subset equally likely."""
    if r > n:
        raise ValueError(f"cannot draw {r} distinct columns from {n}")
    if m == 0 or r == 0:
        return np.zeros((m, r), dtype=np.int64)
    cols = rng.integers(0, n, size=(m, r), dtype=np.int64)
    cols.sort(axis=1)
    bad = np.flatnonzero((np.diff(cols, axis=1) == 0).any(axis=1)) if r > 1 else np.empty(0, np.int64)
    while bad.size:
        redraw = rng.integers(0, n, size=(bad.size, r), dtype=np.int64)
        redraw.sort(axis=1)
        cols[bad] = redraw
        still = (np.diff(redraw, axis=1) == 0).any(axis=1)
        bad = bad[still]
    return cols


def uniform_csr(m: int, n: int, r: int, rng: np.random.Generator, dtype=np.float64,
                values: str = "sym") -> HostCSR:
    """Uniform random CSR with exactly ``r`` nonzeros in every row.

    values: ``"sym"`` draws 2U-1 in [-1, 1); ``"pos"`` draws 1-U in (0, 1];
    ``"one"`` stores 1.0.
    """
    dt = _check_dtype(dtype)
    cols = _sorted_distinct_rows(rng, m, n, r)
    nnz = m * r
    rowptr = np.arange(0, nnz + 1, r, dtype=np.int64) if r > 0 else np.zeros(m + 1, np.int64)
    vals = _draw_values(rng, nnz, values).astype(dt)
    return HostCSR(m, n, rowptr, cols.reshape(-1).astype(np.int32), vals)


def _draw_values(rng: np.random.Generator, count: int, kind: str) -> np.ndarray:
    if kind == "sym":
        return 2.0 * rng.random(count) - 1.0
    if kind == "pos":
        return 1.0 - rng.random(count)
    if kind == "one":
        return np.ones(count)
    raise ValueError(f"unknown value kind {kind!r}")


def csr_from_coo_unique(m: int, n: int, rows: np.ndarray, cols: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Merge duplicate (row, col) pairs and return (rowptr int64, colidx int32) sorted by (row, col)."""
    key = rows.astype(np.int64) * np.int64(n) + cols.astype(np.int64)
    key = np.unique(key)
    r = key // n
    c = key - r * n
    rowptr = np.zeros(m + 1, dtype=np.int64)
    np.cumsum(np.bincount(r, minlength=m), out=rowptr[1:])
    return rowptr, c.astype(np.int32)


def rmat_pattern(scale: int, edge_factor: int, probs, rng: np.random.Generator) -> tuple[np.ndarray, np.ndarray, int]:
    """R-MAT sparsity pattern of a 2^scale square matrix.

    Samples exactly ``edge_factor * 2^scale`` edges, then merges duplicates.
    Returns (rowptr, colidx, edges_sampled).
    """
    a, b, c, d = probs
    if abs(a + b + c + d - 1.0) > 1e-12:
        raise ValueError("R-MAT quadrant probabilities must sum to 1")
    nv = 1 << scale
    ne = edge_factor * nv
    rows = np.zeros(ne, dtype=np.int64)
    cols = np.zeros(ne, dtype=np.int64)
    t_ab, t_abc = a + b, a + b + c
    for level in range(scale):
        u = rng.random(ne)
        bit = np.int64(1) << np.int64(scale - 1 - level)
        row_one = u >= t_ab  # quadrants c, d
        col_one = ((u >= a) & (u < t_ab)) | (u >= t_abc)  # quadrants b, d
        rows += row_one * bit
        cols += col_one * bit
    rowptr, colidx = csr_from_coo_unique(nv, nv, rows, cols)
    return rowptr, colidx, ne


def random_csr(m: int, n: int, density: float, rng: np.random.Generator, dtype=np.float64,
               values: str = "sym", empty_rows: float = 0.0) -> HostCSR:
    """Bernoulli(density) pattern, optionally with a fraction of rows forced empty.

    Meant for small test shapes; it builds a dense m x n mask.
    """
    dt = _check_dtype(dtype)
    mask = rng.random((m, n)) < density
    if empty_rows > 0 and m > 0:
        mask[rng.random(m) < empty_rows, :] = False
    rr, cc = np.nonzero(mask)
    rowptr = np.zeros(m + 1, dtype=np.int64)
    np.cumsum(np.bincount(rr, minlength=m), out=rowptr[1:])
    vals = _draw_values(rng, rr.size, values).astype(dt)
    return HostCSR(m, n, rowptr, cc.astype(np.int32), vals)


def laplacian_2d(g: int, dtype=np.float64) -> HostCSR:
    """5-point Laplacian on a g x g grid, Dirichlet boundary, row-major numbering."""
    dt = _check_dtype(dtype)
    nv = g * g
    idx = np.arange(nv, dtype=np.int64)
    r, c = idx // g, idx % g
    # Per vertex, candidate neighbours in increasing column order.
    offs = [(-g, r > 0), (-1, c > 0), (0, np.ones(nv, bool)), (1, c < g - 1), (g, r < g - 1)]
    counts = sum(ok.astype(np.int64) for _, ok in offs)
    rowptr = np.zeros(nv + 1, dtype=np.int64)
    np.cumsum(counts, out=rowptr[1:])
    colidx = np.empty(int(rowptr[-1]), dtype=np.int32)
    vals = np.empty(int(rowptr[-1]), dtype=dt)
    pos = rowptr[:-1].copy()
    for off, ok in offs:
        sel = np.flatnonzero(ok)
        colidx[pos[sel]] = (sel + off).astype(np.int32)
        vals[pos[sel]] = 4.0 if off == 0 else -1.0
        pos[sel] += 1
    return HostCSR(nv, nv, rowptr, colidx, vals)


RMAT_PROBS = (0.57, 0.19, 0.19, 0.05)

# name -> short description (sizes as stated in the workload list)
WORKLOADS = {
    "uniform_2k": "uniform random 2048x2048, 8 nnz/row, fp64 in [-1,1], seed 0; C = A*A",
    "laplace2d_512": "2D 5-point Laplacian on a 512x512 grid (262144^2), fp64; C = A*A",
    "rmat16": "R-MAT 2^16, edge factor 16, (a,b,c,d)=(.57,.19,.19,.05), fp64 1.0, seed 1; C = A*A",
    "uniform_rect_1m": "uniform 2^20x2^16 16/row times 2^16x2^16 32/row, fp32 in [-1,1], seed 2; C = A*B",
    "rmat20_x_uniform": "R-MAT 2^20 ef 8 (values in (0,1]) times uniform 2^20^2 4/row (values in (0,1]), fp64, seed 3; C = A*B",
}
WORKLOAD_ORDER = list(WORKLOADS)


def workload(name: str):
    """Return (A, B) for a named workload.  For C = A*A workloads B is A."""
    if isinstance(name, int):
        name = WORKLOAD_ORDER[name]
    if name == "uniform_2k":
        rng = np.random.default_rng(0)
        A = uniform_csr(2048, 2048, 8, rng, np.float64, "sym")
        return A, A
    if name == "laplace2d_512":
        A = laplacian_2d(512, np.float64)
        return A, A
    if name == "rmat16":
        rng = np.random.default_rng(1)
        rp, ci, _ = rmat_pattern(16, 16, RMAT_PROBS, rng)
        A = HostCSR(1 << 16, 1 << 16, rp, ci, np.ones(ci.size, dtype=np.float64))
        return A, A
    if name == "uniform_rect_1m":
        rng = np.random.default_rng(2)
        A = uniform_csr(1 << 20, 1 << 16, 16, rng, np.float32, "sym")
        B = uniform_csr(1 << 16, 1 << 16, 32, rng, np.float32, "sym")
        return A, B
    if name == "rmat20_x_uniform":
        rng = np.random.default_rng(3)
        rp, ci, _ = rmat_pattern(20, 8, RMAT_PROBS, rng)
        va = _draw_values(rng, ci.size, "pos")
        A = HostCSR(1 << 20, 1 << 20, rp, ci, va.astype(np.float64))
        B = uniform_csr(1 << 20, 1 << 20, 4, rng, np.float64, "pos")
        return A, B
    raise KeyError(f"unknown workload {name!r}; known: {WORKLOAD_ORDER}")


def permute_symmetric(A: HostCSR, perm: np.ndarray) -> HostCSR:
    """P A P^T for a square A: entry (i, j) moves to (perm[i], perm[j]) with its value."""
    if A.nrows != A.ncols:
        raise ValueError("symmetric permutation needs a square matrix")
    perm = np.asarray(perm, dtype=np.int64)
    rows = perm[np.repeat(np.arange(A.nrows, dtype=np.int64), np.diff(A.rowptr))]
    cols = perm[A.colidx.astype(np.int64)]
    order = np.argsort(rows * A.ncols + cols, kind="stable")
    rowptr = np.zeros(A.nrows + 1, dtype=np.int64)
    np.cumsum(np.bincount(rows, minlength=A.nrows), out=rowptr[1:])
    return HostCSR(A.nrows, A.ncols, rowptr, cols[order].astype(np.int32), A.vals[order])


# Inputs of the elementwise operations C = A + B and C = A .* B: a power-law
# graph standing in for the SNAP matrices, in the two cases the elementwise
# benchmarks use -- B a randomly relabelled copy of A, and B = A.
EWISE_WORKLOADS = {
    "ewise_rmat20_perm": "R-MAT 2^20, edge factor 8, (a,b,c,d)=(.57,.19,.19,.05), fp64 values in (0,1], "
                         "seed 4; B = P A P^T for a seeded random permutation P",
    "ewise_rmat20_same": "the same R-MAT A (seed 4) with B = A",
}


def ewise_workload(name: str):
    """Return (A, B) for a named elementwise workload."""
    if name not in EWISE_WORKLOADS:
        raise KeyError(f"unknown elementwise workload {name!r}; known: {list(EWISE_WORKLOADS)}")
    rng = np.random.default_rng(4)
    rp, ci, _ = rmat_pattern(20, 8, RMAT_PROBS, rng)
    A = HostCSR(1 << 20, 1 << 20, rp, ci, _draw_values(rng, ci.size, "pos").astype(np.float64))
    if name == "ewise_rmat20_same":
        return A, A
    return A, permute_symmetric(A, rng.permutation(A.nrows))


def transpose_csr(A: HostCSR) -> HostCSR:
    """A^T in CSR (= A in CSC): row j lists the rows i of A's entries in column j, ascending."""
    rows = np.repeat(np.arange(A.nrows, dtype=np.int64), np.diff(A.rowptr))
    cols = A.colidx.astype(np.int64)
    order = np.argsort(cols * max(A.nrows, 1) + rows, kind="stable")
    rowptr = np.zeros(A.ncols + 1, dtype=np.int64)
    np.cumsum(np.bincount(cols, minlength=A.ncols), out=rowptr[1:])
    return HostCSR(A.ncols, A.nrows, rowptr, rows[order].astype(np.int32), A.vals[order])


def sparse_vector(n: int, density: float, rng: np.random.Generator, dtype=np.float64,
                  kind: str = "pos") -> tuple[np.ndarray, np.ndarray]:
    """A sparse vector of length n: round(density * n) distinct indices drawn
    uniformly without replacement (sorted, int32) and values (see _draw_values)."""
    k = int(round(density * n))
    idx = np.sort(rng.choice(n, size=k, replace=False)).astype(np.int32) if k else np.zeros(0, np.int32)
    return idx, _draw_values(rng, k, kind).astype(dtype)


# Inputs of the sparse matrix - sparse vector product y = A x: a power-law
# graph standing in for the SNAP matrices of the paper's SpMSpV benchmark,
# and a vector with 90% of its entries zero.
SPMSPV_WORKLOADS = {
    "spmspv_rmat20": "R-MAT 2^20, edge factor 16, (a,b,c,d)=(.57,.19,.19,.05), fp64 values in (0,1], seed 5; "
                     "x: 10% of the 2^20 indices drawn uniformly without replacement, values in (0,1]",
}


def spmspv_workload(name: str):
    """Return (A, x_idx, x_vals) for a named SpMSpV workload."""
    if name not in SPMSPV_WORKLOADS:
        raise KeyError(f"unknown SpMSpV workload {name!r}; known: {list(SPMSPV_WORKLOADS)}")
    rng = np.random.default_rng(5)
    rp, ci, _ = rmat_pattern(20, 16, RMAT_PROBS, rng)
    A = HostCSR(1 << 20, 1 << 20, rp, ci, _draw_values(rng, ci.size, "pos").astype(np.float64))
    x_idx, x_vals = sparse_vector(A.ncols, 0.1, rng, np.float64, "pos")
    return A, x_idx, x_vals


def row_subset(A: HostCSR, rows: np.ndarray) -> HostCSR:
    """The rows ``rows`` of A (in the given order) as a new CSR with A's column count."""
    rows = np.asarray(rows, dtype=np.int64)
    lens = A.rowptr[rows + 1] - A.rowptr[rows]
    rowptr = np.zeros(rows.size + 1, dtype=np.int64)
    np.cumsum(lens, out=rowptr[1:])
    starts = np.repeat(A.rowptr[rows] - rowptr[:-1], lens)
    src = starts + np.arange(int(rowptr[-1]), dtype=np.int64)
    return HostCSR(rows.size, A.ncols, rowptr, A.colidx[src], A.vals[src])
