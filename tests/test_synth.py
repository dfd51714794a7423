"""The seeded generators produce the stated shapes, counts and CSR structure."""
from __future__ import annotations

import numpy as np
import pytest

from synth import HostCSR, laplacian_2d, rmat_pattern, row_subset, uniform_csr, workload
from tests._helpers import check_csr_invariants, products_per_row


def test_uniform_rows_exact_and_distinct():
    rng = np.random.default_rng(0)
    A = uniform_csr(5000, 40, 8, rng, np.float32, "sym")  # about half the rows are redrawn
    check_csr_invariants(A.nrows, A.ncols, A.rowptr, A.colidx)
    assert np.all(np.diff(A.rowptr) == 8)
    assert A.vals.dtype == np.float32 and A.vals.min() >= -1 and A.vals.max() <= 1


def test_uniform_subsets_are_uniform():
    # every column is equally likely: 3 of 6 columns, 60k rows -> each column ~ 30k times
    rng = np.random.default_rng(1)
    A = uniform_csr(60000, 6, 3, rng)
    counts = np.bincount(A.colidx, minlength=6)
    assert np.all(np.abs(counts - 30000) < 600)


def test_laplacian_structure():
    A = laplacian_2d(4)
    check_csr_invariants(16, 16, A.rowptr, A.colidx)
    assert A.nnz == 5 * 16 - 4 * 4
    D = np.zeros((16, 16))
    D[np.repeat(np.arange(16), np.diff(A.rowptr)), A.colidx] = A.vals
    assert np.array_equal(D, D.T)
    assert np.all(np.diag(D) == 4.0)
    assert np.all(D.sum(axis=1)[[5, 6, 9, 10]] == 0.0)  # interior rows sum to zero


def test_rmat_dedup_and_skew():
    rng = np.random.default_rng(2)
    rp, ci, ne = rmat_pattern(10, 8, (0.57, 0.19, 0.19, 0.05), rng)
    assert ne == 8 * 1024 and rp[-1] <= ne
    check_csr_invariants(1024, 1024, rp, ci)
    lens = np.diff(rp)
    assert lens[:32].sum() > 20 * lens[-32:].sum()  # hubs at low ids


@pytest.mark.slow
def test_named_workload_sizes():
    A, B = workload("uniform_2k")
    assert (A.nrows, A.ncols, A.nnz) == (2048, 2048, 16384)
    assert products_per_row(A, B).sum() == 131_072
    A, B = workload("laplace2d_512")
    assert A.nnz == 1_308_672 and products_per_row(A, B).sum() == 6_535_176
    A, B = workload("rmat16")
    check_csr_invariants(A.nrows, A.ncols, A.rowptr, A.colidx)
    assert np.all(A.vals == 1.0)


def test_row_subset():
    rng = np.random.default_rng(3)
    A = uniform_csr(50, 30, 4, rng)
    S = row_subset(A, np.array([3, 3, 49, 0]))
    assert S.nrows == 4 and S.nnz == 16
    assert np.array_equal(S.colidx[:4], A.colidx[12:16])
    assert np.array_equal(S.vals[8:12], A.vals[196:200])
