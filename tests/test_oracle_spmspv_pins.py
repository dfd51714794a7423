"""Pins for the SpMSpV oracle (y = A x with a sparse x), each against
something other than the oracle itself.

* a hand-worked example (tests/golden), including a cancelled sum kept as 0.0
  and a non-empty row that x does not reach;
* brute force: the dense float64 matrix-vector product and the boolean
  pattern product on tiny shapes, 0-sized and all-empty cases included;
* integer-valued inputs: sums are exact, so values are bit-exact;
* special cases: x a unit vector gives column j of A, x all ones gives the
  row sums, an identity A gives x back, an empty x gives an empty y;
* a library cross-check against scipy.sparse on positive values;
* the CSC view used by the GPU path (the transpose of A) checked against the
  dense transpose;
* sensitivity: planted mistakes (a dropped term, a row missing from the
  pattern, a flipped sign, x read at shifted indices) are rejected.
"""
from __future__ import annotations

import numpy as np
import pytest

from oracle import oracle_spmspv
from synth import HostCSR, random_csr, rmat_pattern, sparse_vector, transpose_csr
from tests._helpers import dense, golden_csr, pattern, read_golden


def _dense_check(A, x_idx, x_vals, y) -> bool:
    xd = np.zeros(A.ncols)
    xd[np.asarray(x_idx, dtype=np.int64)] = x_vals
    mask = np.zeros(A.ncols)
    mask[np.asarray(x_idx, dtype=np.int64)] = 1.0
    P = (pattern(A) @ mask) > 0
    if not np.array_equal(np.flatnonzero(P), np.asarray(y.idx, dtype=np.int64)):
        return False
    D = dense(A) @ xd
    Dabs = np.abs(dense(A)) @ np.abs(xd)
    gamma = max(A.ncols, 1) * np.finfo(np.float64).eps
    return bool(np.all(np.abs(y.vals - D[y.idx]) <= 2 * gamma * Dabs[y.idx]))


def test_golden_hand_example():
    g = read_golden("hand_spmspv_4x5.txt")
    A = golden_csr(g, "A")
    xi = np.array([int(v) for v in g["x.idx"]], dtype=np.int32)
    xv = np.array([float(v) for v in g["x.vals"]])
    y = oracle_spmspv(A, xi, xv)
    assert y.idx.tolist() == [int(v) for v in g["y.idx"]]
    assert y.vals.tolist() == [float(v) for v in g["y.vals"]]
    assert y.absmass.tolist() == [6.0, 2.0]


@pytest.mark.parametrize("seed", range(40))
def test_dense_bruteforce_tiny(seed):
    rng = np.random.default_rng(seed)
    m, n = int(rng.integers(0, 9)), int(rng.integers(0, 9))
    A = random_csr(m, n, float(rng.uniform(0.0, 0.8)), rng, np.float64, "sym")
    xi, xv = sparse_vector(n, float(rng.uniform(0.0, 1.0)), rng, np.float64, "sym")
    assert _dense_check(A, xi, xv, oracle_spmspv(A, xi, xv))


def test_integer_values_bit_exact():
    rng = np.random.default_rng(7)
    A = random_csr(60, 50, 0.3, rng, np.float64, "sym")
    A.vals = rng.integers(-9, 10, A.vals.size).astype(np.float64)
    xi, _ = sparse_vector(50, 0.3, rng)
    xv = rng.integers(-9, 10, xi.size).astype(np.float64)
    y = oracle_spmspv(A, xi, xv)
    xd = np.zeros(50)
    xd[xi] = xv
    assert np.array_equal(y.vals, (dense(A) @ xd)[y.idx])


def test_special_cases():
    rng = np.random.default_rng(3)
    A = random_csr(40, 30, 0.2, rng, np.float64, "sym")
    D = dense(A)
    for j in (0, 7, 29):
        y = oracle_spmspv(A, np.array([j], np.int32), np.array([1.0]))
        assert np.array_equal(y.idx, np.flatnonzero(pattern(A)[:, j]))
        assert np.array_equal(y.vals, D[y.idx, j])
    y = oracle_spmspv(A, np.arange(30, dtype=np.int32), np.ones(30))
    nonempty = np.flatnonzero(np.diff(A.rowptr))
    assert np.array_equal(y.idx, nonempty)
    assert np.allclose(y.vals, D.sum(axis=1)[nonempty], rtol=1e-15, atol=0)
    eye = HostCSR(30, 30, np.arange(31, dtype=np.int64), np.arange(30, dtype=np.int32), np.ones(30))
    xi, xv = sparse_vector(30, 0.4, rng, np.float64, "sym")
    y = oracle_spmspv(eye, xi, xv)
    assert np.array_equal(y.idx, xi) and np.array_equal(y.vals, xv)
    assert oracle_spmspv(A, np.zeros(0, np.int32), np.zeros(0)).nnz == 0


def test_scipy_crosscheck_positive_values():
    sp = pytest.importorskip("scipy.sparse")
    rng = np.random.default_rng(11)
    rp, ci, _ = rmat_pattern(12, 8, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(4096, 4096, rp, ci, rng.uniform(0.5, 1.0, ci.size))
    xi, xv = sparse_vector(4096, 0.1, rng)
    sa = sp.csr_matrix((A.vals, A.colidx, A.rowptr), shape=(4096, 4096))
    sx = sp.csc_matrix((xv, xi, np.array([0, xi.size])), shape=(4096, 1))
    ref = (sa @ sx).tocsc()
    ref.sort_indices()
    y = oracle_spmspv(A, xi, xv)
    assert np.array_equal(y.idx, ref.indices)
    assert np.allclose(y.vals, ref.data, rtol=1e-14, atol=0)


def test_transpose_is_the_column_view():
    rng = np.random.default_rng(2)
    A = random_csr(23, 31, 0.2, rng, np.float64, "sym")
    At = transpose_csr(A)
    assert (At.nrows, At.ncols) == (31, 23)
    assert np.array_equal(dense(At), dense(A).T)
    for j in range(At.nrows):  # columns of each row strictly increasing
        assert np.all(np.diff(At.colidx[At.rowptr[j]:At.rowptr[j + 1]]) > 0)


class _Planted:
    @staticmethod
    def drop_term(A, xi, xv, y):
        y.vals = y.vals.copy()
        j = int(xi[0])
        i = int(np.flatnonzero(pattern(A)[:, j])[0])
        e = int(np.searchsorted(y.idx, i))
        y.vals[e] -= dense(A)[i, j] * xv[0]
        return y

    @staticmethod
    def drop_row(A, xi, xv, y):
        y.idx, y.vals = y.idx[1:], y.vals[1:]
        return y

    @staticmethod
    def flip_sign(A, xi, xv, y):
        y.vals = y.vals.copy()
        y.vals[y.nnz // 2] *= -1.0
        return y

    @staticmethod
    def shifted_x(A, xi, xv, y):
        # x read one index too far (x[j] taken for column j + 1)
        keep = xi.astype(np.int64) + 1 < A.ncols
        return oracle_spmspv(A, (xi[keep] + 1).astype(np.int32), xv[keep])


@pytest.mark.parametrize("mistake", ["drop_term", "drop_row", "flip_sign", "shifted_x"])
def test_pins_reject_planted_mistakes(mistake):
    rng = np.random.default_rng(21)
    A = random_csr(15, 17, 0.35, rng, np.float64, "sym")
    xi, xv = sparse_vector(17, 0.4, rng, np.float64, "sym")
    y = oracle_spmspv(A, xi, xv)
    assert _dense_check(A, xi, xv, y)
    bad = getattr(_Planted, mistake)(A, xi, xv, y)
    assert not _dense_check(A, xi, xv, bad)
