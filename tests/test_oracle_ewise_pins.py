"""Pins for the elementwise oracle (SpAdd and the Hadamard product), each
against something other than the oracle itself.

* a hand-worked example (tests/golden), including cancelled sums kept as 0.0;
* brute force: dense float64 matrices and boolean patterns on tiny shapes,
  0-sized and all-empty cases included;
* integer-valued inputs: sums and products are exact, so values are bit-exact;
* closed forms: A + A = 2A and A .* A = A^2 entrywise on A's pattern,
  A + (-A) keeps A's pattern with zeros, patterns with no common position
  give nnz(A) + nnz(B) entries under + and none under .*, a diagonal
  pattern picks out the diagonal under .*;
* a library cross-check against scipy.sparse on positive values (no
  cancellation, so scipy's dropping of zero sums does not apply);
* CSR invariants on the benchmark-sized inputs;
* sensitivity: planted mistakes (a dropped entry of one operand, the union
  used for the Hadamard product, a flipped sign, subtraction for addition)
  are rejected by these checks.
"""
from __future__ import annotations

import numpy as np
import pytest

from oracle import oracle_ewise
from synth import HostCSR, permute_symmetric, random_csr, rmat_pattern, uniform_csr
from tests._helpers import check_csr_invariants, dense, golden_csr, pattern, read_golden


def _dense_check(A, B, C, op: str) -> bool:
    """True iff C equals the dense elementwise result (structure from the boolean patterns)."""
    PA, PB = pattern(A) > 0, pattern(B) > 0
    P = (PA | PB) if op == "add" else (PA & PB)
    D = dense(A) + dense(B) if op == "add" else dense(A) * dense(B)
    m = C.nrows
    Cs = HostCSR(m, C.ncols, C.rowptr, C.colidx, C.vals)
    if not np.array_equal(pattern(Cs) > 0, P):
        return False
    rows = np.repeat(np.arange(m), np.diff(C.rowptr))
    # one rounding of a float64 sum or product: exact in these small cases
    return bool(np.array_equal(C.vals, D[rows, C.colidx]))


def test_golden_hand_example():
    g = read_golden("hand_ewise_3x5.txt")
    A, B = golden_csr(g, "A"), golden_csr(g, "B")
    for op, key in (("add", "ADD"), ("mul", "MUL")):
        C = oracle_ewise(A, B, op)
        assert C.rowptr.tolist() == [int(x) for x in g[f"{key}.rowptr"]]
        assert C.colidx.tolist() == [int(x) for x in g[f"{key}.colidx"]]
        assert C.vals.tolist() == [float(x) for x in g[f"{key}.vals"]]
    C = oracle_ewise(A, B, "add")
    # absmass of the cancelled entry C[0,2] = |-2| + |2|
    assert C.absmass[1] == 4.0


@pytest.mark.parametrize("seed", range(40))
@pytest.mark.parametrize("op", ["add", "mul"])
def test_dense_bruteforce_tiny(seed, op):
    rng = np.random.default_rng(seed)
    m, n = int(rng.integers(0, 9)), int(rng.integers(0, 9))
    A = random_csr(m, n, float(rng.uniform(0.0, 0.8)), rng, np.float64, "sym")
    B = random_csr(m, n, float(rng.uniform(0.0, 0.8)), rng, np.float64, "sym")
    C = oracle_ewise(A, B, op)
    check_csr_invariants(C.nrows, C.ncols, C.rowptr, C.colidx)
    assert _dense_check(A, B, C, op)


@pytest.mark.parametrize("op", ["add", "mul"])
def test_integer_values_bit_exact(op):
    rng = np.random.default_rng(7)
    A = random_csr(40, 50, 0.3, rng, np.float64, "sym")
    B = random_csr(40, 50, 0.3, rng, np.float64, "sym")
    A.vals = rng.integers(-9, 10, A.vals.size).astype(np.float64)
    B.vals = rng.integers(-9, 10, B.vals.size).astype(np.float64)
    assert _dense_check(A, B, oracle_ewise(A, B, op), op)


def test_closed_forms_same_operand():
    rng = np.random.default_rng(3)
    A = uniform_csr(300, 200, 9, rng, np.float64, "sym")
    C = oracle_ewise(A, A, "add")
    assert np.array_equal(C.rowptr, A.rowptr) and np.array_equal(C.colidx, A.colidx)
    assert np.array_equal(C.vals, 2.0 * A.vals)
    H = oracle_ewise(A, A, "mul")
    assert np.array_equal(H.rowptr, A.rowptr) and np.array_equal(H.colidx, A.colidx)
    assert np.array_equal(H.vals, A.vals * A.vals)
    neg = HostCSR(A.nrows, A.ncols, A.rowptr, A.colidx, -A.vals)
    Z = oracle_ewise(A, neg, "add")
    assert np.array_equal(Z.colidx, A.colidx) and not np.any(Z.vals)
    assert np.array_equal(Z.absmass, 2.0 * np.abs(A.vals))


def test_disjoint_patterns_and_diagonal():
    n = 64
    rows = np.arange(n)
    even = HostCSR(n, n, np.arange(n + 1, dtype=np.int64), ((rows // 2) * 2).astype(np.int32),
                   np.arange(1, n + 1, dtype=np.float64))
    odd = HostCSR(n, n, np.arange(n + 1, dtype=np.int64), ((rows // 2) * 2 + 1).astype(np.int32),
                  np.arange(1, n + 1, dtype=np.float64))
    C = oracle_ewise(even, odd, "add")
    assert C.nnz == 2 * n and np.all(np.diff(C.rowptr) == 2)
    assert oracle_ewise(even, odd, "mul").nnz == 0
    rng = np.random.default_rng(5)
    M = random_csr(n, n, 0.3, rng, np.float64, "sym")
    eye = HostCSR(n, n, np.arange(n + 1, dtype=np.int64), rows.astype(np.int32), np.ones(n))
    D = oracle_ewise(eye, M, "mul")
    dm = dense(M)
    diag_rows = np.flatnonzero(np.diag(pattern(M)))
    assert np.array_equal(np.repeat(np.arange(n), np.diff(D.rowptr)), diag_rows)
    assert np.array_equal(D.colidx, diag_rows) and np.array_equal(D.vals, dm[diag_rows, diag_rows])


@pytest.mark.parametrize("op", ["add", "mul"])
def test_scipy_crosscheck_positive_values(op):
    sp = pytest.importorskip("scipy.sparse")
    rng = np.random.default_rng(11)
    rp, ci, _ = rmat_pattern(12, 8, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(4096, 4096, rp, ci, rng.uniform(0.5, 1.0, ci.size))
    B = permute_symmetric(A, rng.permutation(4096))
    B = HostCSR(B.nrows, B.ncols, B.rowptr, B.colidx, rng.uniform(0.5, 1.0, B.colidx.size))
    for X, Y in ((A, B), (A, A)):
        sx = sp.csr_matrix((X.vals, X.colidx, X.rowptr), shape=(4096, 4096))
        sy = sp.csr_matrix((Y.vals, Y.colidx, Y.rowptr), shape=(4096, 4096))
        ref = (sx + sy if op == "add" else sx.multiply(sy)).tocsr()
        ref.sort_indices()
        C = oracle_ewise(X, Y, op)
        assert np.array_equal(C.rowptr, ref.indptr) and np.array_equal(C.colidx, ref.indices)
        assert np.allclose(C.vals, ref.data, rtol=1e-15, atol=0)


def test_permuted_copy_is_a_relabelling():
    rng = np.random.default_rng(2)
    A = random_csr(30, 30, 0.2, rng, np.float64, "sym")
    perm = rng.permutation(30)
    B = permute_symmetric(A, perm)
    check_csr_invariants(B.nrows, B.ncols, B.rowptr, B.colidx)
    P = np.zeros((30, 30))
    P[perm, np.arange(30)] = 1.0  # P e_i = e_perm[i]
    assert np.array_equal(dense(B), P @ dense(A) @ P.T)


class _Planted:
    """Planted mistakes applied to a correct oracle result on the CPU."""

    @staticmethod
    def drop_one_operand_entry(A, B, C, op):
        # drop the first entry of C that is stored in exactly one operand
        only = np.flatnonzero((pattern(A) > 0) ^ (pattern(B) > 0))
        rows = np.repeat(np.arange(C.nrows), np.diff(C.rowptr))
        keys = rows * C.ncols + C.colidx
        e = int(np.flatnonzero(np.isin(keys, only))[0])
        keep = np.ones(C.nnz, dtype=bool)
        keep[e] = False
        rowptr = C.rowptr.copy()
        rowptr[rows[e] + 1:] -= 1
        C.rowptr, C.colidx, C.vals = rowptr, C.colidx[keep], C.vals[keep]
        return C

    @staticmethod
    def flip_sign(A, B, C, op):
        C.vals = C.vals.copy()
        C.vals[C.nnz // 2] = -C.vals[C.nnz // 2] if C.vals[C.nnz // 2] != 0 else 1.0
        return C

    @staticmethod
    def subtract(A, B, C, op):
        return oracle_ewise(A, HostCSR(B.nrows, B.ncols, B.rowptr, B.colidx, -B.vals), op)

    @staticmethod
    def union_for_product(A, B, C, op):
        # the SpAdd pattern (union) where the product keeps only the intersection
        return oracle_ewise(A, B, "add")


@pytest.mark.parametrize("mistake,op", [("drop_one_operand_entry", "add"), ("flip_sign", "add"),
                                        ("flip_sign", "mul"), ("subtract", "add"),
                                        ("union_for_product", "mul")])
def test_pins_reject_planted_mistakes(mistake, op):
    rng = np.random.default_rng(21)
    A = random_csr(12, 13, 0.4, rng, np.float64, "sym")
    B = random_csr(12, 13, 0.4, rng, np.float64, "sym")
    C = oracle_ewise(A, B, op)
    assert _dense_check(A, B, C, op)
    bad = getattr(_Planted, mistake)(A, B, C, op)
    assert not _dense_check(A, B, bad, op)
