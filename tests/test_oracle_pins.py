"""Pins for the CPU oracle, each against something other than the oracle itself.

* a hand-worked example (tests/golden), including a cancelled entry kept as 0.0;
* brute force: dense float64 matrix product (numpy) and boolean pattern
  product on tiny shapes, 0-sized and all-empty cases included;
* integer-valued inputs: the sums are exact, so values are bit-exact;
* identity and permutation products: bit-exact re-arrangements of the input;
* R-MAT with unit values: C = A*A counts length-2 paths (exact integers);
* the closed form of the squared 2D 5-point Laplacian (13-point stencil and
  its 3,397,636 nonzeros on the 512 x 512 grid);
* a library cross-check against scipy.sparse on positive values;
* CSR invariants and nnz(C) <= sum of products;
* sensitivity: planted mistakes (a dropped term, a flipped sign, a transposed
  operand, a shifted column) are rejected by these checks.
"""
from __future__ import annotations

import numpy as np
import pytest

from oracle import oracle_spgemm
from synth import HostCSR, laplacian_2d, random_csr, rmat_pattern, uniform_csr, workload
from tests._helpers import (check_csr_invariants, dense, golden_csr, pattern, products_per_row,
                            read_golden, value_error)


def _as_csr(C) -> HostCSR:
    return HostCSR(C.nrows, C.ncols, C.rowptr, C.colidx, C.vals)


def _dense_check(A, B, C, exact: bool) -> bool:
    """True iff C matches the dense product of A and B (structure from the pattern product)."""
    Pc = (pattern(A) @ pattern(B)) > 0
    D = dense(A) @ dense(B)
    Dabs = np.abs(dense(A)) @ np.abs(dense(B))
    Cs = _as_csr(C)
    if not np.array_equal(pattern(Cs) > 0, Pc):
        return False
    rows = np.repeat(np.arange(C.nrows), np.diff(C.rowptr))
    ref = D[rows, C.colidx]
    if exact:
        return bool(np.array_equal(C.vals, ref))
    kmax = max(A.ncols, 1)
    gamma = kmax * np.finfo(np.float64).eps
    err = np.abs(C.vals - ref)
    return bool(np.all(err <= 2 * gamma * Dabs[rows, C.colidx]))


def test_golden_hand_example():
    g = read_golden("hand_3x4_times_4x3.txt")
    A, B = golden_csr(g, "A"), golden_csr(g, "B")
    C = oracle_spgemm(A, B)
    assert C.rowptr.tolist() == [int(x) for x in g["C.rowptr"]]
    assert C.colidx.tolist() == [int(x) for x in g["C.colidx"]]
    assert C.vals.tolist() == [float(x) for x in g["C.vals"]]
    # absmass of the cancelled entry C[0,0] = |2*1| + |-1*2| = 4
    assert C.absmass[0] == 4.0


@pytest.mark.parametrize("seed", range(40))
def test_dense_bruteforce_tiny(seed):
    rng = np.random.default_rng(1000 + seed)
    m, k, n = (int(x) for x in rng.integers(0, 13, size=3))
    dens = float(rng.choice([0.0, 0.1, 0.3, 0.7, 1.0]))
    A = random_csr(m, k, dens, rng, np.float64, "sym", empty_rows=0.2)
    B = random_csr(k, n, float(rng.choice([0.1, 0.4, 1.0])), rng, np.float64, "sym", empty_rows=0.2)
    C = oracle_spgemm(A, B)
    check_csr_invariants(m, n, C.rowptr, C.colidx)
    assert _dense_check(A, B, C, exact=False)
    # absmass is the dense product of |A| and |B|
    rows = np.repeat(np.arange(m), np.diff(C.rowptr))
    Dabs = np.abs(dense(A)) @ np.abs(dense(B))
    assert np.allclose(C.absmass, Dabs[rows, C.colidx], rtol=1e-14, atol=0)


@pytest.mark.parametrize("seed", range(10))
def test_integer_values_bit_exact(seed):
    rng = np.random.default_rng(2000 + seed)
    m, k, n = 17, 23, 19
    A = random_csr(m, k, 0.3, rng, np.float64, "one", empty_rows=0.1)
    B = random_csr(k, n, 0.3, rng, np.float64, "one", empty_rows=0.1)
    A.vals = rng.integers(-5, 6, size=A.nnz).astype(np.float64)  # zeros stay structural
    B.vals = rng.integers(-5, 6, size=B.nnz).astype(np.float64)
    C = oracle_spgemm(A, B)
    assert _dense_check(A, B, C, exact=True)


def test_empty_and_degenerate_shapes():
    rng = np.random.default_rng(7)
    for m, k, n in [(0, 0, 0), (0, 5, 3), (4, 0, 3), (4, 5, 0), (3, 3, 3)]:
        A = random_csr(m, k, 0.0 if (m, k, n) == (3, 3, 3) else 0.5, rng)
        B = random_csr(k, n, 0.5, rng)
        C = oracle_spgemm(A, B)
        assert C.nnz == 0
        assert C.rowptr.tolist() == [0] * (m + 1)


def test_identity_products_bit_exact():
    rng = np.random.default_rng(11)
    A = uniform_csr(300, 200, 7, rng, np.float64, "sym")
    I_left = HostCSR(300, 300, np.arange(301, dtype=np.int64), np.arange(300, dtype=np.int32), np.ones(300))
    I_right = HostCSR(200, 200, np.arange(201, dtype=np.int64), np.arange(200, dtype=np.int32), np.ones(200))
    for C in (oracle_spgemm(I_left, A), oracle_spgemm(A, I_right)):
        assert np.array_equal(C.rowptr, A.rowptr)
        assert np.array_equal(C.colidx, A.colidx)
        assert np.array_equal(C.vals, A.vals)


def test_permutation_products_bit_exact():
    rng = np.random.default_rng(12)
    A = uniform_csr(250, 180, 9, rng, np.float64, "sym")
    perm = rng.permutation(250)
    # P has P[i, perm[i]] = 1, so (P*A)[i, :] = A[perm[i], :]
    P = HostCSR(250, 250, np.arange(251, dtype=np.int64), perm.astype(np.int32), np.ones(250))
    C = oracle_spgemm(P, A)
    lens = np.diff(A.rowptr)[perm]
    assert np.array_equal(np.diff(C.rowptr), lens)
    for i in range(250):
        s, e = A.rowptr[perm[i]], A.rowptr[perm[i] + 1]
        cs, ce = C.rowptr[i], C.rowptr[i + 1]
        assert np.array_equal(C.colidx[cs:ce], A.colidx[s:e])
        assert np.array_equal(C.vals[cs:ce], A.vals[s:e])
    # Q has Q[q, sig[q]] = 1, so (A*Q)[i, sig[q]] = A[i, q]
    sig = rng.permutation(180)
    Q = HostCSR(180, 180, np.arange(181, dtype=np.int64), sig.astype(np.int32), np.ones(180))
    C = oracle_spgemm(A, Q)
    assert np.array_equal(C.rowptr, A.rowptr)
    for i in range(250):
        s, e = A.rowptr[i], A.rowptr[i + 1]
        newc = sig[A.colidx[s:e]]
        order = np.argsort(newc)
        assert np.array_equal(C.colidx[s:e], newc[order])
        assert np.array_equal(C.vals[s:e], A.vals[s:e][order])


def test_rmat_unit_values_count_paths():
    rng = np.random.default_rng(5)
    rp, ci, _ = rmat_pattern(9, 8, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(512, 512, rp, ci, np.ones(ci.size))
    C = oracle_spgemm(A, A, threads=4)
    P = pattern(A)
    paths = P @ P  # exact integer path counts
    rows = np.repeat(np.arange(512), np.diff(C.rowptr))
    assert np.array_equal(pattern(_as_csr(C)) > 0, paths > 0)
    assert np.array_equal(C.vals, paths[rows, C.colidx].astype(np.float64))


def _laplacian_square_closed_form(g: int):
    """Expected (row, col, val) of L^2 for the Dirichlet 5-point Laplacian L on a g x g grid.

    L = 4I - N with N the grid adjacency.  Then L^2 = 16I - 8N + N^2 and
      diagonal            16 + deg(v)
      grid neighbour      -8   (adjacent grid vertices share no neighbour)
      straight distance 2 +1   (one middle vertex)
      diagonal (+-1,+-1)  +2   (two corner vertices, both inside the grid)
    """
    nv = g * g
    r, c = np.divmod(np.arange(nv, dtype=np.int64), g)
    deg = (r > 0).astype(np.int64) + (r < g - 1) + (c > 0) + (c < g - 1)
    rows, cols, vals = [], [], []
    for dr, dc, val in [(0, 0, None), (-1, 0, -8), (1, 0, -8), (0, -1, -8), (0, 1, -8),
                        (-2, 0, 1), (2, 0, 1), (0, -2, 1), (0, 2, 1),
                        (-1, -1, 2), (-1, 1, 2), (1, -1, 2), (1, 1, 2)]:
        rr, cc = r + dr, c + dc
        ok = (rr >= 0) & (rr < g) & (cc >= 0) & (cc < g)
        rows.append(np.flatnonzero(ok))
        cols.append((rr * g + cc)[ok])
        vals.append((16.0 + deg[ok]) if val is None else np.full(ok.sum(), float(val)))
    rows, cols, vals = np.concatenate(rows), np.concatenate(cols), np.concatenate(vals)
    order = np.lexsort((cols, rows))
    return rows[order], cols[order], vals[order]


def test_laplacian_square_closed_form_512():
    g = 512
    A = laplacian_2d(g)
    C = oracle_spgemm(A, A, threads=8)
    # nnz(C) = sum over stencil offsets of (g - |dr|)(g - |dc|)
    assert C.nnz == g * g + 4 * g * (g - 1) + 4 * g * (g - 2) + 4 * (g - 1) ** 2 == 3_397_636
    rows, cols, vals = _laplacian_square_closed_form(g)
    assert np.array_equal(np.repeat(np.arange(g * g), np.diff(C.rowptr)), rows)
    assert np.array_equal(C.colidx, cols.astype(np.int32))
    assert np.array_equal(C.vals, vals)


def test_scipy_crosscheck_positive_values():
    sp = pytest.importorskip("scipy.sparse")
    rng = np.random.default_rng(21)
    A = uniform_csr(3000, 2000, 11, rng, np.float64, "pos")
    B = uniform_csr(2000, 2500, 13, rng, np.float64, "pos")
    C = oracle_spgemm(A, B, threads=4)
    SA = sp.csr_matrix((A.vals, A.colidx, A.rowptr), shape=(3000, 2000))
    SB = sp.csr_matrix((B.vals, B.colidx, B.rowptr), shape=(2000, 2500))
    SC = (SA @ SB).tocsr()
    SC.sort_indices()
    assert np.array_equal(SC.indptr, C.rowptr)
    assert np.array_equal(SC.indices, C.colidx)
    assert value_error(SC.data, C.vals, C.absmass) < 1e-14


def test_invariants_and_product_bound_uniform_2k():
    A, B = workload("uniform_2k")
    C = oracle_spgemm(A, B, threads=4)
    check_csr_invariants(A.nrows, B.ncols, C.rowptr, C.colidx)
    ub = products_per_row(A, B)
    assert ub.sum() == 131_072
    assert np.all(np.diff(C.rowptr) <= ub)
    assert np.array_equal(np.diff(C.rowptr) > 0, ub > 0)


def test_row_subset_matches_full():
    rng = np.random.default_rng(3)
    A = uniform_csr(500, 400, 6, rng)
    B = uniform_csr(400, 300, 5, rng)
    full = oracle_spgemm(A, B, threads=3)
    sel = np.array([499, 0, 17, 17, 250], dtype=np.int64)
    part = oracle_spgemm(A, B, rows=sel, threads=2)
    for t, i in enumerate(sel):
        a, b = full.rowptr[i], full.rowptr[i + 1]
        c, d = part.rowptr[t], part.rowptr[t + 1]
        assert np.array_equal(full.colidx[a:b], part.colidx[c:d])
        assert np.array_equal(full.vals[a:b], part.vals[c:d])


def test_thread_count_does_not_change_result():
    A, B = workload("uniform_2k")
    c1 = oracle_spgemm(A, B, threads=1)
    c7 = oracle_spgemm(A, B, threads=7)
    assert np.array_equal(c1.rowptr, c7.rowptr)
    assert np.array_equal(c1.colidx, c7.colidx)
    assert np.array_equal(c1.vals, c7.vals)


class _Planted:
    """Planted mistakes applied to a correct oracle result on the CPU."""

    @staticmethod
    def drop_term(A, B, C):
        # remove one product's contribution from one entry (a dropped term)
        C.vals = C.vals.copy()
        i = int(np.flatnonzero(np.diff(A.rowptr))[0])
        p = A.rowptr[i]
        k = A.colidx[p]
        q = B.rowptr[k]
        j = B.colidx[q]
        e = C.rowptr[i] + int(np.searchsorted(C.colidx[C.rowptr[i]:C.rowptr[i + 1]], j))
        C.vals[e] -= A.vals[p] * B.vals[q]
        return C

    @staticmethod
    def flip_sign(A, B, C):
        C.vals = C.vals.copy()
        C.vals[len(C.vals) // 2] *= -1.0
        return C

    @staticmethod
    def shift_column(A, B, C):
        C.colidx = C.colidx.copy()
        r = int(np.flatnonzero(np.diff(C.rowptr))[0])
        e = C.rowptr[r + 1] - 1
        C.colidx[e] = min(C.colidx[e] + 1, C.ncols - 1) if C.colidx[e] + 1 < C.ncols else C.colidx[e] - 1
        return C


@pytest.mark.parametrize("mistake", ["drop_term", "flip_sign", "shift_column", "transposed"])
def test_pins_reject_planted_mistakes(mistake):
    rng = np.random.default_rng(99)
    A = random_csr(9, 11, 0.4, rng, np.float64, "sym")
    B = random_csr(11, 9, 0.4, rng, np.float64, "sym")
    if mistake == "transposed":
        # a transposed operand: computing (A*B)^T = B^T A^T in place of A*B
        D = dense(B).T @ dense(A).T
        rows, cols = np.nonzero((pattern(B).T @ pattern(A).T) > 0)
        rowptr = np.zeros(D.shape[0] + 1, dtype=np.int64)
        np.cumsum(np.bincount(rows, minlength=D.shape[0]), out=rowptr[1:])
        bad = type("R", (), {})()
        bad.nrows, bad.ncols = D.shape
        bad.rowptr, bad.colidx, bad.vals = rowptr, cols.astype(np.int32), D[rows, cols]
        assert not _dense_check(A, B, bad, exact=False)
        return
    C = oracle_spgemm(A, B)
    assert _dense_check(A, B, C, exact=False)
    bad = getattr(_Planted, mistake)(A, B, C)
    assert not _dense_check(A, B, bad, exact=False)
