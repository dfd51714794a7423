"""GPU parity of the outer-product SpGEMM (k split into blocks, partial
products coalesced by sparse additions) and of the submatrix extraction it
uses, through the C ABI.

Submatrices must equal numpy's dense slices exactly.  The outer product must
match the CPU oracle of C = A*B: structure bit-exact, values within 1e-12
(float64) or 1e-5 (float32) of sum |a*b| (the summation order differs: sums
per k block, then block sums).
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2606_20855_gb300 import _abi
from paper_2606_20855_gb300.spgemm import DeviceCSR, spgemm_outer, submatrix
from synth import HostCSR, laplacian_2d, random_csr, rmat_pattern, uniform_csr
from tests._gpu import assert_matches_oracle
from tests._helpers import check_csr_invariants, dense

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.mark.parametrize("seed", range(12))
def test_submatrix_matches_dense_slice(seed):
    rng = np.random.default_rng(300 + seed)
    m, n = (int(v) for v in rng.integers(1, 300, size=2))
    A = random_csr(m, n, float(rng.choice([0.01, 0.1, 0.5])), rng, np.float64, "sym", empty_rows=0.1)
    dA = DeviceCSR.from_host(A, DEV)
    D = dense(A)
    for _ in range(6):
        r0, r1 = sorted(int(v) for v in rng.integers(0, m + 1, size=2))
        c0, c1 = sorted(int(v) for v in rng.integers(0, n + 1, size=2))
        S = submatrix(dA, r0, r1, c0, c1)
        rp, ci, vv = S.to_host()
        check_csr_invariants(r1 - r0, c1 - c0, rp, ci)
        Sd = np.zeros((r1 - r0, c1 - c0))
        rows = np.repeat(np.arange(r1 - r0), np.diff(rp))
        Sd[rows, ci] = vv
        assert np.array_equal(Sd, D[r0:r1, c0:c1])
        assert rp[-1] == np.count_nonzero(dense_pattern(A)[r0:r1, c0:c1])


def dense_pattern(A):
    P = np.zeros((A.nrows, A.ncols), dtype=bool)
    P[np.repeat(np.arange(A.nrows), np.diff(A.rowptr)), A.colidx] = True
    return P


def test_submatrix_errors():
    rng = np.random.default_rng(1)
    dA = DeviceCSR.from_host(random_csr(20, 30, 0.2, rng, np.float64, "sym"), DEV)
    with pytest.raises(_abi.WsError, match="WS_ERR_INVALID_ARG"):
        submatrix(dA, 5, 21, 0, 30)
    with pytest.raises(_abi.WsError, match="WS_ERR_INVALID_ARG"):
        submatrix(dA, 0, 20, 10, 5)


def _outer(A, B, parts):
    dA = DeviceCSR.from_host(A, DEV)
    dB = dA if B is A else DeviceCSR.from_host(B, DEV)
    C = spgemm_outer(dA, dB, parts)
    torch.cuda.synchronize()
    return C.to_host()


@pytest.mark.parametrize("parts", [1, 2, 3, 7])
@pytest.mark.parametrize("dtype", [np.float64, np.float32])
@pytest.mark.parametrize("seed", range(4))
def test_outer_random(seed, dtype, parts):
    rng = np.random.default_rng(400 + seed)
    m, k, n = (int(v) for v in rng.integers(1, 300, size=3))
    A = random_csr(m, k, float(rng.choice([0.01, 0.05, 0.2])), rng, dtype, "sym", empty_rows=0.1)
    B = random_csr(k, n, float(rng.choice([0.01, 0.05, 0.2])), rng, dtype, "sym", empty_rows=0.1)
    rowptr, colidx, vals = _outer(A, B, parts)
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("parts", [2, 8])
def test_outer_workload_shapes(parts):
    rng = np.random.default_rng(0)
    A = uniform_csr(2048, 2048, 8, rng, np.float64, "sym")
    assert_matches_oracle(A, A, *_outer(A, A, parts))
    L = laplacian_2d(64)
    assert_matches_oracle(L, L, *_outer(L, L, parts))
    rp, ci, _ = rmat_pattern(11, 8, (0.57, 0.19, 0.19, 0.05), rng)
    R = HostCSR(2048, 2048, rp, ci, np.ones(ci.size))
    assert_matches_oracle(R, R, *_outer(R, R, parts))


def test_outer_cancellation_and_empty():
    # partial sums of opposite sign in different k blocks: the entry is kept as 0.0
    A = HostCSR(1, 4, np.array([0, 2], np.int64), np.array([0, 3], np.int32), np.array([1.0, 1.0]))
    B = HostCSR(4, 2, np.array([0, 1, 1, 1, 2], np.int64), np.array([1, 1], np.int32), np.array([2.0, -2.0]))
    rowptr, colidx, vals = _outer(A, B, 2)
    assert rowptr.tolist() == [0, 1] and colidx.tolist() == [1] and vals.tolist() == [0.0]
    Z = HostCSR(3, 5, np.zeros(4, np.int64), np.zeros(0, np.int32), np.zeros(0))
    W = random_csr(5, 6, 0.5, np.random.default_rng(2), np.float64, "sym")
    rowptr, colidx, vals = _outer(Z, W, 3)
    assert rowptr.tolist() == [0, 0, 0, 0] and colidx.size == 0


def test_outer_repeated_on_one_handle_and_errors():
    """The same operator run twice gives the same product; the ABI refuses
    parts < 1 and a numeric pass before the symbolic pass."""
    from paper_2606_20855_gb300.spgemm import SpGEMMOuter
    rng = np.random.default_rng(9)
    A = random_csr(150, 90, 0.06, rng, np.float64, "sym")
    B = random_csr(90, 120, 0.08, rng, np.float64, "sym")
    dA, dB = DeviceCSR.from_host(A, DEV), DeviceCSR.from_host(B, DEV)
    with SpGEMMOuter(dA, dB, parts=3) as op:
        with pytest.raises(_abi.WsError, match="WS_ERR_STATE"):
            _abi.ws_spgemm_outer_numeric(op._hA, op._hB, op._hC, 0, 0, 0)
        results = []
        for _ in range(2):
            op.symbolic()
            C = op.numeric()
            op.wait()
            results.append(C.to_host())
        for rowptr, colidx, vals in results:
            assert_matches_oracle(A, B, rowptr, colidx, vals)
        assert np.array_equal(results[0][1], results[1][1])
        op.parts = 0
        with pytest.raises(_abi.WsError, match="WS_ERR_INVALID_ARG"):
            op.symbolic()
