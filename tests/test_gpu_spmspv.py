"""GPU parity of the sparse matrix - sparse vector product y = A x against the
CPU oracle, through the C ABI (A passed by columns, as the CSR of A^T).

y's indices must be bit-exact; values within 1e-12 (float64) or 1e-5
(float32) of sum |A[i,j] x[j]| (the summation-order bound; the GPU adds with
global atomics in no fixed order).  Cases: random shapes and densities of x,
a power-law matrix, a heavily shared output position, degenerate shapes and
vectors, repeated calls on one handle, the full-size input, and the errors.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import oracle_spmspv
from paper_2606_20855_gb300 import _abi
from paper_2606_20855_gb300.spgemm import DeviceCSR, SpMSpV
from synth import HostCSR, random_csr, rmat_pattern, sparse_vector, spmspv_workload, transpose_csr
from tests._helpers import TOL, value_error

pytestmark = pytest.mark.gpu

DTYPES = [np.float64, np.float32]


def run(A, xi, xv, op=None):
    At = transpose_csr(A)
    dev = torch.device("cuda:0")
    dxi = torch.from_numpy(np.ascontiguousarray(xi, dtype=np.int32)).to(dev)
    dxv = torch.from_numpy(np.ascontiguousarray(xv, dtype=A.vals.dtype)).to(dev)
    if op is not None:
        yi, yv = op(dxi, dxv)
    else:
        with SpMSpV(DeviceCSR.from_host(At, dev)) as o:
            yi, yv = o(dxi, dxv)
            yi, yv = yi.clone(), yv.clone()
    return yi.cpu().numpy(), yv.cpu().numpy()


def check(A, xi, xv, op=None):
    yi, yv = run(A, xi, xv, op)
    ref = oracle_spmspv(A, xi, xv)
    np.testing.assert_array_equal(yi, ref.idx)
    err = value_error(yv, ref.vals, ref.absmass)
    tol = TOL[np.dtype(A.vals.dtype)]
    assert err <= tol, f"value error {err:.3e} > {tol:.1e}"


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("seed", range(12))
def test_random_shapes(seed, dtype):
    rng = np.random.default_rng(700 + seed)
    m, n = (int(v) for v in rng.integers(1, 3000, size=2))
    A = random_csr(m, n, float(rng.choice([0.001, 0.01, 0.05])), rng, dtype, "sym", empty_rows=0.1)
    xi, xv = sparse_vector(n, float(rng.choice([0.0, 0.01, 0.1, 0.5, 1.0])), rng, dtype, "sym")
    check(A, xi, xv)


@pytest.mark.parametrize("dtype", DTYPES)
def test_power_law_several_tiles(dtype):
    # 2^15 rows: eight compaction tiles and hub rows hit by many columns
    rng = np.random.default_rng(4)
    rp, ci, _ = rmat_pattern(15, 16, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(1 << 15, 1 << 15, rp, ci, rng.uniform(0.0, 1.0, ci.size).astype(dtype))
    xi, xv = sparse_vector(1 << 15, 0.1, rng, dtype, "pos")
    check(A, xi, xv)


def test_shared_output_position():
    # row 0 holds every column: all products of x meet in y[0]
    n = 20_000
    rng = np.random.default_rng(6)
    B = random_csr(50, n, 0.001, rng, np.float64, "pos")
    rowptr = np.concatenate([[0], B.rowptr + n]).astype(np.int64)
    A = HostCSR(51, n, rowptr, np.concatenate([np.arange(n, dtype=np.int32), B.colidx]),
                np.concatenate([rng.uniform(0.5, 1.0, n), B.vals]))
    xi, xv = sparse_vector(n, 0.5, rng, np.float64, "pos")
    check(A, xi, xv)


def test_degenerate():
    for m, n in ((0, 5), (5, 0), (0, 0), (7, 9)):
        Z = HostCSR(m, n, np.zeros(m + 1, np.int64), np.zeros(0, np.int32), np.zeros(0))
        xi = np.arange(min(n, 3), dtype=np.int32)
        check(Z, xi, np.ones(xi.size))
    rng = np.random.default_rng(9)
    A = random_csr(100, 80, 0.05, rng, np.float64, "sym")
    check(A, np.zeros(0, np.int32), np.zeros(0))
    check(A, np.arange(80, dtype=np.int32), rng.uniform(-1, 1, 80))


def test_repeated_calls_on_one_handle():
    rng = np.random.default_rng(12)
    A = random_csr(5000, 4000, 0.002, rng, np.float64, "sym")
    dev = torch.device("cuda:0")
    with SpMSpV(DeviceCSR.from_host(transpose_csr(A), dev)) as op:
        for density in (0.1, 0.0, 0.7, 0.1):
            xi, xv = sparse_vector(4000, density, rng, np.float64, "sym")
            check(A, xi, xv, op)


def test_index_out_of_range_is_reported():
    rng = np.random.default_rng(1)
    A = random_csr(30, 20, 0.2, rng, np.float64, "sym")
    dev = torch.device("cuda:0")
    with SpMSpV(DeviceCSR.from_host(transpose_csr(A), dev)) as op:
        bad = torch.tensor([3, 25], dtype=torch.int32, device=dev)  # 25 >= n = 20
        with pytest.raises(_abi.WsError, match="WS_ERR_DEVICE"):
            op(bad, torch.ones(2, dtype=torch.float64, device=dev))
        with pytest.raises(_abi.WsError, match="WS_ERR_INVALID_ARG"):
            _abi.ws_spmspv(op._h, 21, 0, 0, 0, 0, 0)  # more x entries than columns
        # the handle stays usable
        xi, xv = sparse_vector(20, 0.5, rng, np.float64, "sym")
        check(A, xi, xv, op)


@pytest.mark.slow
def test_full_size_workload():
    A, xi, xv = spmspv_workload("spmspv_rmat20")
    check(A, xi, xv)
