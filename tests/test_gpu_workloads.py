"""Parity on the five named workloads at full size, through the same ABI calls the benchmark times.

Every workload is compared with the oracle on every row: the row pointer and
column indices bit-exact, the values within the dtype's tolerance.  The large
results (up to 4.3 GB) are streamed: the oracle computes a block of rows,
the matching segment of C is copied from the device, and the two are compared
before the next block, so host memory stays bounded.  CSR invariants of the
whole result are also checked on the device.
"""
from __future__ import annotations

import functools

import numpy as np
import pytest

from synth import workload
from tests._gpu import assert_matches_oracle, device_invariants
from tests._helpers import products_per_row

pytestmark = pytest.mark.gpu


@functools.lru_cache(maxsize=1)
def _workload(name):
    return workload(name)


def _run_full(name):
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    A, B = _workload(name)
    dA = DeviceCSR.from_host(A)
    dB = dA if B is A else DeviceCSR.from_host(B)
    op = SpGEMM(dA, dB)
    nnz = op.symbolic()
    C = op.numeric()
    op.wait()
    return A, B, op, C, nnz



@pytest.mark.parametrize("name", ["uniform_2k", "laplace2d_512"])
def test_small_workloads_every_row(name):
    A, B, op, C, nnz = _run_full(name)
    with op:
        rowptr, colidx, vals = C.to_host()
    err = assert_matches_oracle(A, B, rowptr, colidx, vals)
    if name == "laplace2d_512":
        assert nnz == 3_397_636
        assert err == 0.0  # small-integer sums are exact in any order
    else:
        assert nnz == 129_319


def _compare_blocks(A, B, C, block_rows):
    """Streams C = A*B against the oracle in blocks of `block_rows` rows; returns the largest value error."""
    import torch

    from oracle import oracle_spgemm
    from tests._gpu import ORACLE_THREADS
    from tests._helpers import TOL, value_error

    tol = TOL[np.dtype(A.vals.dtype)]
    rowptr = C.rowptr.cpu().numpy()
    worst = 0.0
    for r0 in range(0, A.nrows, block_rows):
        r1 = min(A.nrows, r0 + block_rows)
        rows = np.arange(r0, r1, dtype=np.int64)
        ref = oracle_spgemm(A, B, rows=rows, threads=ORACLE_THREADS)
        # row pointer of the block, relative to its first entry, bit-exact
        np.testing.assert_array_equal(rowptr[r0:r1 + 1] - rowptr[r0], ref.rowptr, err_msg=f"rows {r0}..{r1}")
        s0, s1 = int(rowptr[r0]), int(rowptr[r1])
        col = C.colidx[s0:s1].cpu().numpy()
        val = C.vals[s0:s1].cpu().numpy()
        np.testing.assert_array_equal(col, ref.colidx, err_msg=f"rows {r0}..{r1}")
        err = value_error(val, ref.vals, ref.absmass)
        assert err <= tol, f"rows {r0}..{r1}: value error {err:.3e} > {tol:.1e}"
        worst = max(worst, err)
        del ref, col, val
    torch.cuda.synchronize()
    return worst


@pytest.mark.slow
@pytest.mark.parametrize("name,block_rows", [("rmat16", 8192), ("uniform_rect_1m", 65536),
                                             ("rmat20_x_uniform", 131072)])
def test_large_workloads_every_row(name, block_rows):
    A, B, op, C, nnz = _run_full(name)
    with op:
        info = op.plan_info()
        device_invariants(C)
        ub = products_per_row(A, B)
        assert info["products"] == int(ub.sum())
        assert nnz <= int(ub.sum())
        err = _compare_blocks(A, B, C, block_rows)
        if name == "rmat16":
            assert err == 0.0  # path counts: exact integers in any order
