"""Parity on the five named workloads at full size, through the same ABI calls the benchmark times.

Small workloads are compared with the oracle row for row; the large ones on
a row sample the oracle computes one row at a time (the heaviest rows, the
first and last rows and a seeded random sample), plus CSR invariants of the
whole result checked on the device.
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


def _sample_rows(A, B, n_random, seed):
    ub = products_per_row(A, B)
    rng = np.random.default_rng(seed)
    heavy = np.argsort(ub)[-8:]
    rand = rng.choice(A.nrows, size=min(n_random, A.nrows), replace=False)
    return np.unique(np.concatenate([heavy, rand, [0, A.nrows - 1]])), ub


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


@pytest.mark.slow
@pytest.mark.parametrize("name,n_random", [("rmat16", 600), ("uniform_rect_1m", 3000), ("rmat20_x_uniform", 3000)])
def test_large_workloads_sampled_rows(name, n_random):
    A, B, op, C, nnz = _run_full(name)
    with op:
        info = op.plan_info()
        device_invariants(C)
        rowptr = C.rowptr.cpu().numpy()
        rows, ub = _sample_rows(A, B, n_random, seed=sum(map(ord, name)))
        assert info["products"] == int(ub.sum())
        assert nnz <= int(ub.sum())
        # gather just the sampled rows' entries from the device
        import torch
        lens = rowptr[rows + 1] - rowptr[rows]
        idx = np.concatenate([np.arange(rowptr[r], rowptr[r + 1]) for r in rows]) if lens.sum() else np.zeros(0, np.int64)
        ti = torch.from_numpy(idx).to(C.colidx.device)
        col_s = C.colidx[ti].cpu().numpy()
        val_s = C.vals[ti].cpu().numpy()
    # rebuild a compact CSR of the sampled rows and compare row by row
    sub_rowptr = np.zeros(A.nrows + 1, dtype=np.int64)
    full_lens = np.zeros(A.nrows, dtype=np.int64)
    full_lens[rows] = lens
    np.cumsum(full_lens, out=sub_rowptr[1:])
    colidx = np.zeros(sub_rowptr[-1], dtype=np.int32)
    vals = np.zeros(sub_rowptr[-1], dtype=val_s.dtype)
    colidx[:] = col_s
    vals[:] = val_s
    assert_matches_oracle(A, B, sub_rowptr, colidx, vals, rows=rows)
    if name == "rmat16":
        assert np.all(val_s == np.round(val_s))  # path counts
    if name == "uniform_rect_1m":
        assert nnz > 534_000_000
