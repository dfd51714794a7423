"""GPU-side test helpers: run C = A*B through the C ABI and compare with the oracle."""
from __future__ import annotations

import contextlib
import os

import numpy as np
import torch

from oracle import oracle_spgemm
from paper_2606_20855_gb300 import _abi
from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
from tests._helpers import TOL, check_csr_invariants, value_error

ORACLE_THREADS = max(1, min(16, os.cpu_count() or 1))


def run_gpu(A, B, validate: bool = False, device: str = "cuda:0"):
    """Returns (rowptr, colidx, vals, plan_info) of C = A*B computed on the GPU."""
    dA = DeviceCSR.from_host(A, device)
    dB = dA if B is A else DeviceCSR.from_host(B, device)
    with SpGEMM(dA, dB, validate=validate) as op:
        nnz = op.symbolic()
        C = op.numeric()
        op.wait()
        info = op.plan_info()
        rowptr, colidx, vals = C.to_host()
    assert rowptr[-1] == nnz
    return rowptr, colidx, vals, info


def assert_matches_oracle(A, B, rowptr, colidx, vals, rows=None):
    """Structure bit-exact, values within the dtype's tolerance, for all rows or a row sample."""
    tol = TOL[np.dtype(A.vals.dtype)]
    if rows is None:
        ref = oracle_spgemm(A, B, threads=ORACLE_THREADS)
        check_csr_invariants(A.nrows, B.ncols, rowptr, colidx)
        np.testing.assert_array_equal(rowptr, ref.rowptr)
        np.testing.assert_array_equal(colidx, ref.colidx)
        err = value_error(vals, ref.vals, ref.absmass)
        assert err <= tol, f"value error {err:.3e} > {tol:.1e}"
        return err
    rows = np.asarray(rows, dtype=np.int64)
    ref = oracle_spgemm(A, B, rows=rows, threads=ORACLE_THREADS)
    lens = rowptr[rows + 1] - rowptr[rows]
    np.testing.assert_array_equal(lens, np.diff(ref.rowptr))
    starts = np.repeat(rowptr[rows] - ref.rowptr[:-1], lens)
    src = starts + np.arange(ref.nnz)
    np.testing.assert_array_equal(colidx[src], ref.colidx)
    err = value_error(vals[src], ref.vals, ref.absmass)
    assert err <= tol, f"value error {err:.3e} > {tol:.1e}"
    return err


@contextlib.contextmanager
def tuning(**kv):
    try:
        for k, v in kv.items():
            _abi.ws_set_tuning(k, v)
        yield
    finally:
        for k, v in _abi.TUNING_DEFAULTS.items():
            _abi.ws_set_tuning(k, v)


def device_invariants(C: DeviceCSR) -> None:
    """CSR invariants of a (possibly huge) device result, checked with torch on the GPU."""
    rp, ci = C.rowptr, C.colidx
    assert int(rp[0]) == 0 and int(rp[-1]) == ci.numel()
    assert bool((rp[1:] >= rp[:-1]).all())
    if ci.numel() == 0:
        return
    assert int(ci.min()) >= 0 and int(ci.max()) < C.ncols
    d = ci[1:].to(torch.int64) - ci[:-1].to(torch.int64)
    start = torch.zeros(ci.numel(), dtype=torch.bool, device=ci.device)
    nonempty = rp[:-1][rp[1:] > rp[:-1]]
    start[nonempty] = True
    ok = (d > 0) | start[1:]
    assert bool(ok.all()), "columns not strictly increasing within a row"
