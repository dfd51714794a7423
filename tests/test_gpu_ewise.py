"""GPU parity of the elementwise operations (SpAdd, Hadamard product) against
the CPU oracle, through the C ABI.

Structure (rowptr, colidx) must be bit-exact; values within 1e-12 (float64)
or 1e-5 (float32) of |A[i,j]| + |B[i,j]| (SpAdd) or |A[i,j] B[i,j]|
(Hadamard): one rounding in the value type against the float64 oracle.
Cases: random shapes, every lane-group size, rows cut into many chunks with
equal columns on both sides of the cuts, empty operands and shapes, cancelled
sums, the full-size R-MAT inputs (B a relabelled copy of A, and B = A), and
the error paths.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import oracle_ewise
from paper_2606_20855_gb300 import _abi
from paper_2606_20855_gb300.spgemm import DeviceCSR, Ewise, SpGEMM
from synth import EWISE_WORKLOADS, HostCSR, ewise_workload, random_csr, uniform_csr
from tests._gpu import device_invariants, tuning
from tests._helpers import TOL, check_csr_invariants, value_error

pytestmark = pytest.mark.gpu

OPS = ["add", "mul"]
DTYPES = [np.float64, np.float32]


def run_ewise(A, B, op, validate=False):
    dA = DeviceCSR.from_host(A, "cuda:0")
    dB = dA if B is A else DeviceCSR.from_host(B, "cuda:0")
    with Ewise(dA, dB, op, validate=validate) as e:
        nnz = e.symbolic()
        C = e.numeric()
        e.wait()
        info = e.plan_info()
        rowptr, colidx, vals = C.to_host()
    assert rowptr[-1] == nnz
    return rowptr, colidx, vals, info


def check(A, B, op, validate=False):
    rowptr, colidx, vals, info = run_ewise(A, B, op, validate)
    ref = oracle_ewise(A, B, op)
    check_csr_invariants(A.nrows, A.ncols, rowptr, colidx)
    np.testing.assert_array_equal(rowptr, ref.rowptr)
    np.testing.assert_array_equal(colidx, ref.colidx)
    err = value_error(vals, ref.vals, ref.absmass)
    tol = TOL[np.dtype(A.vals.dtype)]
    assert err <= tol, f"value error {err:.3e} > {tol:.1e}"
    return info


# lanes per chunk: 1 (one thread per chunk), 2 (one lane per chunk of a
# warp-staged tile of 32 chunks), 0 (lane groups of 4..32 sized from the mean
# row length) and 64 (a warp per 64-position chunk ranking every entry by
# binary search)
LANES = [1, 2, 0, 64]


@pytest.mark.parametrize("lanes", LANES)
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("seed", range(10))
def test_random_shapes(seed, dtype, op, lanes):
    rng = np.random.default_rng(900 + seed)
    m, n = (int(x) for x in rng.integers(1, 500, size=2))
    A = random_csr(m, n, float(rng.choice([0.005, 0.03, 0.2])), rng, dtype, "sym", empty_rows=0.1)
    B = random_csr(m, n, float(rng.choice([0.005, 0.03, 0.2])), rng, dtype, "sym", empty_rows=0.1)
    with tuning(ewise_lanes=lanes):
        check(A, B, op, validate=True)


@pytest.mark.parametrize("lanes", LANES)
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("per_row", [2, 6, 12, 40, 200])
def test_every_group_size(per_row, op, lanes):
    # mean merged row lengths 4 .. 400 select 4, 8, 16 and 32 lanes per chunk
    # (lanes 0), or cut rows into 1..7 chunks of 64 (lanes 1); 30,011 rows
    # give many CTAs and a ragged last one
    rng = np.random.default_rng(per_row)
    n = max(64, per_row * per_row // 2)  # rejection sampling of distinct columns needs n >> per_row^2 / 2
    A = uniform_csr(30_011, n, per_row, rng, np.float64, "sym")
    B = uniform_csr(30_011, n, per_row, rng, np.float64, "sym")
    with tuning(ewise_lanes=lanes):
        check(A, B, op)


def _long_rows(m, n, lens, rng, overlap):
    """Rows of the given lengths; B shares about `overlap` of A's columns per row."""
    ra, rb = [], []
    for ln in lens:
        a = np.sort(rng.choice(n, size=ln, replace=False))
        keep = a[rng.random(ln) < overlap]
        extra = np.setdiff1d(rng.choice(n, size=ln, replace=False), a)[: max(0, ln - keep.size)]
        ra.append(a)
        rb.append(np.sort(np.concatenate([keep, extra])))
    def build(rows):
        rp = np.zeros(m + 1, dtype=np.int64)
        np.cumsum([r.size for r in rows], out=rp[1:])
        ci = np.concatenate(rows).astype(np.int32) if rows else np.zeros(0, np.int32)
        return HostCSR(m, n, rp, ci, rng.uniform(-1.0, 1.0, ci.size))
    return build(ra), build(rb)


@pytest.mark.parametrize("lanes,chunk", [(1, 64), (1, 2), (1, 7), (2, 16), (2, 2), (2, 7), (0, 64), (32, 64),
                                         (64, 64), (-1, 64)])
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("overlap", [0.0, 0.5, 1.0])
def test_long_rows_many_chunks(overlap, op, lanes, chunk):
    # rows of up to 20,000 entries per operand are cut into hundreds of chunks
    # (tens of thousands with chunks of 2); with overlap 1.0 every column is an
    # equal pair, so pairs meet every cut
    rng = np.random.default_rng(31)
    lens = [20_000, 1, 0, 5_000, 777, 3, 12_345, 64, 65, 0]
    A, B = _long_rows(len(lens), 40_000, lens, rng, overlap)
    with tuning(ewise_lanes=lanes, ewise_chunk=chunk):
        check(A, B, op)


@pytest.mark.parametrize("op", OPS)
def test_same_operand_long_rows(op):
    rng = np.random.default_rng(5)
    A, _ = _long_rows(6, 50_000, [30_000, 2, 9_999, 0, 1, 17_000], rng, 0.0)
    rowptr, colidx, vals, _ = run_ewise(A, A, op)
    np.testing.assert_array_equal(rowptr, A.rowptr)
    np.testing.assert_array_equal(colidx, A.colidx)
    ref = 2.0 * A.vals if op == "add" else A.vals * A.vals
    np.testing.assert_array_equal(vals, ref)  # one exact doubling / one rounded square


@pytest.mark.parametrize("op", OPS)
def test_degenerate(op):
    for m, n in ((0, 0), (0, 7), (5, 0), (4, 9)):
        Z = HostCSR(m, n, np.zeros(m + 1, np.int64), np.zeros(0, np.int32), np.zeros(0))
        check(Z, Z, op)
    rng = np.random.default_rng(2)
    A = random_csr(50, 60, 0.1, rng, np.float64, "sym")
    Z = HostCSR(50, 60, np.zeros(51, np.int64), np.zeros(0, np.int32), np.zeros(0))
    check(A, Z, op)
    check(Z, A, op)


def test_cancelled_sums_are_kept():
    rng = np.random.default_rng(8)
    A = random_csr(200, 300, 0.05, rng, np.float64, "sym")
    neg = HostCSR(A.nrows, A.ncols, A.rowptr, A.colidx, -A.vals)
    rowptr, colidx, vals, _ = run_ewise(A, neg, "add")
    np.testing.assert_array_equal(rowptr, A.rowptr)
    np.testing.assert_array_equal(colidx, A.colidx)
    assert not np.any(vals)


@pytest.mark.slow
@pytest.mark.parametrize("lanes", [None, 1, 64])
@pytest.mark.parametrize("op", OPS)
@pytest.mark.parametrize("name", list(EWISE_WORKLOADS))
def test_full_size_workloads(name, op, lanes):
    A, B = ewise_workload(name)
    dA = DeviceCSR.from_host(A, "cuda:0")
    dB = dA if B is A else DeviceCSR.from_host(B, "cuda:0")
    with tuning(**({} if lanes is None else {"ewise_lanes": lanes})):
        with Ewise(dA, dB, op) as e:
            e.symbolic()
            C = e.numeric()
            e.wait()
            device_invariants(C)
            rowptr, colidx, vals = C.to_host()
    ref = oracle_ewise(A, B, op)
    np.testing.assert_array_equal(rowptr, ref.rowptr)
    np.testing.assert_array_equal(colidx, ref.colidx)
    assert value_error(vals, ref.vals, ref.absmass) <= TOL[np.dtype(np.float64)]


def test_errors():
    rng = np.random.default_rng(1)
    A = DeviceCSR.from_host(random_csr(10, 12, 0.3, rng, np.float64, "sym"), "cuda:0")
    B = DeviceCSR.from_host(random_csr(10, 13, 0.3, rng, np.float64, "sym"), "cuda:0")
    with pytest.raises(_abi.WsError, match="WS_ERR_SHAPE"):
        with Ewise(A, B, "add") as e:
            e.symbolic()
    B32 = DeviceCSR.from_host(random_csr(10, 12, 0.3, rng, np.float32, "sym"), "cuda:0")
    with pytest.raises(TypeError):
        Ewise(A, B32, "add")
    with pytest.raises(ValueError):
        Ewise(A, A, "sub")
    # passes of one kind cannot be finished by the other kind's numeric call
    with Ewise(A, A, "mul") as e:
        e.symbolic()
        with pytest.raises(_abi.WsError, match="WS_ERR_STATE"):
            _abi.ws_spgemm_numeric(e._hA, e._hB, e._hC, 1, 1, 0)
    Bsq = DeviceCSR.from_host(random_csr(12, 12, 0.3, rng, np.float64, "sym"), "cuda:0")
    with SpGEMM(A, Bsq) as op:
        op.symbolic()
        with pytest.raises(_abi.WsError, match="WS_ERR_STATE"):
            _abi.ws_ewise_numeric(op._hA, op._hB, op._hC, 1, 1, 0)
    torch.cuda.synchronize()
