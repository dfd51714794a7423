"""GPU parity against the CPU oracle on small and adversarial inputs (through the C ABI).

Structure (rowptr, colidx) must be bit-exact; values within max relative
error 1e-12 (float64) or 1e-5 (float32) of the summation-order bound.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import HostCSR, random_csr, rmat_pattern, uniform_csr
from tests._gpu import assert_matches_oracle, run_gpu, tuning
from tests._helpers import TOL

pytestmark = pytest.mark.gpu

DTYPES = [np.float64, np.float32]


def _csr(m, n, rows_cols, vals=None, dtype=np.float64):
    rowptr = np.zeros(m + 1, dtype=np.int64)
    cols = []
    for i in range(m):
        c = sorted(set(rows_cols.get(i, [])))
        cols.extend(c)
        rowptr[i + 1] = len(cols)
    colidx = np.array(cols, dtype=np.int32)
    v = np.ones(colidx.size, dtype=dtype) if vals is None else np.asarray(vals, dtype=dtype)
    return HostCSR(m, n, rowptr, colidx, v)


PATHS = {"bitmap": {}, "bitmap_generic": {"register_rows_max_a": 0}, "hash": {"bitmap_span": 0}}


@pytest.mark.parametrize("path", list(PATHS))
@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("seed", range(12))
def test_random_shapes(seed, dtype, path):
    rng = np.random.default_rng(500 + seed)
    m, k, n = (int(x) for x in rng.integers(1, 400, size=3))
    A = random_csr(m, k, float(rng.choice([0.005, 0.02, 0.08])), rng, dtype, "sym", empty_rows=0.1)
    B = random_csr(k, n, float(rng.choice([0.01, 0.05, 0.2])), rng, dtype, "sym", empty_rows=0.1)
    with tuning(**PATHS[path]):
        rowptr, colidx, vals, _ = run_gpu(A, B, validate=True)
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("path", list(PATHS))
@pytest.mark.parametrize("dtype", DTYPES)
def test_uniform_several_tiles(dtype, path):
    # enough rows for many CTAs and a ragged last tile of every kernel
    rng = np.random.default_rng(7)
    A = uniform_csr(40_003, 3_001, 9, rng, dtype, "sym")
    B = uniform_csr(3_001, 5_003, 17, rng, dtype, "sym")
    with tuning(**PATHS[path]):
        rowptr, colidx, vals, info = run_gpu(A, B)
    assert info[f"{path.split('_')[0]}_rows"] == 40_003
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def _banded(m, n, lens, halfwidth, rng, dtype, centre):
    """Rows of the given lengths with distinct columns within halfwidth of centre(i)."""
    rows = {}
    for i, L in enumerate(lens):
        c = int(centre(i))
        lo, hi = max(0, c - halfwidth), min(n, c + halfwidth + 1)
        L = min(L, hi - lo)
        rows[i] = (lo + rng.choice(hi - lo, size=L, replace=False)).tolist()
    M = _csr(m, n, rows, dtype=dtype)
    M.vals = (2 * rng.random(M.nnz) - 1).astype(dtype)
    return M


@pytest.mark.parametrize("b_len", [4, 8])
@pytest.mark.parametrize("dtype", DTYPES)
def test_grouped_register_rows(dtype, b_len):
    """Banded products over more than 65,536 columns whose B rows fit 4 or 8
    lanes: rows of at most 4096 columns are ranked by groups of lanes, several
    rows per warp, with stored-entry counts 0..16 mixed inside every warp,
    repeated columns, a ragged last warp, and wider rows (other bins) between
    them."""
    rng = np.random.default_rng(40 + b_len)
    k = n = 100_000
    B = _banded(k, n, [b_len] * k, 600, rng, dtype, lambda j: j)
    m = 20_011
    lens = rng.integers(0, 17, size=m)
    A = _banded(m, k, lens, 700, rng, dtype, lambda i: i * (k // m))
    wide = rng.choice(m, size=200, replace=False)  # rows spread over a wider range
    rows = {i: A.colidx[A.rowptr[i]:A.rowptr[i + 1]].tolist() for i in range(m)}
    for i in wide:
        L = int(rng.integers(2, 17))
        rows[int(i)] = rng.choice(k, size=L, replace=False).tolist()
    A = _csr(m, k, rows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B, validate=True)
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [2_000, 16_000, 60_000])
def test_bitmap_bins(dtype, n):
    """Rows of every bitmap bin: narrow and wide column ranges, small and large rows."""
    rng = np.random.default_rng(n)
    k = 2500
    B = uniform_csr(k, n, 24, rng, dtype, "sym")
    lens = [2, 3, 6, 11, 20, 40, 90, 200, 330]
    rows = {i: rng.choice(k, size=L, replace=False).tolist() for i, L in enumerate(lens * 20)}
    A = _csr(len(lens) * 20, k, rows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["bitmap_rows"] > 0
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("n", [60_000, 70_000])
@pytest.mark.parametrize("dtype", DTYPES)
def test_every_row_class(dtype, n):
    """Rows of every class: empty, direct, register bitmap, bitmap, hash, dense window.

    With n <= 65,536 the planning pass counts the short rows and leaves the
    others (empty, single-entry, long) to the analysis kernel."""
    rng = np.random.default_rng(11)
    k = 3000
    B = uniform_csr(k, n, 40, rng, dtype, "sym")
    lens = [0, 1, 1, 2, 3, 5, 9, 17, 33, 65, 100, 150, 200, 400, 1000, 2000, 3000]
    rows = {}
    for i, L in enumerate(lens * 3):
        rows[i] = rng.choice(k, size=L, replace=False).tolist()
    A = _csr(len(lens) * 3, k, rows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B, validate=True)
    assert info["direct_rows"] == 6 and info["empty_rows"] == 3
    assert info["dense_rows"] + info["rcd_rows"] + info["wb_rows"] > 0
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_dense_window_path_everywhere(dtype):
    rng = np.random.default_rng(12)
    A = uniform_csr(3000, 800, 6, rng, dtype, "sym")
    B = uniform_csr(800, 9000, 12, rng, dtype, "sym")
    with tuning(hash_max_products=0, dense_width=1024, bitmap_span=0, wide_bitmap_span=0):
        rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["hash_rows"] == 0 and info["dense_rows"] == 3000 and info["dense_slices"] > 3000
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_sort_path_everywhere(dtype):
    rng = np.random.default_rng(13)
    A = uniform_csr(2000, 900, 8, rng, dtype, "sym")
    B = uniform_csr(900, 4000, 20, rng, dtype, "sym")
    with tuning(run_limit=1, bitmap_span=0):
        rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["sorted_rows"] > 0
    assert_matches_oracle(A, B, rowptr, colidx, vals)


HEAVY = {"default": {}, "no_dense_rows": {"dense_rows_max_a": 0}, "wide_bitmap_only": {"dense_rows_max_a": 0, "bitmap_span": 0},
         "sliced_only": {"dense_rows_max_a": 0, "bitmap_span": 0, "wide_bitmap_span": 0, "hash_max_products": 0},
         "dense_rows_few_a": {"dense_rows_max_a": 64}}


@pytest.mark.parametrize("heavy", list(HEAVY))
@pytest.mark.parametrize("dtype", DTYPES)
def test_heavy_rows(heavy, dtype):
    """Hub rows of a skewed product (few stored A entries, long B rows) and
    wide rows with many short B rows, on every heavy-row path."""
    rng = np.random.default_rng(31)
    rp, ci, _ = rmat_pattern(13, 16, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(8192, 8192, rp, ci, (1.0 - rng.random(ci.size)).astype(dtype))
    from synth import row_subset
    from tests._helpers import products_per_row
    lens, ub = np.diff(rp), products_per_row(A, A)
    hubs = np.argsort(lens)[-100:]                               # many stored entries
    fed = np.flatnonzero((ub > 4096) & (lens <= 64))[:300]      # few entries, long (hub) B rows
    light = rng.choice(8192, size=100, replace=False)
    H = row_subset(A, np.unique(np.concatenate([hubs, fed, light])))
    with tuning(**HEAVY[heavy]):
        rowptr, colidx, vals, info = run_gpu(H, A)
    if heavy == "default":
        assert info["rcd_rows"] > 0
    if heavy == "wide_bitmap_only":
        assert info["wb_rows"] > 0
    if heavy == "sliced_only":
        assert info["dense_rows"] > 0
    assert_matches_oracle(H, A, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_direct_rows_long_and_short(dtype):
    """Rows of A with one stored entry copy a scaled B row: B rows of 0 to
    5000 entries around the length where a whole warp takes over (512), among
    many short ones so the lane groups stay small."""
    rng = np.random.default_rng(34)
    n = 20_000
    lens = [0, 1, 3, 31, 32, 33, 511, 512, 513, 1000, 5000]
    rows = {i: rng.choice(n, size=L, replace=False).tolist() for i, L in enumerate(lens)}
    k = 3000
    for i in range(len(lens), k):
        rows[i] = rng.choice(n, size=int(rng.integers(1, 6)), replace=False).tolist()
    B = _csr(k, n, rows, dtype=dtype)
    B.vals = (2 * rng.random(B.nnz) - 1).astype(dtype)
    picks = list(range(len(lens))) * 3 + rng.choice(k, size=400).tolist()
    A = _csr(len(picks), k, {i: [c] for i, c in enumerate(picks)}, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B)
    blen = np.diff(B.rowptr)
    assert info["direct_rows"] == int(np.count_nonzero(blen[picks]))  # an empty B row gives an empty row
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_dense_rows_slice_parts(dtype):
    """Dense heavy rows whose B rows give every kind of part inside a value
    window slice: empty, one entry, just below / at / just above the short-part
    limit (32) and the piece size (128), many pieces, a B row covering all
    65,536 columns, columns on the slice starts and just before them, a B row
    inside one slice; one row with more than 256 stored entries; and rows
    whose output is below, exactly at and one above the value window's size
    (the compact window takes the first two)."""
    rng = np.random.default_rng(33)
    n = 1 << 16
    slice_w = 8192 if dtype == np.float64 else 16384
    lens = [0, 1, 2, 31, 32, 33, 127, 128, 129, 257, 1000, 4000, 20000]
    rows = {i: rng.choice(n, size=L, replace=False).tolist() for i, L in enumerate(lens)}
    rows[len(lens)] = list(range(n))                                       # every column
    rows[len(lens) + 1] = [s * slice_w + d for s in range(n // slice_w) for d in (-1, 0) if 0 <= s * slice_w + d < n]
    rows[len(lens) + 2] = (3 * slice_w + rng.choice(slice_w, size=300, replace=False)).tolist()  # one slice
    x = rng.permutation(n)[:slice_w]                      # exactly one window of distinct columns
    rows[len(lens) + 3] = x.tolist()
    rows[len(lens) + 4] = rng.choice(x, size=500, replace=False).tolist()            # inside x
    outside = np.setdiff1d(np.arange(n), x)
    rows[len(lens) + 5] = rng.choice(x, size=100, replace=False).tolist() + [int(outside[7])]  # one column more
    k = 400
    for i in range(len(lens) + 6, k):
        rows[i] = rng.choice(n, size=int(rng.integers(0, 300)), replace=False).tolist()
    B = _csr(k, n, rows, dtype=dtype)
    B.vals = (2 * rng.random(B.nnz) - 1).astype(dtype)
    special = list(range(len(lens) + 3))
    X = len(lens) + 3
    arows = {0: special, 1: special[:5] + [len(lens)], 2: [len(lens) + 1, len(lens) + 2, 12],
             3: rng.choice(k, size=300, replace=False).tolist(),                 # 300 > 256 entries
             4: [6, 7, 8, 9, 10, 11],                 # output fits one value window
             5: [X, X + 1],                           # output exactly one window wide
             6: [X, X + 2]}                           # one column more than a window
    for i in range(7, 40):
        arows[i] = rng.choice(k, size=int(rng.integers(2, 200)), replace=False).tolist() + [12]
    A = _csr(40, k, arows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["rcd_rows"] >= 38
    assert np.diff(rowptr)[5] == slice_w and np.diff(rowptr)[6] == slice_w + 1
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_dense_rows_many_products_few_columns(dtype):
    """Dense heavy rows with far more products than output entries: 200
    stored entries whose B rows (1000 entries each) share a pool of 6000
    columns, so 200,000 products fall on at most 6000 outputs.  The output fits
    one value window, but the products are too many for the per-piece first
    flags, so the column indices come from the bitmap walk instead."""
    rng = np.random.default_rng(36)
    n = 1 << 16
    pool = rng.choice(n, size=6000, replace=False)
    k = 260
    rows = {i: rng.choice(pool, size=1000, replace=False).tolist() for i in range(k)}
    B = _csr(k, n, rows, dtype=dtype)
    B.vals = (2 * rng.random(B.nnz) - 1).astype(dtype)
    arows = {i: rng.choice(k, size=200, replace=False).tolist() for i in range(6)}
    A = _csr(6, k, arows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["rcd_rows"] == 6
    assert assert_matches_oracle(A, B, rowptr, colidx, vals) <= TOL[np.dtype(dtype)]


@pytest.mark.parametrize("dtype", DTYPES)
def test_wide_heavy_rows(dtype):
    """Rows with thousands of stored A entries over short B rows spanning ~2^20 columns."""
    rng = np.random.default_rng(32)
    k, n = 20_000, 1 << 20
    B = uniform_csr(k, n, 4, rng, dtype, "pos")
    rows = {i: rng.choice(k, size=int(L), replace=False).tolist() for i, L in enumerate([1500, 3000, 6000, 2, 40])}
    A = _csr(5, k, rows, dtype=dtype)
    A.vals = (1.0 - rng.random(A.nnz)).astype(dtype)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["wb_rows"] == 3
    assert_matches_oracle(A, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
def test_wide_rows_cluster_split(dtype):
    """Wide-bitmap rows whose column ranges sit at the edges of the split of a
    row's bitmap over a cluster of CTAs (runs of a power of two of 128-column
    chunks): one chunk (spans 1 and 128), one chunk past a power of two,
    ranges that leave some CTAs of the cluster without a chunk, the full
    2^20 columns, and one row of many stored entries in the same kernel."""
    rng = np.random.default_rng(33)
    n = 1 << 20
    spans = [1, 127, 128, 129, 1024, 1025, 65537, (1 << 19) + 1, (1 << 20) - 5, 1 << 20]
    b_rows, a_rows = [], {}
    for i, s in enumerate(spans):
        c0 = int(rng.integers(0, n - s + 1))
        first = len(b_rows)
        for j in range(40):
            cols = set(int(c) for c in c0 + rng.integers(0, s, size=int(rng.integers(1, 9))))
            if j == 0:
                cols.add(c0)            # the row's range is exactly [c0, c0 + s)
            if j == 39:
                cols.add(c0 + s - 1)
            b_rows.append(sorted(cols))
        a_rows[i] = list(range(first, first + 40))
    hub = len(spans)  # many stored entries over rows spanning all columns
    first = len(b_rows)
    for j in range(3000):
        b_rows.append(sorted(set(int(c) for c in rng.integers(0, n, size=5))))
    a_rows[hub] = list(range(first, first + 3000))
    B = _csr(len(b_rows), n, dict(enumerate(b_rows)), dtype=dtype)
    B.vals = (1.0 - rng.random(B.nnz)).astype(dtype)
    A = _csr(len(spans) + 1, B.nrows, a_rows, dtype=dtype)
    A.vals = (2 * rng.random(A.nnz) - 1).astype(dtype)
    with tuning(hash_max_products=0, bitmap_span=0, dense_rows_max_a=0, register_rows_max_a=0):
        rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["wb_rows"] == len(spans) + 1
    assert_matches_oracle(A, B, rowptr, colidx, vals)
    assert rowptr[1] == 1  # span 1: forty products, one column


@pytest.mark.parametrize("path", list(PATHS))
def test_skewed_rmat_square(path):
    rng = np.random.default_rng(14)
    rp, ci, _ = rmat_pattern(12, 16, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(4096, 4096, rp, ci, (1.0 - rng.random(ci.size)))
    with tuning(**PATHS[path]):
        rowptr, colidx, vals, info = run_gpu(A, A)
    if path == "hash":
        assert info["dense_rows"] + info["rcd_rows"] + info["wb_rows"] > 0 and info["bitmap_rows"] == 0
    else:
        assert info["bitmap_rows"] > 0
    assert_matches_oracle(A, A, rowptr, colidx, vals)


def test_rmat_unit_values_exact():
    rng = np.random.default_rng(15)
    rp, ci, _ = rmat_pattern(11, 16, (0.57, 0.19, 0.19, 0.05), rng)
    A = HostCSR(2048, 2048, rp, ci, np.ones(ci.size))
    rowptr, colidx, vals, _ = run_gpu(A, A)
    err = assert_matches_oracle(A, A, rowptr, colidx, vals)
    assert err == 0.0  # path counts are exact integers in any summation order


@pytest.mark.parametrize("m,k,n", [(0, 5, 3), (4, 0, 3), (4, 5, 0), (1, 1, 1), (7, 3, 1)])
def test_degenerate_shapes(m, k, n):
    rng = np.random.default_rng(m * 100 + k * 10 + n)
    A = random_csr(m, k, 0.6, rng)
    B = random_csr(k, n, 0.6, rng)
    rowptr, colidx, vals, _ = run_gpu(A, B, validate=True)
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def test_all_rows_empty_and_empty_b_rows():
    A = _csr(50, 20, {i: [i % 20] for i in range(0, 50, 2)})
    B = _csr(20, 30, {j: [j, j + 1] for j in range(1, 20, 2)})  # even rows of B empty
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert rowptr[-1] == 0 and info["empty_rows"] == 50


def test_direct_rows_scaled_copy():
    rng = np.random.default_rng(16)
    perm = rng.permutation(500)
    A = HostCSR(500, 500, np.arange(501, dtype=np.int64), perm.astype(np.int32), 2 * rng.random(500) - 1)
    B = uniform_csr(500, 2000, 37, rng)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["direct_rows"] == 500
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def test_single_dense_row_and_wide_output():
    rng = np.random.default_rng(17)
    k, n = 600, 1 << 20
    A = _csr(3, k, {0: list(range(k)), 2: [5, 7]}, dtype=np.float64)
    A.vals = 2 * rng.random(A.nnz) - 1
    B = uniform_csr(k, n, 30, rng)
    rowptr, colidx, vals, info = run_gpu(A, B)
    assert info["wb_rows"] == 1
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def test_cancellation_keeps_structural_zero():
    A = _csr(1, 2, {0: [0, 1]}, vals=[1.0, -1.0])
    B = _csr(2, 3, {0: [0, 2], 1: [0, 1]}, vals=[2.0, 5.0, 2.0, 3.0])
    rowptr, colidx, vals, _ = run_gpu(A, B)
    assert rowptr.tolist() == [0, 3]
    assert colidx.tolist() == [0, 1, 2]
    assert vals.tolist() == [0.0, -3.0, 5.0]


def test_handle_reuse_and_growth():
    """One SpGEMM object re-run, then a second, larger product: scratch grows, results stay exact."""
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(18)
    A = uniform_csr(1000, 700, 5, rng)
    B = uniform_csr(700, 900, 7, rng)
    dA, dB = DeviceCSR.from_host(A), DeviceCSR.from_host(B)
    with SpGEMM(dA, dB) as op:
        outs = []
        for _ in range(3):
            op.symbolic()
            C = op.numeric()
            op.wait()
            outs.append(C.to_host())
    for o in outs[1:]:
        for a, b in zip(outs[0][:2], o[:2]):
            np.testing.assert_array_equal(a, b)
    assert_matches_oracle(A, B, *outs[-1])
    A2 = uniform_csr(30_000, 700, 9, rng)
    rowptr, colidx, vals, _ = run_gpu(A2, B)
    assert_matches_oracle(A2, B, rowptr, colidx, vals)


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("shift", [0, 1, 3])
def test_output_arrays_at_any_alignment(dtype, shift):
    """C's column and value arrays given at an offset of `shift` elements (not
    16-byte aligned unless shift is 0): the register-bitmap rows, copied out
    in 16-byte groups when both arrays are aligned, must give the same C."""
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(35)
    A = uniform_csr(5000, 3000, 12, rng, dtype, "sym")   # 12 entries per row
    B = uniform_csr(3000, 40_000, 30, rng, dtype, "sym")  # 30 per row: 32-lane groups, ~360 entries per C row
    dA, dB = DeviceCSR.from_host(A), DeviceCSR.from_host(B)
    tdt = torch.float32 if dtype == np.float32 else torch.float64
    with SpGEMM(dA, dB) as op:
        nnz = op.symbolic()
        ci = torch.empty(nnz + shift, dtype=torch.int32, device="cuda")[shift:]
        cv = torch.empty(nnz + shift, dtype=tdt, device="cuda")[shift:]
        C = op.numeric(out=DeviceCSR(A.nrows, B.ncols, op.c_rowptr, ci, cv))
        op.wait()
        info = op.plan_info()
        rowptr, colidx, vals = C.to_host()
    assert info["bitmap_rows"] == A.nrows
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def test_many_live_handles():
    """More live products than one block of recycled pinned summaries (64):
    each of 150 open SpGEMM objects keeps its own summary and result, and
    closing them returns the blocks for the next 150."""
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(19)
    A = uniform_csr(300, 200, 4, rng)
    B = uniform_csr(200, 250, 5, rng)
    dA, dB = DeviceCSR.from_host(A), DeviceCSR.from_host(B)
    ref = None
    for _ in range(2):
        ops = [SpGEMM(dA, dB) for _ in range(150)]
        nnzs = [op.symbolic() for op in ops]
        outs = [op.numeric() for op in ops]
        for op in ops:
            op.wait()
        assert len(set(nnzs)) == 1
        hosts = [C.to_host() for C in outs]
        for op in ops:
            op.close()
        for h in hosts[1:]:  # structure is unique; values may differ in rounding (atomic order)
            for a, b in zip(hosts[0][:2], h[:2]):
                np.testing.assert_array_equal(a, b)
        assert_matches_oracle(A, B, *hosts[-1])
        if ref is None:
            ref = hosts[0]
        for a, b in zip(ref[:2], hosts[0][:2]):
            np.testing.assert_array_equal(a, b)


def test_device_count_check_reports_error():
    """A row pointer altered between the passes is caught by the numeric pass's count check."""
    from paper_2606_20855_gb300 import _abi
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(19)
    A = uniform_csr(256, 300, 6, rng)
    B = uniform_csr(300, 5000, 8, rng)
    with SpGEMM(DeviceCSR.from_host(A), DeviceCSR.from_host(B)) as op:
        nnz = op.symbolic()
        # move one entry from row 10 to row 11: every write stays inside [0, nnz)
        op.c_rowptr[11] -= 1
        C = op.numeric()
        with pytest.raises(_abi.WsError) as ei:
            op.wait()
        assert ei.value.status_name == "WS_ERR_DEVICE"
        assert C.nnz == nnz
        # the handle stays usable
        op.symbolic()
        C = op.numeric()
        op.wait()
        rowptr, colidx, vals = C.to_host()
    assert_matches_oracle(A, B, rowptr, colidx, vals)


def test_host_side_errors():
    from paper_2606_20855_gb300 import _abi
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(20)
    A = uniform_csr(10, 8, 3, rng)
    B = uniform_csr(9, 8, 3, rng)
    with pytest.raises(_abi.WsError) as ei:
        with SpGEMM(DeviceCSR.from_host(A), DeviceCSR.from_host(B)) as op:
            op.symbolic()
    assert ei.value.status_name == "WS_ERR_SHAPE"
    B32 = uniform_csr(8, 8, 3, rng, np.float32)
    with pytest.raises(TypeError):
        SpGEMM(DeviceCSR.from_host(A), DeviceCSR.from_host(B32))
    # invalid CSR: unsorted columns, duplicate, out of range, non-monotone rowptr
    good = uniform_csr(6, 10, 3, rng)
    bads = []
    b = HostCSR(6, 10, good.rowptr.copy(), good.colidx.copy(), good.vals.copy())
    b.colidx[0], b.colidx[1] = b.colidx[1], b.colidx[0]
    bads.append(b)
    b = HostCSR(6, 10, good.rowptr.copy(), good.colidx.copy(), good.vals.copy())
    b.colidx[4] = b.colidx[3]
    bads.append(b)
    b = HostCSR(6, 10, good.rowptr.copy(), good.colidx.copy(), good.vals.copy())
    b.colidx[-1] = 10
    bads.append(b)
    b = HostCSR(6, 10, good.rowptr.copy(), good.colidx.copy(), good.vals.copy())
    b.rowptr[2], b.rowptr[3] = b.rowptr[3], b.rowptr[2]
    bads.append(b)
    for bad in bads:
        with pytest.raises(_abi.WsError) as ei:
            SpGEMM(DeviceCSR.from_host(bad), DeviceCSR.from_host(uniform_csr(10, 4, 2, rng)), validate=True)
        assert ei.value.status_name == "WS_ERR_INVALID_CSR"
    # numeric before symbolic
    with SpGEMM(DeviceCSR.from_host(good), DeviceCSR.from_host(uniform_csr(10, 4, 2, rng))) as op:
        with pytest.raises(RuntimeError):
            op.numeric()
        h = op._hC
        with pytest.raises(_abi.WsError) as ei:
            _abi.ws_spgemm_numeric(op._hA, op._hB, h, 0, 0, torch.cuda.current_stream().cuda_stream)
        assert ei.value.status_name == "WS_ERR_STATE"
