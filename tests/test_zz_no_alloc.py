"""The allocation-free row-pointer scan, ws_rowptr_scan_static, called through the C ABI.

Some callers cannot allocate device memory where they build a row pointer: a
framework that owns all device memory through its own pool, or a
latency-critical loop where cudaMalloc/cudaFree would block on the whole
device.  For them the library keeps the scan's scratch in a fixed array.

Checks:
- the result equals numpy's cumulative sum of the host counts (a check that
  shares nothing with the library's scan), at sizes that take the one-launch
  path, the three-launch path with a ragged tail, the multi-round scan of the
  tile sums (more than 1024 tiles) and exactly the 16,777,216-row limit;
- it equals the row pointer that the regular symbolic pass
  (ws_spgemm_symbolic) writes for the same product, on two calls in a row
  with different sizes (the second call must not see the first call's
  leftovers in the shared array);
- rowptr[0] is set to 0 whatever it held, also for zero rows;
- sizes beyond the fixed scratch are refused.
The file is named to be collected last.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import uniform_csr

pytestmark = pytest.mark.gpu

MAX_ROWS = 1 << 24


def _scan(rp, m):
    from paper_2606_20855_gb300 import _abi
    _abi.ws_rowptr_scan_static(rp.data_ptr(), m, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()


@pytest.mark.parametrize("m", [1, 16_384, 16_385, 300_001, 4_194_305, MAX_ROWS])
def test_static_scan_matches_numpy_cumsum(m):
    rng = np.random.default_rng(m)
    counts = rng.integers(0, 1000, size=m, dtype=np.int64)
    want = np.zeros(m + 1, dtype=np.int64)
    np.cumsum(counts, out=want[1:])
    rp = torch.empty(m + 1, dtype=torch.int64, device="cuda")
    rp[1:] = torch.from_numpy(counts).cuda()
    rp[0] = -987_654_321  # ignored on entry, must become 0
    _scan(rp, m)
    np.testing.assert_array_equal(rp.cpu().numpy(), want)


def _reference_rowptr(m, k, n, r_a, r_b, seed):
    """C.rowptr of A*B from the regular symbolic pass."""
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpGEMM
    rng = np.random.default_rng(seed)
    A = uniform_csr(m, k, r_a, rng)
    B = uniform_csr(k, n, r_b, rng)
    with SpGEMM(DeviceCSR.from_host(A), DeviceCSR.from_host(B)) as op:
        op.symbolic()
        return op.c_rowptr.clone()


def test_static_scan_matches_symbolic_rowptr_twice():
    # two products of different sizes; the first spans many scan tiles and a ragged tail
    for m, k, n, ra, rb, seed in [(300_001, 5_000, 70_000, 7, 9, 1), (9_999, 700, 3_000, 5, 4, 2)]:
        ref = _reference_rowptr(m, k, n, ra, rb, seed)
        rp = torch.empty_like(ref)
        rp[1:] = ref[1:] - ref[:-1]  # per-row counts
        rp[0] = 123_456_789          # ignored on entry, must become 0
        _scan(rp, m)
        assert torch.equal(rp, ref)


def test_static_scan_zero_rows_and_refusal():
    from paper_2606_20855_gb300 import _abi
    rp = torch.full((2,), 55, dtype=torch.int64, device="cuda")
    _scan(rp, 0)
    assert int(rp[0]) == 0 and int(rp[1]) == 55  # only rowptr[0] is written
    with pytest.raises(_abi.WsError) as ei:
        _abi.ws_rowptr_scan_static(rp.data_ptr(), MAX_ROWS + 1, torch.cuda.current_stream().cuda_stream)
    assert ei.value.status_name == "WS_ERR_OVERFLOW"
