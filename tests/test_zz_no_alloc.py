"""The allocation-free row-pointer scan, ws_rowptr_scan_static, called through the C ABI.

Some callers cannot allocate device memory where they build a row pointer: a
framework that owns all device memory through its own pool, or a
latency-critical loop where cudaMalloc/cudaFree would block on the whole
device.  For them the library keeps the scan's scratch in a fixed array.
This test checks that the entry point reproduces the row pointer that the
regular symbolic pass (ws_spgemm_symbolic) writes for the same product, on two
calls in a row with different sizes (the second call must not see the first
call's leftovers), and that sizes beyond the fixed scratch are refused.  The
file is named to be collected last.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import uniform_csr

pytestmark = pytest.mark.gpu


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
    from paper_2606_20855_gb300 import _abi
    stream = torch.cuda.current_stream().cuda_stream
    # two products of different sizes; the first spans many scan tiles and a ragged tail
    for m, k, n, ra, rb, seed in [(300_001, 5_000, 70_000, 7, 9, 1), (9_999, 700, 3_000, 5, 4, 2)]:
        ref = _reference_rowptr(m, k, n, ra, rb, seed)
        rp = torch.empty_like(ref)
        rp[1:] = ref[1:] - ref[:-1]  # per-row counts
        rp[0] = 123_456_789          # ignored on entry, must become 0
        _abi.ws_rowptr_scan_static(rp.data_ptr(), m, stream)
        torch.cuda.synchronize()
        assert torch.equal(rp, ref)


def test_static_scan_refuses_sizes_beyond_its_scratch():
    from paper_2606_20855_gb300 import _abi
    rp = torch.zeros(2, dtype=torch.int64, device="cuda")
    with pytest.raises(_abi.WsError) as ei:
        _abi.ws_rowptr_scan_static(rp.data_ptr(), (1 << 24) + 1, torch.cuda.current_stream().cuda_stream)
    assert ei.value.status_name == "WS_ERR_OVERFLOW"
    _abi.ws_rowptr_scan_static(rp.data_ptr(), 0, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert int(rp[0]) == 0
