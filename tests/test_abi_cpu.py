"""The C-ABI library builds, loads and exports every entry point of include/ws_spgemm.h.

Host-only checks: argument validation that returns before any CUDA call, the
status strings and the tuning knob.  No kernel runs here.
"""
from __future__ import annotations

import ctypes
import os
import re

import pytest

from paper_2606_20855_gb300 import _abi
from paper_2606_20855_gb300 import build as pkg_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ws_spgemm.h")


@pytest.fixture(scope="module")
def lib():
    pkg_build.build()
    return _abi.load()


def declared_functions() -> list[str]:
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ws_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_four_calls():
    names = declared_functions()
    for n in ("ws_csr_create", "ws_spgemm_symbolic", "ws_spgemm_numeric", "ws_csr_destroy"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert names, "no declarations parsed"
    for n in names:
        assert hasattr(lib, n), f"{n} not exported"
    assert sorted(n for n, _, _ in _abi.SIGNATURES) == names


def test_status_strings(lib):
    for code in range(10):
        s = _abi.ws_status_string(code)
        assert s and s != "unknown status"
    assert _abi.ws_status_string(12345) == "unknown status"


def test_host_argument_errors(lib):
    h = ctypes.c_void_p()
    # NULL out pointer
    assert lib.ws_csr_create(None, 1, 1, 0, 8, None, None, 2, 0, None) == 1
    # negative sizes / unknown dtype / missing rowptr
    assert lib.ws_csr_create(ctypes.byref(h), -1, 1, 0, 8, None, None, 2, 0, None) == 1
    assert lib.ws_csr_create(ctypes.byref(h), 1, 1, 0, 8, None, None, 7, 0, None) == 1
    assert lib.ws_csr_create(ctypes.byref(h), 1, 1, 0, None, None, None, 2, 0, None) == 1
    assert lib.ws_csr_create(ctypes.byref(h), 1, 1, 5, 8, None, None, 2, 0, None) == 1
    assert "NULL" in _abi.ws_last_error()
    # too many columns for int32 indices
    assert lib.ws_csr_create(ctypes.byref(h), 1, 2**31, 0, 8, None, None, 2, 0, None) == 5
    nnz = ctypes.c_int64()
    assert lib.ws_spgemm_symbolic(None, None, None, ctypes.byref(nnz), None) == 1
    assert lib.ws_spgemm_numeric(None, None, None, None, None, None) == 1
    assert lib.ws_spgemm_wait(None, None) == 1
    assert lib.ws_csr_destroy(None) == 0
    assert lib.ws_csr_nnz(None, ctypes.byref(nnz)) == 1
    with pytest.raises(_abi.WsError) as ei:
        _abi.ws_spgemm_symbolic(0, 0, 0, 0)
    assert ei.value.status_name == "WS_ERR_INVALID_ARG"


def test_tuning_knob_validation(lib):
    try:
        for key, bad in [(1, -1), (1, 5000), (2, 0), (3, 1000), (3, 20480), (4, -1), (4, 65537), (5, 17), (6, 8193), (7, (1 << 20) + 1), (9, 1)]:
            with pytest.raises(_abi.WsError):
                _abi.ws_set_tuning(key, bad)
        _abi.ws_set_tuning("hash_max_products", 0)
        _abi.ws_set_tuning("run_limit", 8)
        _abi.ws_set_tuning("dense_width", 2048)
        _abi.ws_set_tuning("bitmap_span", 0)
    finally:
        for k, v in _abi.TUNING_DEFAULTS.items():
            _abi.ws_set_tuning(k, v)


def test_binding_refuses_to_run_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(_abi, "_lib", None)
    monkeypatch.setattr(_abi, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        _abi.load()
