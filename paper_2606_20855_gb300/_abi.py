"""ctypes binding of the C ABI in include/ws_spgemm.h.

Argument marshalling only: every function here has the name and the
arguments of the C entry point it wraps (device pointers and streams are
passed as integers) and raises :class:`WsError` on a non-OK status.  All
computation happens in libws_spgemm.so; if the library is missing the
binding raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libws_spgemm.so")

WS_F32 = 1
WS_F64 = 2

STATUS_NAMES = {
    0: "WS_OK",
    1: "WS_ERR_INVALID_ARG",
    2: "WS_ERR_INVALID_CSR",
    3: "WS_ERR_SHAPE",
    4: "WS_ERR_DTYPE",
    5: "WS_ERR_OVERFLOW",
    6: "WS_ERR_ALLOC",
    7: "WS_ERR_CUDA",
    8: "WS_ERR_DEVICE",
    9: "WS_ERR_STATE",
}

# (name, restype, argtypes) for every entry point of include/ws_spgemm.h
_i64, _i32, _p = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
SIGNATURES = [
    ("ws_csr_create", _i32, [ctypes.POINTER(_p), _i64, _i64, _i64, _p, _p, _p, _i32, _i32, _p]),
    ("ws_spgemm_symbolic", _i32, [_p, _p, _p, ctypes.POINTER(_i64), _p]),
    ("ws_spgemm_numeric", _i32, [_p, _p, _p, _p, _p, _p]),
    ("ws_spgemm_wait", _i32, [_p, _p]),
    ("ws_csr_destroy", _i32, [_p]),
    ("ws_status_string", ctypes.c_char_p, [_i32]),
    ("ws_last_error", ctypes.c_char_p, []),
    ("ws_csr_nnz", _i32, [_p, ctypes.POINTER(_i64)]),
    ("ws_spgemm_plan_info", _i32, [_p, ctypes.POINTER(_i64), _i32]),
    ("ws_set_tuning", _i32, [_i32, _i64]),
    ("ws_rowptr_scan_static", _i32, [_p, _i64, _p]),
    ("ws_ewise_symbolic", _i32, [_p, _p, _p, _i32, ctypes.POINTER(_i64), _p]),
    ("ws_ewise_numeric", _i32, [_p, _p, _p, _p, _p, _p]),
    ("ws_spmspv", _i32, [_p, _i64, _p, _p, _p, _p, ctypes.POINTER(_i64), _p]),
    ("ws_csr_submatrix_symbolic", _i32, [_p, _i64, _i64, _i64, _i64, _p, ctypes.POINTER(_i64), _p]),
    ("ws_csr_submatrix_numeric", _i32, [_p, _p, _p, _p, _p]),
    ("ws_spgemm_outer_symbolic", _i32, [_p, _p, _p, _i32, ctypes.POINTER(_i64), _p]),
    ("ws_spgemm_outer_numeric", _i32, [_p, _p, _p, _p, _p, _p]),
]

EWISE_OPS = {"add": 1, "mul": 2}  # ws_ewise_op_t


class WsError(RuntimeError):
    """A non-OK ws_status_t from the library."""

    def __init__(self, func: str, status: int, detail: str):
        self.status = status
        self.status_name = STATUS_NAMES.get(status, str(status))
        super().__init__(f"{func}: {self.status_name}: {detail}")


_lib = None


def load():
    """Loads libws_spgemm.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing; build it with `python -c 'import __graft_entry__ as g; g.build()'` "
                "(no CPU fallback exists)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, res, args in SIGNATURES:
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _check(func: str, status: int) -> None:
    if status != 0:
        lib = load()
        detail = (lib.ws_last_error() or b"").decode(errors="replace")
        raise WsError(func, status, detail)


def ws_csr_create(nrows: int, ncols: int, nnz: int, rowptr: int, colidx: int, vals: int, dtype: int,
                  validate: bool, stream: int) -> int:
    h = ctypes.c_void_p()
    _check("ws_csr_create", load().ws_csr_create(ctypes.byref(h), nrows, ncols, nnz, rowptr or None,
                                                 colidx or None, vals or None, dtype, int(bool(validate)),
                                                 stream or None))
    return h.value


def ws_spgemm_symbolic(A: int, B: int, C: int, stream: int) -> int:
    nnz = ctypes.c_int64(-1)
    _check("ws_spgemm_symbolic", load().ws_spgemm_symbolic(A, B, C, ctypes.byref(nnz), stream or None))
    return nnz.value


def ws_spgemm_numeric(A: int, B: int, C: int, c_colidx: int, c_vals: int, stream: int) -> None:
    _check("ws_spgemm_numeric", load().ws_spgemm_numeric(A, B, C, c_colidx or None, c_vals or None,
                                                         stream or None))


def ws_spgemm_outer_symbolic(A: int, B: int, C: int, parts: int, stream: int) -> int:
    nnz = ctypes.c_int64(-1)
    _check("ws_spgemm_outer_symbolic", load().ws_spgemm_outer_symbolic(A, B, C, int(parts), ctypes.byref(nnz),
                                                                       stream or None))
    return nnz.value


def ws_spgemm_outer_numeric(A: int, B: int, C: int, c_colidx: int, c_vals: int, stream: int) -> None:
    _check("ws_spgemm_outer_numeric", load().ws_spgemm_outer_numeric(A, B, C, c_colidx or None, c_vals or None,
                                                                     stream or None))


def ws_ewise_symbolic(A: int, B: int, C: int, op, stream: int) -> int:
    k = EWISE_OPS[op] if isinstance(op, str) else int(op)
    nnz = ctypes.c_int64(-1)
    _check("ws_ewise_symbolic", load().ws_ewise_symbolic(A, B, C, k, ctypes.byref(nnz), stream or None))
    return nnz.value


def ws_ewise_numeric(A: int, B: int, C: int, c_colidx: int, c_vals: int, stream: int) -> None:
    _check("ws_ewise_numeric", load().ws_ewise_numeric(A, B, C, c_colidx or None, c_vals or None,
                                                       stream or None))


def ws_spmspv(At: int, nnz_x: int, x_idx: int, x_vals: int, y_idx: int, y_vals: int, stream: int) -> int:
    nnz = ctypes.c_int64(-1)
    _check("ws_spmspv", load().ws_spmspv(At, nnz_x, x_idx or None, x_vals or None, y_idx or None, y_vals or None,
                                         ctypes.byref(nnz), stream or None))
    return nnz.value


def ws_csr_submatrix_symbolic(A: int, r0: int, r1: int, c0: int, c1: int, S: int, stream: int) -> int:
    nnz = ctypes.c_int64(-1)
    _check("ws_csr_submatrix_symbolic", load().ws_csr_submatrix_symbolic(A, r0, r1, c0, c1, S, ctypes.byref(nnz),
                                                                         stream or None))
    return nnz.value


def ws_csr_submatrix_numeric(A: int, S: int, s_colidx: int, s_vals: int, stream: int) -> None:
    _check("ws_csr_submatrix_numeric", load().ws_csr_submatrix_numeric(A, S, s_colidx or None, s_vals or None,
                                                                       stream or None))


def ws_spgemm_wait(C: int, stream: int) -> None:
    _check("ws_spgemm_wait", load().ws_spgemm_wait(C, stream or None))


def ws_csr_destroy(h) -> None:
    _check("ws_csr_destroy", load().ws_csr_destroy(h or None))


def ws_status_string(status: int) -> str:
    return load().ws_status_string(status).decode()


def ws_last_error() -> str:
    return (load().ws_last_error() or b"").decode(errors="replace")


def ws_csr_nnz(h: int) -> int:
    v = ctypes.c_int64(0)
    _check("ws_csr_nnz", load().ws_csr_nnz(h, ctypes.byref(v)))
    return v.value


PLAN_INFO_KEYS = ("empty_rows", "direct_rows", "hash_rows", "sorted_rows", "dense_rows", "dense_slices",
                  "products", "symbolic_launches", "numeric_launches", "bitmap_rows", "rcd_rows", "wb_rows")


def ws_spgemm_plan_info(C: int) -> dict:
    arr = (ctypes.c_int64 * len(PLAN_INFO_KEYS))()
    _check("ws_spgemm_plan_info", load().ws_spgemm_plan_info(C, arr, len(PLAN_INFO_KEYS)))
    return dict(zip(PLAN_INFO_KEYS, list(arr)))


TUNING_KEYS = {"hash_max_products": 1, "run_limit": 2, "dense_width": 3, "bitmap_span": 4, "register_rows_max_a": 5,
               "dense_rows_max_a": 6, "wide_bitmap_span": 7, "ewise_lanes": 8, "ewise_chunk": 9}
TUNING_DEFAULTS = {"hash_max_products": 4096, "run_limit": 64, "dense_width": 0, "bitmap_span": 65536,
                   "register_rows_max_a": 16, "dense_rows_max_a": 8192, "wide_bitmap_span": 1 << 20,
                   "ewise_lanes": -1, "ewise_chunk": 64}


def ws_set_tuning(key, value: int) -> None:
    k = TUNING_KEYS[key] if isinstance(key, str) else int(key)
    _check("ws_set_tuning", load().ws_set_tuning(k, int(value)))


def ws_rowptr_scan_static(rowptr: int, nrows: int, stream: int) -> None:
    """Allocation-free row-pointer scan (see include/ws_spgemm.h): rowptr[1:]
    holds per-row counts on entry and the prefix sums on exit."""
    status = load().ws_rowptr_scan_static(rowptr or None, nrows, stream or None)
    if status != 0:
        raise WsError("ws_rowptr_scan_static", status, STATUS_NAMES.get(status, str(status)))
