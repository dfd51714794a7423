"""GB300 (sm_103a) SpGEMM: C = A*B for CSR matrices, computed by hand-written CUDA kernels;
also the elementwise operations C = A + B and C = A .* B and the sparse
matrix - sparse vector product y = A x.

The C ABI lives in include/ws_spgemm.h and libws_spgemm.so (built by
``paper_2606_20855_gb300.build``).  ``_abi`` is the ctypes binding with the
same function names; ``spgemm`` holds the PyTorch-facing wrapper.  Importing
this package loads nothing; the library is loaded on first use.
"""

__all__ = ["DeviceCSR", "SpGEMM", "SpGEMMOuter", "spgemm", "spgemm_outer", "submatrix", "Ewise", "ewise", "SpMSpV", "spmspv"]


def __getattr__(name):
    if name in __all__:
        from . import spgemm as _m
        return getattr(_m, name)
    raise AttributeError(name)
