"""Seeded synthetic inputs shared by the oracle tests, the CUDA tests and the benchmark.

Holds input generation only; no part of the sparse product is computed here.
"""
from .matrices import *  # noqa: F401,F403
from .matrices import (EWISE_WORKLOADS, SPMSPV_WORKLOADS, HostCSR, WORKLOADS, WORKLOAD_ORDER,  # noqa: F401
                       ewise_workload, permute_symmetric, row_subset, sparse_vector, spmspv_workload,
                       transpose_csr, workload)
