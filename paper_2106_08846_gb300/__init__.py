"""GB300 (sm_103a) block-sparse-row x dense product, Y = X W^T + b.

The product at the centre of "Algorithm to Compilation Co-design" (Section
2.2): a pruned weight stored in BSR form (data, indices, indptr) multiplied
with dense activations. The compute lives in libbsr_gb300.so (include/bsr.h);
this package is its ctypes binding and its build script.
"""
from .bsrlib import (  # noqa: F401
    BSR_BF16, BSR_F32, BsrError, Handle, Plan, bsr_check_device_status, bsr_create, bsr_destroy,
    bsr_from_dense, bsr_get_schedule, bsr_reserve, bsr_spmm, bsr_spmm_batch, bsr_spmm_noalloc, bsr_status_str, load,
    bsr_plan_create, parse_schedule,
)
