"""GB300 (sm_103a) lineage expand / FIFO batch / gather-commit / assemble.

The compute path is the CUDA library ``libro_gb300.so`` behind the C ABI in
``include/rayorch_gpu.h``; this package is its ctypes binding (same function
names) plus the in-tree build step.
"""
from ._binding import (EXPORTS, KERNELS, ro_ctx_profile, ro_ctx_profile_read, RO_ACCEPT, RO_DROPPED, RO_E_CAPACITY, RO_E_CUDA, RO_E_INVAL,
                       RO_E_OOM, RO_E_OVERFLOW, RO_E_STATE, RO_E_TIMEOUT, RO_FAILED, RO_GROUP_FAILURE, RO_OK,
                       RO_PENDING, RO_PRESENT, RO_REJ_BARRIER, RO_REJ_DUPLICATE, RO_REJ_INVALID,
                       RO_REJ_NOT_INFLIGHT, RO_REJ_STALE_GEN, RO_SUPPRESSED, RoError, load,
                       ro_assemble, ro_assemble_list, ro_batch_ready, ro_batch_ready_calls, ro_batch_ready_parent, ro_ctx_selftest_timeout, ro_filter_reports, ro_ctx_create, ro_ctx_destroy, ro_ctx_reset,
                       ro_ctx_set_streams, ro_ctx_set_call_streams, ro_ctx_join, ro_ctx_stats, ro_ctx_sync, ro_expand, ro_expand_noalloc, ro_gather_commit, ro_retry,
                       ro_last_error)

__all__ = [n for n in dir() if n.startswith(("ro_", "RO_"))] + ["RoError", "load", "EXPORTS", "KERNELS"]
