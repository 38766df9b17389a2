"""Plain single-threaded CPU oracle for the lineage expand/gather path.

TEST INFRASTRUCTURE ONLY: imported by the tests, ``__graft_entry__.smoke()``
and the benchmark's CPU-baseline leg; never by the GPU library.
"""
from .oracle import (ACCEPT, DROPPED, E_CAPACITY, E_INVAL, E_OVERFLOW, FAILED, GROUP_FAILURE, OK,
                     PENDING, PRESENT, REJ_BARRIER, REJ_DUPLICATE, REJ_INVALID, REJ_NOT_INFLIGHT,
                     REJ_STALE_GEN, SUPPRESSED, OracleCtx, OracleError)

__all__ = ["OracleCtx", "OracleError", "OK", "E_INVAL", "E_CAPACITY", "E_OVERFLOW",
           "PENDING", "PRESENT", "DROPPED", "FAILED", "SUPPRESSED", "ACCEPT", "REJ_INVALID",
           "REJ_NOT_INFLIGHT", "REJ_STALE_GEN", "REJ_DUPLICATE", "REJ_BARRIER", "GROUP_FAILURE"]
