"""Seeded synthetic inputs shared by the oracle checks, the GPU tests and the bench.

Holds no lineage arithmetic: it draws counts, per-child results, arrival and
readiness orders, and fills result payload bytes from a counter-based hash.
"""
from .configs import (CONFIGS, FAILED, DROPPED, PRESENT, SUPPRESSED, Level, Workload,
                      docpage, skew, streaming, subset, tiny, video)
from .payload import fill_host_arena, level_arena, mix64, record_bytes, records_concat

__all__ = [
    "CONFIGS", "PRESENT", "DROPPED", "FAILED", "SUPPRESSED", "Level", "Workload",
    "tiny", "docpage", "video", "skew", "streaming", "subset",
    "fill_host_arena", "level_arena", "mix64", "record_bytes", "records_concat",
]
