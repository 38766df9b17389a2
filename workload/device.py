"""Device-side input staging: payload fill into a torch uint8 arena."""
from __future__ import annotations

import ctypes as C
import os

from .build import LIB, build

_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            build()
        L = C.CDLL(LIB)
        L.wl_fill_payload.argtypes = [C.c_void_p, C.c_uint64, C.c_void_p, C.c_void_p, C.c_uint64,
                                      C.c_uint64, C.c_void_p]
        L.wl_fill_payload.restype = C.c_int
        _lib = L
    return _lib


def fill_payload(arena, off, length, seed: int, stream=None) -> None:
    """Write every child's record into ``arena`` (torch.uint8 on the GPU).
    ``off`` (int64/uint64) and ``length`` (int32/uint32) are device tensors
    indexed by child."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    rc = _load().wl_fill_payload(arena.data_ptr(), arena.numel(), off.data_ptr(),
                                 length.data_ptr(), off.numel(), int(seed) & ((1 << 64) - 1),
                                 stream.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"wl_fill_payload failed with CUDA error {rc}")
