"""ctypes declarations of libblr.so (the C ABI in include/blr.h).

The library is built in-tree by ``paper_2406_12580_gb300.build``. There is no
fallback: if the shared library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

BLR_F32 = 0
BLR_BF16 = 1

BLR_OK = 0
BLR_ERR_INVALID_ARG = 1
BLR_ERR_UNSUPPORTED = 2
BLR_ERR_CUDA = 3
BLR_ERR_TIMEOUT = 4
BLR_ERR_WORKSPACE = 5


class blr_desc(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int64), ("L", ctypes.c_int64), ("D", ctypes.c_int64),
                ("io", ctypes.c_int), ("c", ctypes.c_float)]


_VP = ctypes.c_void_p
_SZ = ctypes.c_size_t
_ST = ctypes.c_int
_DESC_P = ctypes.POINTER(blr_desc)

# name -> (restype, argtypes); the argument order of include/blr.h
SIGNATURES = {
    "blr_workspace_bytes": (_SZ, [_DESC_P]),
    "blr_scan_family": (ctypes.c_int, [_DESC_P, ctypes.c_int]),
    "blr_scan_fwd": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]),
    "blr_scan_bwd": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]),
    "blr_step": (_ST, [ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_float, _VP, _VP, _VP,
                       _VP, _VP, _VP]),
    "blr_workspace_status": (_ST, [_DESC_P, _VP, _SZ, _VP]),
    "blr_status_string": (ctypes.c_char_p, [_ST]),
    "blr_last_error_string": (ctypes.c_char_p, []),
    "blr_selftest_wait_timeout": (_ST, [_DESC_P, _VP, _SZ, ctypes.c_uint64, _VP]),
    "blr_scan_fwd_noalloc": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP]),
    "blr_scan_fwd_varlen": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]),
    "blr_scan_bwd_varlen": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                  _VP, _SZ, _VP]),
    "blr_steps": (_ST, [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                        ctypes.c_float, _VP, _VP, _VP, _VP, _VP, _VP, _VP]),
    "blr_scan_fwd_gated": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]),
    "blr_scan_bwd_gated": (_ST, [_DESC_P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                 _VP, _VP, _SZ, _VP]),
}

_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIBRARY


def load() -> ctypes.CDLL:
    """Load libblr.so once. Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            path = library_path()
            if not os.path.exists(path):
                raise RuntimeError(
                    f"{path} is missing: build it with `python -m paper_2406_12580_gb300.build` "
                    "(there is no CPU fallback)")
            lib = ctypes.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(lib, name)
                fn.restype = res
                fn.argtypes = args
            _lib = lib
        return _lib
