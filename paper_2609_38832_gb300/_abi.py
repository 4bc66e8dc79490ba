"""ctypes declarations of the C ABI in include/namoh.h (libnamoh.so, built in-tree)."""
from __future__ import annotations

import ctypes
import os
import re
import threading

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libnamoh.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "namoh.h")

NAMOH_OK = 0
NAMOH_ERR_INVALID_ARG = -1
NAMOH_ERR_UNSUPPORTED = -2
NAMOH_ERR_WORKSPACE = -3
NAMOH_ERR_CUDA = -4

NAMOH_DEV_NONFINITE_SCORE = 0x1
NAMOH_DEV_CAPACITY = 0x2
NAMOH_DEV_TIMEOUT = 0x4
NAMOH_DEV_BAD_SEQLENS = 0x8

NAMOH_ROPE_INTERLEAVED = 0x1
NAMOH_ROPE_GLOBAL = 0x2

_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_F = ctypes.c_float
_U = ctypes.c_uint

SIGNATURES = {
    "namoh_status_string": (ctypes.c_char_p, [_I]),
    "namoh_version": (_I, []),
    "namoh_last_error_string": (ctypes.c_char_p, []),
    "namoh_route_workspace_size": (_SZ, [_I, _I, _I, _I]),
    "namoh_route": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "namoh_route_biased": (_I, [_P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "namoh_route_varlen": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "namoh_route_noalloc": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P]),
    "namoh_prefill_workspace_size": (_SZ, [_I, _I, _I, _I, _I, _I]),
    "namoh_prefill": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _P, _P, _P, _I64, _P, _P,
                           _SZ, _P, _P]),
    "namoh_rope_pack": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _P, _I64, _P, _P, _SZ,
                             _P]),
    "namoh_prefill_ex": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _P, _P, _P, _I64,
                              _P, _P, _SZ, _P, _P]),
    "namoh_prefill_varlen_workspace_size": (_SZ, [_I, _I, _I, _I, _I, _I, _I]),
    "namoh_prefill_varlen": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _P, _P,
                                  _P, _I64, _P, _P, _SZ, _P, _P]),
    "namoh_rope_pack_ex": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _P, _P, _I64, _P,
                                _P, _SZ, _P]),
    "namoh_attention_plan_size": (_SZ, [_I, _I, _I, _I, _I]),
    "namoh_attention_plan": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _SZ, _P]),
    "namoh_attention": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _P, _I64, _P, _SZ, _P, _P, _P]),
    "namoh_attention_timeout_probe": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _P, _SZ, _P,
                                           ctypes.c_uint64, _P, _P]),
    "namoh_proj_workspace_size": (_SZ, [_I, _I, _I, _I, _I, _I]),
    "namoh_proj_qkv": (_I, [_P, _I, _I, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "namoh_proj_out": (_I, [_P, _I, _I, _P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _SZ, _P, _P]),
    "namoh_sa_mask_words": (_I, [_I, _I]),
    "namoh_sa_prefill_workspace_size": (_SZ, [_I, _I, _I, _I, _I, _I, _I]),
    "namoh_sa_prefill": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P,
                              _P, _P, _I64, _P, _P, _SZ, _P, _P]),
    "namoh_shared_workspace_size": (_SZ, [_I, _I, _I, _I]),
    "namoh_shared_prefill": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _I64, _P, _P, _SZ, _P,
                                  _P]),
    "namoh_shared_decode_workspace_size": (_SZ, [_I, _I, _I]),
    "namoh_shared_decode": (_I, [_P, _P, _P, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _I64, _P, _P, _SZ, _P, _P]),
    "namoh_decode_workspace_size": (_SZ, [_I, _I, _I, _I, _I]),
    "namoh_decode": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _I64, _P, _P, _SZ, _P,
                          _P]),
    "namoh_decode_ex": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _F, _U, _P, _P, _P, _P, _P, _P, _I64, _P, _P,
                             _SZ, _P, _P]),
}


class NamohError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        text = load().namoh_status_string(status).decode() if _lib is not None else str(status)
        if status == NAMOH_ERR_CUDA and _lib is not None:
            text += ": " + _lib.namoh_last_error_string().decode()
        super().__init__(f"{fn} returned {status} ({text})")


def header_functions() -> list[str]:
    """Names of the entry points declared in include/namoh.h."""
    src = open(HEADER).read()
    return sorted(set(re.findall(r"NAMOH_API\s+[\w\s\*]+?\b(namoh_\w+)\s*\(", src)))


def load():
    """Load libnamoh.so.  Raises if it has not been built: there is no fallback path."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2609_38832_gb300.build.build() "
                               "(or __graft_entry__.build()); there is no CPU fallback")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def check(fn: str, status: int):
    if status != NAMOH_OK:
        raise NamohError(fn, status)
