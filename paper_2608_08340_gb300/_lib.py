"""ctypes declarations of the C ABI in include/oprag.h (argument marshalling
only).  Loading fails loudly when the CUDA library has not been built: there
is no fallback implementation."""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

OPRAG_F32 = 0
OPRAG_BF16 = 1
OPRAG_K_MAX = 256
OPRAG_OPT_PATH = 1
OPRAG_OPT_BLOCK_N = 2
OPRAG_OPT_TIMING = 3
OPRAG_OPT_PAIR = 4
OPRAG_OPT_BOUND_TAG = 5
OPRAG_OPT_GRAPH = 6
OPRAG_OPT_WAIT_LIMIT = 7
OPRAG_OPT_PHASES = 8
OPRAG_OPT_LEX_GATHER = 9

ERRORS = {
    0: "OK",
    -1: "INVALID_ARG",
    -2: "RANGE",
    -3: "OOM",
    -4: "CUDA",
    -5: "NOT_READY",
    -6: "DEVICE",
}

# name -> (restype, argtypes); mirrors include/oprag.h
_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_F = ctypes.c_float
SIGNATURES = {
    "oprag_index_create": (_I32, [ctypes.POINTER(_P), _P, _I64, _I32, _I32, _I32, _I32]),
    "oprag_index_destroy": (None, [_P]),
    "oprag_index_info": (_I32, [_P, ctypes.POINTER(_I64), ctypes.POINTER(_I32),
                                ctypes.POINTER(_I32), ctypes.POINTER(_I32)]),
    "oprag_index_data": (_P, [_P]),
    "oprag_index_get_rows": (_I32, [_P, _I64, _I64, _P]),
    "oprag_index_reserve": (_I32, [_P, _I32, _I32]),
    "oprag_upsert": (_I32, [_P, _P, _P, _I64, _I32, _I32, _P]),
    "oprag_search": (_I32, [_P, _P, _I32, _I32, _P, _P, _P]),
    "oprag_search_host": (_I32, [_P, _P, _I32, _I32, _P, _P, _P]),
    "oprag_search_noalloc": (_I32, [_P, _P, _I32, _I32, _P, _P, _P]),
    "oprag_index_set_sparse": (_I32, [_P, _P, _P, _I32, _F, _F]),
    "oprag_hybrid_search": (_I32, [_P, _P, _I32, _P, _P, _F, _I32, _P, _P, _P]),
    "oprag_index_check": (_I32, [_P]),
    "oprag_index_set_option": (_I32, [_P, _I32, _I32]),
    "oprag_hybrid_search_dense_first": (_I32, [_P, _P, _I32, _P, _P, _F, _I32, _I32, _P, _P, _P]),
    "oprag_embed_pool": (_I32, [_P, _I32, _I32, _I32, _I32, _P, _P, _I32, _P]),
    "oprag_append": (_I32, [_P, _P, _I64, _I32, _I32, _P, _P]),
    "oprag_index_update_sparse": (_I32, [_P, _P, _I64, _P, _P]),
    "oprag_search_two": (_I32, [_P, _P, _P, _I32, _I32, _P, _P, _P, _P]),
    "oprag_index_last_path": (_I32, [_P]),
    "oprag_index_last_launch": (_I32, [_P, ctypes.POINTER(_I32), ctypes.POINTER(_I32),
                                       ctypes.POINTER(_I32)]),
    "oprag_index_last_tiles_per_cta": (_I32, [_P, ctypes.POINTER(_I32)]),
    "oprag_plan_search": (_I32, [ctypes.c_int64, _I32, _I32, _I32, _I32, _I32, _I32, _I32,
                                 ctypes.POINTER(ctypes.c_int64)]),
    "oprag_index_last_timing": (_I32, [_P, ctypes.POINTER(_F), ctypes.POINTER(_F),
                                       ctypes.POINTER(_F), ctypes.POINTER(_F)]),
    "oprag_index_buffer_bytes": (_I32, [_P, ctypes.POINTER(_I64), ctypes.POINTER(_I64),
                                        ctypes.POINTER(_I64)]),
    "oprag_index_last_phases": (_I32, [_P, ctypes.POINTER(_I64), _I32, ctypes.POINTER(_I32)]),
    "oprag_last_error": (ctypes.c_char_p, []),
}

_lock = threading.Lock()
_lib = None


class OpragError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"oprag error {code} ({ERRORS.get(code, '?')}): {message}")
        self.code = code


def library_path() -> str:
    """The in-tree library, or the file named by $OPRAG_LIBRARY."""
    return os.environ.get("OPRAG_LIBRARY") or _build.LIB_PATH


def load(path: str | None = None) -> ctypes.CDLL:
    """Loads liboprag.so (built by paper_2608_08340_gb300.build.build())."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or library_path()
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build the CUDA library first "
                               "(python -m paper_2608_08340_gb300.build)")
        lib = ctypes.CDLL(p)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        if path is None:
            _lib = lib
        return lib


def check(rc: int) -> None:
    if rc != 0:
        msg = load().oprag_last_error()
        raise OpragError(rc, msg.decode() if msg else "")
