"""ctypes declarations of the C ABI in include/tq.h (argument marshalling only)."""
from __future__ import annotations

import ctypes as C
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtq.so")

TQ_OK, TQ_EINVAL, TQ_ENOMEM, TQ_ECUDA, TQ_ETIMEOUT, TQ_EUNSUPPORTED = range(6)
STATUS_NAMES = {0: "TQ_OK", 1: "TQ_EINVAL", 2: "TQ_ENOMEM", 3: "TQ_ECUDA", 4: "TQ_ETIMEOUT",
                5: "TQ_EUNSUPPORTED"}
MARGINALS = {"beta": 0, "gauss": 1}
SCALE_MODES = {"norm": 0, "none": 1, "unbiased": 2}
PATHS = {"auto": 0, "lut": 1, "mma": 2, "lut_fixed": 3, "lut_fold": 4}

# name -> (restype, argtypes); every symbol include/tq.h declares
SIGNATURES = {
    "tq_last_error": (C.c_char_p, []),
    "tq_version": (C.c_int, []),
    "tq_codebook": (C.c_int, [C.c_int, C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_rotation": (C.c_int, [C.c_int, C.c_uint64, C.c_void_p]),
    "tq_encode": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p,
                            C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_filter_build": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.POINTER(C.c_void_p), C.c_void_p]),
    "tq_filter_append": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]),
    "tq_filter_destroy": (C.c_int, [C.c_void_p]),
    "tq_filter_info": (C.c_int, [C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_int),
                                 C.POINTER(C.c_int64)]),
    "tq_search_workspace": (C.c_int, [C.c_int64, C.c_int64, C.c_int, C.c_int, C.c_int, C.c_void_p,
                                      C.POINTER(C.c_size_t)]),
    "tq_search": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_int,
                            C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p,
                            C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "tq_search_ex": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_int,
                               C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p,
                               C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                               C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "tq_calibrate_workspace": (C.c_int, [C.c_int64, C.c_int, C.POINTER(C.c_size_t)]),
    "tq_calibrate": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p,
                               C.c_void_p, C.c_size_t, C.c_void_p]),
    "tq_encode_ex": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int,
                               C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_encode_plan_bytes": (C.c_int, [C.c_int, C.POINTER(C.c_size_t)]),
    "tq_encode_plan": (C.c_int, [C.c_void_p, C.c_int, C.c_void_p, C.c_size_t, C.c_void_p]),
    "tq_encode_planned": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int,
                                    C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_encode_check": (C.c_int, [C.c_void_p, C.c_void_p]),
    "tq_search_host_staging": (C.c_int, [C.c_int64, C.c_int, C.c_int, C.POINTER(C.c_size_t)]),
    "tq_search_host": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_int,
                                 C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p]),
    "tq_idmap_create": (C.c_int, [C.c_int64, C.POINTER(C.c_void_p)]),
    "tq_idmap_destroy": (C.c_int, [C.c_void_p]),
    "tq_idmap_add": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.POINTER(C.c_int64), C.c_void_p]),
    "tq_idmap_remove": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.POINTER(C.c_int64), C.c_void_p]),
    "tq_idmap_lookup": (C.c_int, [C.c_void_p, C.c_uint64, C.POINTER(C.c_int64)]),
    "tq_idmap_info": (C.c_int, [C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_int64), C.POINTER(C.c_int64)]),
    "tq_idmap_device": (C.c_int, [C.c_void_p, C.POINTER(C.c_void_p), C.POINTER(C.c_void_p)]),
    "tq_idmap_export": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_idmap_import": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]),
    "tq_search_static": (C.c_int, [C.c_void_p, C.c_int64, C.c_int, C.c_void_p, C.c_void_p, C.c_int,
                                   C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p,
                                   C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p]),
    "tq_merge_topk": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int64, C.c_int64, C.c_int64, C.c_int, C.c_void_p,
                                C.c_void_p, C.c_void_p]),
    "tq_search_check": (C.c_int, [C.c_void_p, C.c_void_p]),
    "tq_debug_fail_allocs": (C.c_int, [C.c_int]),
    "tq_debug_bounded_wait": (C.c_int, [C.c_longlong, C.c_void_p, C.c_void_p]),
    "tq_set_search_path": (C.c_int, [C.c_int]),
    "tq_profile_events": (C.c_int, [C.c_void_p, C.c_void_p]),
}

_lib = None


class TQError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def load() -> C.CDLL:
    """Loads libtq.so; raises if it has not been built (there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2607_16973_gb300.build`")
        lib = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def check(status: int) -> None:
    if status != TQ_OK:
        raise TQError(status, load().tq_last_error().decode(errors="replace"))
