"""ctypes view of libt2istore.so (the C ABI declared in include/t2istore.h).

Loading fails loudly when the library has not been built: there is no other
implementation of any call behind this module.
"""
from __future__ import annotations

import ctypes as C
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libt2istore.so")

OK, ERR_INVALID, ERR_NOSPACE, ERR_NOT_FOUND, ERR_EVICTED, ERR_CUDA, ERR_NOT_CONTIGUOUS = 0, 1, 2, 3, 4, 5, 6
STATUS_NAMES = {0: "OK", 1: "INVALID", 2: "NOSPACE", 3: "NOT_FOUND", 4: "EVICTED", 5: "CUDA", 6: "NOT_CONTIGUOUS"}


class StoreConfig(C.Structure):
    _fields_ = [("pool_bytes", C.c_uint64), ("page_bytes", C.c_uint64), ("h2d_mode", C.c_uint32),
                ("check_pointers", C.c_uint32), ("alloc_policy", C.c_uint32), ("d2h_mode", C.c_uint32)]


class PutDesc(C.Structure):
    _fields_ = [("src", C.c_void_p), ("nbytes", C.c_uint64), ("src_is_host", C.c_uint32),
                ("dtype_tag", C.c_uint32), ("group", C.c_uint64), ("order", C.c_uint32),
                ("evictable", C.c_uint32), ("consumers", C.c_uint32), ("reserved", C.c_uint32)]


class GetDesc(C.Structure):
    _fields_ = [("id", C.c_uint64), ("dst", C.c_void_p), ("dst_bytes", C.c_uint64), ("cast", C.c_uint32),
                ("reserved", C.c_uint32)]


class Move(C.Structure):
    _fields_ = [("src_page", C.c_uint32), ("dst_page", C.c_uint32), ("valid_bytes", C.c_uint64)]


class Stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in (
        "total_pages", "limit_pages", "used_pages", "free_pages", "live_objects",
        "bytes_put", "bytes_got", "puts", "gets", "misses", "evictions",
        "pages_moved", "bytes_moved", "launches", "h2d_copies", "reclaimed", "views", "d2h_copies")]

    def as_dict(self) -> dict:
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class ObjectInfo(C.Structure):
    _fields_ = [("nbytes", C.c_uint64), ("group", C.c_uint64), ("dtype_tag", C.c_uint32), ("order", C.c_uint32),
                ("evictable", C.c_uint32), ("n_pages", C.c_uint32), ("consumers_left", C.c_uint32),
                ("reserved", C.c_uint32)]


class PagedObject(C.Structure):
    _fields_ = [("nbytes", C.c_uint64), ("pages", C.c_void_p), ("n_pages", C.c_uint32), ("dtype_tag", C.c_uint32)]


_P = C.c_void_p
_S = C.c_int32
_U32 = C.c_uint32
_U64 = C.c_uint64
_PU64 = C.POINTER(C.c_uint64)
_PU32 = C.POINTER(C.c_uint32)

# name -> (restype, argtypes), in the order of include/t2istore.h
PROTOTYPES = {
    "t2i_store_create": (_S, [_P, C.POINTER(StoreConfig), C.c_int, C.POINTER(_P)]),
    "t2i_store_destroy": (_S, [_P]),
    # array arguments of the per-request calls are plain addresses (ints,
    # numpy buffers' ctypes.data or typed pointers all pass): building a
    # typed pointer costs more than the call's other Python work
    "t2i_put_batch": (_S, [_P, _P, _U32, _P, _P]),
    "t2i_get_batch": (_S, [_P, _P, _U32, _P, _P]),
    "t2i_get_batch_after": (_S, [_P, _P, _U32, _P, _P, _P]),
    "t2i_view": (_S, [_P, _U64, _P, C.POINTER(_P), _PU64]),
    "t2i_pull": (_S, [_P, _P, _P, _U32, _U32, _P, _P, _P]),
    "t2i_pull_pages": (_S, [_P, _P, _U64, _P, _U32, _U32, _P, _P]),
    "t2i_free": (_S, [_P, _P, _U32]),
    "t2i_compact": (_S, [_P, _U64, _P, _PU64]),
    "t2i_inject_launch_failure": (_S, [_P, _U32]),
    "t2i_store_stats": (_S, [_P, C.POINTER(Stats)]),
    "t2i_store_ctl": (_P, [_P]),
    "t2i_last_error": (C.c_char_p, [_P]),
    "t2i_ctl_create": (_S, [_U64, _U64, _U32, C.POINTER(_P)]),
    "t2i_ctl_destroy": (_S, [_P]),
    "t2i_ctl_put": (_S, [_P, C.POINTER(PutDesc), _U32, _PU64]),
    "t2i_ctl_get": (_S, [_P, C.POINTER(GetDesc), _U32, C.POINTER(_S)]),
    "t2i_ctl_free": (_S, [_P, _PU64, _U32]),
    "t2i_ctl_compact": (_S, [_P, _U64, C.POINTER(Move), _U64, _PU64]),
    "t2i_ctl_object": (_S, [_P, _U64, C.POINTER(ObjectInfo), _PU32, _U64]),
    "t2i_ctl_free_pages": (_S, [_P, _PU32, _U64, _PU64]),
    "t2i_ctl_last_evictions": (_S, [_P, _PU64, _U64, _PU64]),
    "t2i_ctl_stats": (_S, [_P, C.POINTER(Stats)]),
    "t2i_ctl_last_error": (C.c_char_p, [_P]),
    "t2i_gather_noalloc": (_S, [_P, _U64, _U64, _PU32, _U32, _U64, _P, _U64, _U32, C.c_int, _P]),
    "t2i_e2e_latency": (_S, [_U32, _U32, C.c_double, C.c_double, C.POINTER(C.c_double)]),
    "t2i_prefix_layers": (_S, [_U32, C.c_double, C.c_double, _PU32]),
    "t2i_pipeline_latency": (_S, [C.POINTER(C.c_double), C.POINTER(C.c_double), _U32, _U32, C.POINTER(C.c_double)]),
    "t2i_prefix_layers_pipeline": (_S, [C.POINTER(C.c_double), C.POINTER(C.c_double), _U32, _PU32]),
    "t2i_put_layers": (_S, [_P, C.POINTER(PutDesc), _PU32, _U32, _U32, _PU64, _P, C.POINTER(_P)]),
}

_lib = None
_pycall = False  # not looked up yet


def load() -> C.CDLL:
    """The loaded library with prototypes set. Raises if it is not built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with `python -m paper_2607_26566_gb300.build` "
                              "(or __graft_entry__.build()); the store has no other implementation")
        lib = C.CDLL(LIB_PATH)
        for name, (res, args) in PROTOTYPES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def pycall():
    """The CPython entry points of csrc/pycall.c (put_batch, get_batch,
    get_batch_ids, free: the same C-ABI calls without ctypes' per-call
    argument conversion), or None where Python.h was missing at build time.
    Loads the library first."""
    global _pycall
    if _pycall is False:
        load()
        try:
            from . import _pycall as m
        except ImportError:
            m = None
        _pycall = m
    return _pycall
