"""ctypes binding of libdms.so: the C ABI of include/dms.h, same names, same arguments.

Argument marshalling only; every step of the path runs in the library's CUDA
kernels.  Loading fails loudly (DmsLibraryError) when the library is missing:
there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libdms.so")

DMS_OK = 0
DMS_ERR_INVALID_ARGUMENT = 1
DMS_ERR_OUT_OF_MEMORY = 2
DMS_ERR_CAPACITY = 3
DMS_ERR_CUDA = 4
DMS_ERR_TIMEOUT = 5
DMS_ERR_STATE = 6
DMS_EVICT_DELAYED = 0
DMS_EVICT_IMMEDIATE = 1
DMS_PREFILL_TCGEN05 = 0
DMS_PREFILL_MMA_SYNC = 1
DMS_DECODE_TILED = 0
DMS_DECODE_SIMPLE = 1
DMS_DECODE_SPLIT = 2
DMS_DECODE_CLUSTER = 3
DMS_KV_BF16 = 0
DMS_KV_FP8_E4M3 = 1

# Every symbol the header declares (checked by the CPU test suite).
EXPORTS = (
    "dms_cache_create", "dms_cache_destroy", "dms_cache_reset", "dms_append_and_evict",
    "dms_decode_attention", "dms_cache_stats", "dms_cache_export_positions",
    "dms_cache_layer_length", "dms_status_string", "dms_decode_attention_paged_noalloc",
    "dms_append_and_decode", "dms_selftest_bounded_wait", "dms_append_and_evict_borrowed",
    "dms_decode_attention_borrowed", "dms_append_and_decode_borrowed",
    "dms_prefill_workspace_bytes", "dms_prefill_attention", "dms_prefill_attention_borrowed",
    "dms_prefill_device_error", "dms_prefill_attention_ex", "dms_append_shared_prefix",
    "dms_cache_export_kv", "dms_decode_noalloc_device_error", "dms_selftest_noalloc_timeout",
    "dms_decode_plan", "dms_selftest_stale_flag",
)


class DmsLibraryError(RuntimeError):
    """libdms.so could not be loaded (not built, or built for another host)."""


class dms_options(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("page_tokens", ctypes.c_int32),
                ("pool_tokens", ctypes.c_int64), ("decode_kernel", ctypes.c_int32),
                ("ctas_per_sm", ctypes.c_int32), ("min_pages_per_cta", ctypes.c_int32),
                ("eviction_policy", ctypes.c_int32), ("kv_format", ctypes.c_int32),
                ("reserved", ctypes.c_int32 * 3)]


class dms_stats(ctypes.Structure):
    _fields_ = [("total_retained", ctypes.c_int64), ("total_appended", ctypes.c_int64),
                ("total_evicted", ctypes.c_int64), ("pages_in_use", ctypes.c_int64),
                ("pool_pages", ctypes.c_int64), ("peak_pages", ctypes.c_int64),
                ("max_retained", ctypes.c_int32), ("min_retained", ctypes.c_int32),
                ("device_error", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libdms.so and declare the prototypes (once)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise DmsLibraryError(
            f"{path} is missing: build it first (python -c 'import __graft_entry__ as g; g.build()')")
    try:
        lib = ctypes.CDLL(path)
    except OSError as e:
        raise DmsLibraryError(f"cannot load {path}: {e}") from e
    vp, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
    st = ctypes.c_int
    proto = {
        "dms_cache_create": (st, [i32, i32, i32, i32, i64, ctypes.POINTER(dms_options),
                                  ctypes.POINTER(vp)]),
        "dms_cache_destroy": (st, [vp]),
        "dms_cache_reset": (st, [vp, vp]),
        "dms_append_and_evict": (st, [vp, i32, vp, vp, vp, i32, vp]),
        "dms_decode_attention": (st, [vp, i32, vp, vp, i32, f32, vp]),
        "dms_append_and_decode": (st, [vp, i32, vp, vp, vp, vp, vp, i32, f32, vp]),
        "dms_selftest_bounded_wait": (st, [i32, i64, vp]),
        "dms_append_and_evict_borrowed": (st, [vp, i32, vp, vp, vp, i32, i32, vp]),
        "dms_decode_attention_borrowed": (st, [vp, i32, vp, vp, i32, f32, vp]),
        "dms_append_and_decode_borrowed": (st, [vp, i32, vp, vp, vp, vp, i32, f32, vp]),
        "dms_prefill_workspace_bytes": (st, [i32, i32, i32, ctypes.POINTER(ctypes.c_size_t)]),
        "dms_prefill_attention": (st, [vp, vp, vp, vp, i32, i32, i32, i32, i32, f32, vp,
                                       ctypes.c_size_t, vp, vp]),
        "dms_prefill_attention_borrowed": (st, [vp, vp, vp, i32, i32, i32, i32, i32, f32, vp,
                                                ctypes.c_size_t, vp, vp]),
        "dms_prefill_device_error": (st, [vp, vp, ctypes.POINTER(st)]),
        "dms_append_shared_prefix": (st, [vp, i32, vp, vp, vp, i32, vp]),
        "dms_prefill_attention_ex": (st, [vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, f32,
                                          vp, ctypes.c_size_t, vp, vp]),
        "dms_cache_stats": (st, [vp, ctypes.POINTER(dms_stats), vp, vp]),
        "dms_cache_export_positions": (st, [vp, i32, vp, vp]),
        "dms_cache_export_kv": (st, [vp, i32, vp, vp, vp, vp]),
        "dms_cache_layer_length": (st, [vp, i32, ctypes.POINTER(i64)]),
        "dms_decode_plan": (st, [vp, i32, i32, ctypes.POINTER(i32), ctypes.POINTER(i32),
                                 ctypes.POINTER(i32)]),
        "dms_selftest_stale_flag": (st, [vp, i32, i64]),
        "dms_status_string": (ctypes.c_char_p, [st]),
        "dms_decode_attention_paged_noalloc": (st, [vp, vp, vp, i32, i32, i32, vp, vp, i32, f32,
                                                    vp]),
        "dms_decode_noalloc_device_error": (st, [vp, ctypes.POINTER(st)]),
        "dms_selftest_noalloc_timeout": (st, [i64, vp]),
    }
    for name, (res, args) in proto.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def status_string(code: int) -> str:
    return load().dms_status_string(int(code)).decode()
