"""ctypes binding of libmlkv_gb300.so (the C ABI of include/mlkv_gpu.h).

Argument marshalling only: every step of the store runs in the CUDA library.
PyTorch supplies device memory and the current stream.  There is no fallback:
if the library is missing or does not load, loading raises.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmlkv_gb300.so")

OK = 0
ERR_INVALID = 1
ERR_UNSUPPORTED = 2
ERR_CUDA = 3
ERR_NOMEM = 4
ERR_FULL = 5
ERR_PROBE_LIMIT = 6
ERR_NOT_FOUND = 7
ERR_TIMEOUT = 8
SEQ_SEGMENT_MAX = 32
PROBE_LIMIT = 1024
IDENTITY_HASH = 2
MAX_STALENESS = 64
STALENESS_ASYNC = 2**63 - 1  # staleness_bound of the asynchronous mode (INT64_MAX)

K_GET_GATHER = 1
K_PROBE = 2
K_SORT_SCATTER = 3
K_REDUCE_SHORT = 4
K_REDUCE_LONG = 5
K_SEGMENTS = 6
K_LONG_COMBINE = 7
K_TIER_FETCH = 8
K_PUT_SCATTER = 9
K_REDUCE_SINGLE = 10
K_REDUCE_SMALL = 11

EXPORTED = [
    "mlkv_open", "mlkv_close", "mlkv_get", "mlkv_put", "mlkv_insert", "mlkv_apply_grad",
    "mlkv_lookahead", "mlkv_find", "mlkv_export", "mlkv_dedup", "mlkv_get_host",
    "mlkv_apply_grad_host", "mlkv_sync", "mlkv_clear_status", "mlkv_size", "mlkv_launch_count",
    "mlkv_time_kernel", "mlkv_kernel_time", "mlkv_last_unique", "mlkv_last_error",
    "mlkv_status_string", "mlkv_dedup_keys_static", "mlkv_tier_stats", "mlkv_import", "mlkv_dump_keys",
    "mlkv_debug_fail",
]
FAULT_ALLOC = 1
FAULT_COPY = 2
FAULT_WAIT = 3
STATIC_MAX_KEYS = 65536


class Config(ctypes.Structure):
    _fields_ = [
        ("dim", ctypes.c_int32),
        ("insert_on_miss", ctypes.c_int32),
        ("capacity", ctypes.c_int64),
        ("max_batch", ctypes.c_int64),
        ("lr", ctypes.c_float),
        ("eps", ctypes.c_float),
        ("state_init", ctypes.c_float),
        ("init_lo", ctypes.c_float),
        ("init_hi", ctypes.c_float),
        ("seed", ctypes.c_uint64),
        ("staleness_bound", ctypes.c_int64),
        ("hbm_cache_rows", ctypes.c_int64),
        ("flags", ctypes.c_uint32),
        ("reserved", ctypes.c_uint32),
    ]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Loads the CUDA library; raises if it was not built (run __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"CUDA library {path} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.mlkv_open.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(vp)]
    lib.mlkv_close.argtypes = [vp]
    lib.mlkv_get.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_put.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_insert.argtypes = [vp, vp, i64, vp]
    lib.mlkv_apply_grad.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_lookahead.argtypes = [vp, vp, i64, vp]
    lib.mlkv_find.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_export.argtypes = [vp, vp, i64, vp, vp, vp]
    lib.mlkv_dedup.argtypes = [vp, vp, i64, vp, vp, vp, vp]
    lib.mlkv_dedup_keys_static.argtypes = [vp, i64, vp, vp, vp, vp]
    lib.mlkv_get_host.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_apply_grad_host.argtypes = [vp, vp, i64, vp, vp]
    lib.mlkv_sync.argtypes = [vp]
    lib.mlkv_clear_status.argtypes = [vp]
    lib.mlkv_size.argtypes = [vp]
    lib.mlkv_size.restype = i64
    lib.mlkv_launch_count.argtypes = [vp]
    lib.mlkv_launch_count.restype = i64
    lib.mlkv_time_kernel.argtypes = [vp, i32]
    lib.mlkv_kernel_time.argtypes = [vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64)]
    lib.mlkv_tier_stats.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(i64), ctypes.POINTER(i64)]
    lib.mlkv_import.argtypes = [vp, vp, i64, vp, vp, vp]
    lib.mlkv_dump_keys.argtypes = [vp, vp, i64, vp]
    lib.mlkv_debug_fail.argtypes = [i32, i64]
    lib.mlkv_last_unique.argtypes = [vp]
    lib.mlkv_last_unique.restype = i64
    lib.mlkv_last_error.argtypes = [vp]
    lib.mlkv_last_error.restype = ctypes.c_char_p
    lib.mlkv_status_string.argtypes = [i32]
    lib.mlkv_status_string.restype = ctypes.c_char_p
    for name in ("mlkv_open", "mlkv_close", "mlkv_get", "mlkv_put", "mlkv_insert", "mlkv_apply_grad",
                 "mlkv_lookahead", "mlkv_find", "mlkv_export", "mlkv_dedup", "mlkv_get_host",
                 "mlkv_apply_grad_host", "mlkv_sync", "mlkv_clear_status", "mlkv_time_kernel",
                 "mlkv_kernel_time", "mlkv_dedup_keys_static", "mlkv_tier_stats", "mlkv_import",
                 "mlkv_dump_keys", "mlkv_debug_fail"):
        getattr(lib, name).restype = i32
    _lib = lib
    return lib
