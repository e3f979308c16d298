"""ctypes view of ``include/unicache.h`` and loading of ``lib/libunicache.so``.

Argument marshalling only. Loading fails loudly if the library was not
built: there is no fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "lib", "libunicache.so")

UC_OK, UC_ERR_ARG, UC_ERR_SHAPE, UC_ERR_BUDGET, UC_ERR_RANGE, UC_ERR_OOM, UC_ERR_CUDA, UC_ERR_TIMEOUT = range(8)
STATUS_NAMES = ["UC_OK", "UC_ERR_ARG", "UC_ERR_SHAPE", "UC_ERR_BUDGET", "UC_ERR_RANGE",
                "UC_ERR_OOM", "UC_ERR_CUDA", "UC_ERR_TIMEOUT"]
KIND_FULL, KIND_EVICT, KIND_QUANT, KIND_EVICT_QUANT = range(4)
POLICY_PROTECTED, POLICY_EVICT, POLICY_QUANT = -1, 0, 1
HEAD_DIM = 128
GROUP = 32
MAX_BATCH = 64
MAX_SEGMENTS = 8
MAX_QTOKENS = 8


class UcSegment(C.Structure):
    _fields_ = [
        ("kind", C.c_int32), ("bits", C.c_int32), ("batch", C.c_int32), ("n_kv_heads", C.c_int32),
        ("head_dim", C.c_int32), ("n_src", C.c_int32), ("cap", C.c_int32), ("label", C.c_int32),
        ("n_kept_host", C.c_int32 * MAX_BATCH),
        ("n_kept", C.c_void_p), ("kept_idx", C.c_void_p), ("k", C.c_void_p), ("v", C.c_void_p),
        ("row_stride", C.c_int64), ("row_offset", C.c_int64), ("rows_total", C.c_int64),
        ("k_codes", C.c_void_p), ("k_params", C.c_void_p), ("v_codes", C.c_void_p),
        ("v_params", C.c_void_p), ("cache_key", C.c_uint64), ("cache", C.c_uint8 * 256),
    ]


class UcSegmentSizes(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in
                ("k", "v", "k_codes", "k_params", "v_codes", "v_params", "kept_idx", "n_kept")]


class UcSegmentTable(C.Structure):
    _fields_ = [
        ("n_types", C.c_int32),
        ("candidate", C.c_int32 * MAX_SEGMENTS), ("n_tokens", C.c_int32 * MAX_SEGMENTS),
        ("policy", C.c_int32 * MAX_SEGMENTS), ("concentration", C.c_double * MAX_SEGMENTS),
        ("mass", C.c_double * MAX_SEGMENTS), ("budget", C.c_double * MAX_SEGMENTS),
        ("keep", C.c_int32 * MAX_SEGMENTS), ("bits", C.c_int32 * MAX_SEGMENTS),
        ("kind", C.c_int32 * MAX_SEGMENTS),
    ]


class UcTypeConfig(C.Structure):
    _fields_ = [("kind", C.c_int32), ("bits", C.c_int32), ("full_view", C.c_int32), ("max_keep", C.c_int32)]


class UcAttendCall(C.Structure):
    _fields_ = [
        ("q", C.c_void_p), ("n_q_heads", C.c_int32), ("n_qtok", C.c_int32),
        ("segs", C.c_void_p), ("n_seg", C.c_int32),
        ("out", C.c_void_p), ("lse", C.c_void_p), ("mass", C.c_void_p),
    ]


class UcAttendPlanInfo(C.Structure):
    _fields_ = [
        ("items_per_bh", C.c_int32), ("n_heavy", C.c_int32), ("n_light", C.c_int32), ("grid", C.c_int32),
        ("merge_kernel", C.c_int32), ("n_chunks", C.c_int32 * MAX_SEGMENTS), ("light", C.c_int32 * MAX_SEGMENTS),
    ]


MAX_CALLS = 8

# uc_allocator: stream-ordered device memory hooks for library-owned segments
ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p)
FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p, C.c_void_p)


class UcAllocator(C.Structure):
    _fields_ = [("alloc", ALLOC_FN), ("free", FREE_FN), ("ctx", C.c_void_p)]


_P = C.c_void_p
_SIGS = {
    "uc_last_error": (C.c_char_p, []),
    "uc_version": (C.c_int32, []),
    "uc_launch_count": (C.c_uint64, []),
    "uc_set_dense_serial_pv": (C.c_int32, [C.c_int32]),
    "uc_set_wait_limit": (C.c_uint64, [C.c_uint64]),
    "uc_debug_withhold_tile": (None, [C.c_int32]),
    "uc_set_programmatic_launch": (C.c_int32, [C.c_int32]),
    "uc_workspace_status": (C.c_int, [_P, _P]),
    "uc_segment_sizes_of": (C.c_int, [C.POINTER(UcSegment), C.POINTER(UcSegmentSizes)]),
    "uc_concentration": (C.c_int, [_P, C.c_int64, C.c_double, C.POINTER(C.c_double)]),
    "uc_calibrate_policy": (C.c_int, [C.POINTER(UcSegmentTable), _P, C.c_int32, C.c_double, C.c_double]),
    "uc_allocate_budget": (C.c_int, [C.POINTER(UcSegmentTable), C.c_double, C.c_int32]),
    "uc_retention_schedule": (C.c_int, [C.c_double] * 5 + [C.POINTER(C.c_double)]),
    "uc_retention_step": (C.c_int, [C.POINTER(UcSegmentTable), C.c_int32, C.c_double, C.c_double, C.c_double,
                                    C.POINTER(C.c_double), C.POINTER(C.c_double)]),
    "uc_plan_batch": (C.c_int, [C.POINTER(UcSegmentTable), C.c_int32, C.c_int32, C.POINTER(C.c_int32),
                                C.POINTER(UcTypeConfig)]),
    "uc_keep_count": (C.c_int, [C.c_int32, C.c_double, C.POINTER(C.c_int32)]),
    "uc_score_accumulate": (C.c_int, [_P, _P, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                                      C.c_int64, _P, _P, C.c_size_t, _P]),
    "uc_score_workspace_size": (C.c_size_t, [C.c_int32] * 5),
    "uc_segment_mass": (C.c_int, [_P, C.c_int32, C.c_int32, C.c_int32, _P, _P, C.c_int32, C.c_int32,
                                  C.c_int32, C.c_float, C.c_int32, _P, _P]),
    "uc_compress_segment": (C.c_int, [_P, _P, C.c_int64, C.c_int64, _P, C.c_int64, C.c_int64, C.c_int32,
                                      C.POINTER(UcSegment), _P, C.c_size_t, _P]),
    "uc_compress_workspace_size": (C.c_size_t, [C.POINTER(UcSegment)]),
    "uc_compress_budget": (C.c_int, [_P, _P, C.c_int32, C.c_int32, C.c_int32, C.c_int64, C.c_int64, _P,
                                     C.c_int64, C.c_int64, C.c_int32, _P, C.c_int32, _P, _P,
                                     C.POINTER(C.POINTER(UcSegment))]),
    "uc_segment_free": (None, [_P]),
    "uc_recompress_segment": (C.c_int, [C.POINTER(UcSegment), _P, C.c_int64, C.c_int64, C.c_int32,
                                        C.POINTER(UcSegment), _P, C.c_size_t, _P]),
    "uc_recompress_workspace_size": (C.c_size_t, [C.POINTER(UcSegment), C.POINTER(UcSegment)]),
    "uc_accumulate_scores": (C.c_int, [_P, C.c_int32, C.c_int32, C.POINTER(UcSegment), _P, _P, C.c_int64,
                                       C.c_int64, _P, C.c_size_t, _P]),
    "uc_attention_mass": (C.c_int, [_P, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_float, C.c_int32,
                                    _P, _P]),
    "uc_attend": (C.c_int, [_P, C.c_int32, C.c_int32, _P, C.c_int32, _P, _P, _P, _P, C.c_size_t, _P]),
    "uc_attend_workspace_size": (C.c_size_t, [_P, C.c_int32, C.c_int32, C.c_int32]),
    "uc_attend_plan": (C.c_int, [_P, C.c_int32, C.c_int32, C.c_int32, C.c_int32, _P]),
    "uc_attend_batch": (C.c_int, [_P, C.c_int32, _P, C.c_size_t, _P]),
    "uc_attend_batch_workspace_size": (C.c_size_t, [_P, C.c_int32]),
    "uc_attend_static": (C.c_int, [_P, C.c_int32, C.c_int32, _P, C.c_int32, _P, _P, _P, _P]),
    "uc_append": (C.c_int, [C.POINTER(UcSegment), _P, _P, C.c_int32, _P, C.c_size_t, _P]),
    "uc_append_next": (C.c_int, [C.POINTER(UcSegment), _P, _P, C.c_int32, _P, C.c_size_t, _P]),
}

_lock = threading.Lock()
_lib = None


class UniCacheError(RuntimeError):
    def __init__(self, fn: str, code: int, msg: str):
        name = STATUS_NAMES[code] if 0 <= code < len(STATUS_NAMES) else str(code)
        super().__init__(f"{fn}: {name}: {msg}")
        self.code = code


def lib():
    """The loaded C library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        with _lock:
            if _lib is None:
                if not os.path.exists(LIB_PATH):
                    raise ImportError(
                        f"{LIB_PATH} is missing: build the CUDA library first "
                        "(python -m paper_2609_32831_gb300.build); there is no CPU fallback")
                h = C.CDLL(LIB_PATH)
                for name, (res, args) in _SIGS.items():
                    f = getattr(h, name)
                    f.restype = res
                    f.argtypes = args
                _lib = h
    return _lib


def check(fn: str, code: int) -> None:
    if code != UC_OK:
        raise UniCacheError(fn, code, lib().uc_last_error().decode())
