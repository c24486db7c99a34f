"""ctypes declarations of libparason.so (include/parason.h).

Loading never builds and never falls back: if the in-tree library is missing
the import raises, so a GPU run cannot silently use anything else.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libparason.so")

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EUNSUPPORTED, ENOSPACE, ERANGE = range(8)
MODES = {"bf16": 0, "fp32": 1, "fp8": 2}
(TABLE_ITEMS, TABLE_DFS_LEAVES, TABLE_MERGE_RANGES, TABLE_MERGE, TABLE_WIDE_QUEUE,
 TABLE_NARROW_QUEUE, TABLE_ITEM_ROWS, TABLE_STREAM_ROWS, TABLE_ITEM_KEY0,
 TABLE_SHARD_BRANCHES) = range(10)
SHARD_REQUESTS, SHARD_KV_HEADS = 0, 1
DEBUG_SKIP_FIRST_LOAD = 1
DEBUG_FAIL_UPDATE = 2
NO_ALLOC_SCRATCH_BYTES = 64 << 20   # PARASON_NO_ALLOC_SCRATCH_BYTES

# every function include/parason.h declares, with (restype, argtypes)
_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_sz = ctypes.c_size_t
_pp = ctypes.POINTER(ctypes.c_void_p)


class AttnConfig(ctypes.Structure):
    _fields_ = [("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("mode", ctypes.c_int32), ("sm_scale", ctypes.c_float)]


class PlanInfo(ctypes.Structure):
    _fields_ = [("num_items", ctypes.c_int32), ("num_leaves", ctypes.c_int32),
                ("num_merge_entries", ctypes.c_int32), ("chunk_pages", ctypes.c_int32),
                ("num_slots", ctypes.c_int64), ("unique_tokens", ctypes.c_int64),
                ("path_tokens", ctypes.c_int64), ("num_sms", ctypes.c_int32),
                ("on_device", ctypes.c_int32), ("num_ctas", ctypes.c_int32),
                ("num_wide_ctas", ctypes.c_int32), ("num_wide_items", ctypes.c_int32),
                ("num_narrow_items", ctypes.c_int32), ("num_stream_rows", ctypes.c_int64),
                ("tile_pairs", ctypes.c_int32)]


class TraceStats(ctypes.Structure):
    _fields_ = [("total_tokens", ctypes.c_int64), ("latency_tokens", ctypes.c_int64),
                ("subtask_tokens", ctypes.c_int64), ("trial_tokens", ctypes.c_int64),
                ("parallel_blocks", ctypes.c_int32), ("threads", ctypes.c_int32),
                ("max_depth", ctypes.c_int32), ("top_level_blocks", ctypes.c_int32),
                ("acceleration", ctypes.c_double), ("eta", ctypes.c_double)]


SIGNATURES = {
    "parason_attn_plan": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p, _p, _i32,
                                         _p, _i64, _p, _pp]),
    "parason_attn_plan_host": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p, _p,
                                              _i32, _p, _i64, _i32, _pp]),
    "parason_prefill_plan": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p, _p, _i32,
                                            _p, _i64, _p, _pp]),
    "parason_prefill_plan_host": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p, _p,
                                                 _i32, _p, _i64, _i32, _pp]),
    "parason_attn_plan_shard": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p, _p,
                                               _i32, _p, _i64, _i32, _i32, _i32, _p, _pp]),
    "parason_attn_plan_shard_host": (ctypes.c_int, [ctypes.POINTER(AttnConfig), _i32, _p, _p, _p,
                                                    _p, _i32, _p, _i64, _i32, _i32, _i32, _i32,
                                                    _pp]),
    "parason_plan_workspace_bytes": (_sz, [_p]),
    "parason_attn_decode": (ctypes.c_int, [_p, _p, _p, _p, _p, _p, _p, _p, _p, _sz, _p]),
    "parason_attn_decode_no_alloc": (ctypes.c_int, [_p, _p, _p, _p, _p, _p, _p, _p, _p]),
    "parason_plan_append": (ctypes.c_int, [_p, _p, _p]),
    "parason_plan_fork": (ctypes.c_int, [_p, _i32, _i32, _p, _p, _p, _p]),
    "parason_trace_analyze": (ctypes.c_int, [_p, _i64, ctypes.POINTER(TraceStats),
                                             ctypes.POINTER(ctypes.c_int64)]),
    "parason_trace_fork_tree": (ctypes.c_int, [_p, _i64, _i32, _i32, _p, _p, _p,
                                               ctypes.POINTER(ctypes.c_int32),
                                               ctypes.POINTER(ctypes.c_int32)]),
    "parason_lse_merge": (ctypes.c_int, [_p, _p, _p, _p, _p, _p, _i64, _i32, _i32, _p]),
    "parason_plan_check": (ctypes.c_int, [_p, _p]),
    "parason_plan_destroy": (None, [_p]),
    "parason_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "parason_plan_get_info": (ctypes.c_int, [_p, ctypes.POINTER(PlanInfo)]),
    "parason_plan_export": (ctypes.c_int, [_p, _i32, _p, _sz]),
    "parason_plan_set_debug": (ctypes.c_int, [_p, ctypes.c_uint32, _i64]),
    "parason_plan_enable_timing": (ctypes.c_int, [_p, _i32]),
    "parason_plan_read_timing": (ctypes.c_int, [_p, _p, _p, _i32, ctypes.POINTER(ctypes.c_int32)]),
    "parason_plan_launches_per_decode": (_i32, [_p]),
    "parason_version": (ctypes.c_char_p, []),
}

_lib = None


def load() -> ctypes.CDLL:
    """Load the in-tree libparason.so; raise if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"libparason.so not found at {LIB_PATH}; build it with "
                "`python -m paper_2608_24658_gb300.build` (nvcc, sm_103a)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class ParasonError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        name = load().parason_status_string(status).decode()
        super().__init__(f"{what}: {name} (status {status})" if what else name)


def check(status: int, what: str = "") -> None:
    if status != OK:
        raise ParasonError(status, what)
