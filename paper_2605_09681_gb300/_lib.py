"""ctypes declarations of the C ABI in include/fk.h.  Loading fails loudly when the
compiled library is missing: there is no fallback implementation."""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfk.so")

FK_OK, FK_ERR_CONFIG, FK_ERR_ARG, FK_ERR_STATE, FK_ERR_FULL = 0, 1, 2, 3, 4
FK_ERR_RANGE, FK_ERR_TIMEOUT, FK_ERR_CUDA, FK_ERR_NOMEM = 5, 6, 7, 8
STATUS_NAMES = {0: "FK_OK", 1: "FK_ERR_CONFIG", 2: "FK_ERR_ARG", 3: "FK_ERR_STATE",
                4: "FK_ERR_FULL", 5: "FK_ERR_RANGE", 6: "FK_ERR_TIMEOUT", 7: "FK_ERR_CUDA",
                8: "FK_ERR_NOMEM"}
FK_SCOPE_PER_FRAME, FK_SCOPE_POOLED = 0, 1
FK_SCORE_PER_HEAD, FK_SCORE_LAYER0_POOLED = 0, 1
FK_SELECT = {"similarity": 0, "all": 1, "uniform": 2, "random": 3}
FK_ATTN = {"bf16": 0, "fp8_qk": 1, "fp8": 2}
KERNEL_KINDS = {"append": 0, "score": 1, "select": 2, "compact": 3, "attend": 4}

EXPORTS = [
    "fk_validate_config", "fk_create", "fk_destroy", "fk_append_frames", "fk_append_chunk",
    "fk_set_current", "fk_compress", "fk_attend", "fk_cache_bytes", "fk_reserved_bytes",
    "fk_key_count", "fk_get_kept", "fk_get_scores", "fk_sync_status", "fk_profile_enable",
    "fk_profile_read", "fk_profile_reset", "fk_launch_count", "fk_status_str", "fk_abi_version",
    "fk_segment_scores_noalloc", "fk_head_profile", "fk_classify_heads", "fk_set_host_overlap",
    "fk_wait_selftest", "fk_wait_outputs", "fk_quantize_e4m3", "fk_stream_read",
]


class FkConfig(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("tokens_per_frame", ctypes.c_int32), ("frames_per_chunk", ctypes.c_int32),
        ("n_sink_frames", ctypes.c_int32), ("window_frames", ctypes.c_int32),
        ("n_segments", ctypes.c_int32), ("keep_budget_permille", ctypes.c_int32),
        ("select_scope", ctypes.c_int32), ("score_source", ctypes.c_int32),
        ("incremental", ctypes.c_int32), ("max_history_frames", ctypes.c_int32),
        ("device", ctypes.c_int32), ("head_is_static", ctypes.POINTER(ctypes.c_uint8)),
        ("selection", ctypes.c_int32), ("select_seed", ctypes.c_uint32),
        ("static_drop_anchor", ctypes.c_int32), ("attn_precision", ctypes.c_int32),
    ]


class FkError(RuntimeError):
    def __init__(self, status: int, call: str):
        self.status = status
        self.name = STATUS_NAMES.get(status, str(status))
        super().__init__("%s failed: %s" % (call, self.name))


_lib = None


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libfk.so (built by paper_2605_09681_gb300.build); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise ImportError("libfk.so not built (%s); run paper_2605_09681_gb300.build.build()" % path)
    lib = ctypes.CDLL(path)
    vp, i32, cp = ctypes.c_void_p, ctypes.c_int, ctypes.c_char_p
    st = ctypes.c_int
    sig = {
        "fk_validate_config": (st, [ctypes.POINTER(FkConfig)]),
        "fk_create": (st, [ctypes.POINTER(FkConfig), ctypes.POINTER(vp)]),
        "fk_destroy": (None, [vp]),
        "fk_append_frames": (st, [vp, i32, vp, vp, i32, vp]),
        "fk_append_chunk": (st, [vp, i32, vp, vp, vp]),
        "fk_set_current": (st, [vp, i32, vp, vp, vp]),
        "fk_compress": (st, [vp, vp]),
        "fk_attend": (st, [vp, i32, vp, vp, vp]),
        "fk_cache_bytes": (ctypes.c_size_t, [vp]),
        "fk_reserved_bytes": (ctypes.c_size_t, [vp]),
        "fk_key_count": (st, [vp, i32, i32, ctypes.POINTER(i32)]),
        "fk_get_kept": (st, [vp, i32, i32, ctypes.POINTER(ctypes.c_int32), i32, ctypes.POINTER(i32), vp]),
        "fk_get_scores": (st, [vp, i32, i32, ctypes.POINTER(ctypes.c_float), i32,
                               ctypes.POINTER(i32), ctypes.POINTER(i32), vp]),
        "fk_sync_status": (st, [vp, vp]),
        "fk_profile_enable": (st, [vp, i32]),
        "fk_profile_read": (st, [vp, i32, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64)]),
        "fk_profile_reset": (st, [vp]),
        "fk_launch_count": (ctypes.c_int64, [vp]),
        "fk_set_host_overlap": (st, [vp, i32]),
        "fk_wait_selftest": (st, [vp, i32, vp]),
        "fk_wait_outputs": (st, [vp, vp]),
        "fk_status_str": (cp, [i32]),
        "fk_abi_version": (i32, []),
        "fk_segment_scores_noalloc": (st, [vp, i32, i32, i32, i32, vp, vp, vp]),
        "fk_head_profile": (st, [vp, vp, i32, i32, i32, i32, i32, i32, i32, vp, vp, vp]),
        "fk_classify_heads": (st, [ctypes.POINTER(ctypes.c_double), i32, i32,
                                   ctypes.POINTER(ctypes.c_uint8)]),
        "fk_quantize_e4m3": (st, [vp, ctypes.c_int64, i32, i32, vp, vp, vp]),
        "fk_stream_read": (st, [vp, ctypes.c_size_t, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib
