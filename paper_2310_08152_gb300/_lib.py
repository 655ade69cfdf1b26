"""ctypes declarations of include/kvc.h.  Loading fails loudly if libkvc.so is missing."""
from __future__ import annotations

import ctypes
import os

from . import build as _build

c_int, c_int32, c_int64, c_size_t, c_float, c_void_p, c_char_p = (ctypes.c_int, ctypes.c_int32, ctypes.c_int64,
                                                                   ctypes.c_size_t, ctypes.c_float, ctypes.c_void_p,
                                                                   ctypes.c_char_p)
P = c_void_p


class KvcConfig(ctypes.Structure):
    _fields_ = [
        ("M", c_int),
        ("H", c_int),
        ("d_head", c_int),
        ("b", c_int),
        ("dtype", c_int),
        ("rotary_dim", c_int),
        ("rope_base", c_float),
        ("policy", c_int),
        ("seq_capacity", P),
        ("k_base", P),
        ("v_base", P),
        ("pos_base", P),
        ("orig_base", P),
        ("workspace", P),
        ("workspace_bytes", c_size_t),
        ("local_ratio", c_float),
    ]


# (name, restype, argtypes) for every function declared in include/kvc.h
SIGNATURES = [
    ("kvc_status_string", c_char_p, [c_int]),
    ("kvc_last_error", c_char_p, []),
    ("kvc_book_create", c_int, [c_int, c_int, P, P]),
    ("kvc_book_create_local", c_int, [c_int, c_float, P, P]),
    ("kvc_book_destroy", None, [P]),
    ("kvc_book_next_positions", c_int, [P, P, P, P]),
    ("kvc_book_append", c_int, [P, P, P, P]),
    ("kvc_book_append_free_closed", c_int, [P, P, P, P]),
    ("kvc_book_compress", c_int, [P, P, P, P, c_int]),
    ("kvc_book_pending_spans", c_int, [P, c_int, P, P, c_int64, P]),
    ("kvc_book_lengths", c_int, [P, P, P]),
    ("kvc_book_prefill_keys", c_int, [P, c_int, c_int64, P, c_int64, P]),
    ("kvc_book_layout", c_int, [P, c_int, c_int64, P, P, P, P, P, P, P]),
    ("kvc_required_bytes", c_int, [P, P, P, P, P]),
    ("kvc_create", c_int, [P, P]),
    ("kvc_destroy", None, [P]),
    ("kvc_get_book", P, [P]),
    ("kvc_append", c_int, [P, c_int, P, P, P, P, P, P]),
    ("kvc_append_free_closed", c_int, [P, c_int, P, P, P, P, P, P]),
    ("kvc_compress_spans", c_int, [P, P, P, P, c_int, P]),
    ("kvc_decode_attention", c_int, [P, c_int, P, c_float, P, P]),
    ("kvc_decode_attention_static_scratch", c_int, [P, c_int, P, c_float, P, P]),
    ("kvc_decode_attention_layers", c_int, [P, c_int, c_int, P, c_int64, c_float, P, c_int64, P]),
    ("kvc_prefill_attention", c_int, [P, c_int, P, P, c_float, P, P]),
    ("kvc_masked_reference_layout", c_int, [P, c_int, c_int64, P, P, P, P, P, P, P, P]),
    ("kvc_device_status", c_int, [P, P, P]),
    ("kvc_launch_count", c_int64, [P]),
    ("kvc_check_bounded_wait", c_int, [P, ctypes.c_uint64, P]),
    ("kvc_last_decode_plan", c_int, [P, P]),
    ("kvc_set_compaction_timing", c_int, [P, c_int]),
    ("kvc_last_compaction_ms", c_int, [P, P, P]),
]

_lib = None


def so_path() -> str:
    return _build.SO


def load(build_if_missing: bool = True):
    """The loaded libkvc.so.  Builds it in-tree first if it is missing or stale (nvcc required)."""
    global _lib
    if _lib is None:
        path = _build.build() if build_if_missing else _build.SO
        if not os.path.exists(path):
            raise OSError(f"libkvc.so not found at {path}; run __graft_entry__.build()")
        lib = ctypes.CDLL(path)
        for name, res, args in SIGNATURES:
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib
