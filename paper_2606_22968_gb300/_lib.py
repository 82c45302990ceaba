"""ctypes loader for libmocap.so (the C ABI declared in include/mocap.h)."""

from __future__ import annotations

import ctypes
import os
import threading

from . import _build

_LOCK = threading.Lock()
_LIB = None

c_i32, c_i64, c_f32, c_sz, c_vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t, ctypes.c_void_p


class VarlenItem(ctypes.Structure):
    _fields_ = [("q_row", c_i64), ("kv_row", c_i64), ("prefix", c_i64), ("len", c_i64)]


class AppendItem(ctypes.Structure):
    _fields_ = [("k_src", c_vp), ("v_src", c_vp), ("dst_row", c_i64), ("rows", c_i64)]


class CopyItem(ctypes.Structure):
    _fields_ = [("dst", c_vp), ("src", c_vp), ("bytes", c_i64)]


SIGNATURES = {
    "mocap_lbcp_partition": (c_i32, [c_i64, c_i32, c_i32, c_i32, ctypes.POINTER(c_i64)]),
    "mocap_lbcp_partition_dp": (c_i32, [c_i64, c_i32, c_i32, c_i32, c_i32, c_i64,
                                        ctypes.POINTER(c_i64)]),
    "mocap_lbcp_partition_dp_latency": (c_i32, [c_i64, c_i32, c_i32, c_i32, c_i32, c_i32, c_i32,
                                                c_i32, ctypes.POINTER(c_i64)]),
    "mocap_lbcp_gemm_weight": (c_i32, [ctypes.c_double, ctypes.c_double, c_i32,
                                       ctypes.POINTER(c_i64)]),
    "mocap_kv_append": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_i32, c_i32, c_vp]),
    "mocap_kv_append_overlap": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_i32, c_i32,
                                        c_vp]),
    "mocap_qkv_rope_append": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_i32,
                                      c_i32, c_i32, c_i32, c_f32, c_vp]),
    "mocap_chunk_attn": (c_i32, [c_vp, c_vp, c_vp, c_i64, c_i64, c_i32, c_i32, c_i32, c_f32,
                                 c_vp, c_vp, c_vp, c_sz, c_vp]),
    "mocap_chunk_attn_workspace_size": (c_sz, [c_i64, c_i64, c_i32, c_i32, c_i32]),
    "mocap_chunk_attn_noalloc": (c_i32, [c_vp, c_vp, c_vp, c_i64, c_i64, c_i32, c_i32, c_i32, c_f32,
                                         c_vp, c_vp, c_vp]),
    "mocap_chunk_attn_varlen": (c_i32, [c_vp, c_vp, c_vp, ctypes.POINTER(VarlenItem), c_i32,
                                        c_i64, c_i64, c_i32, c_i32, c_i32, c_f32, c_vp, c_vp,
                                        c_vp, c_sz, c_vp]),
    "mocap_copy_from_host": (c_i32, [ctypes.POINTER(CopyItem), c_i32, c_i32, c_vp]),
    "mocap_copy_to_host": (c_i32, [ctypes.POINTER(CopyItem), c_i32, c_i32, c_vp]),
    "mocap_chunk_attn_varlen_dev_workspace_size": (c_sz, [c_i32, c_i64, c_i32, c_i32, c_i32]),
    "mocap_chunk_attn_varlen_dev": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_i32, c_i64, c_i64, c_i64,
                                            c_i32, c_i32, c_i32, c_f32, c_vp, c_vp, c_vp, c_sz,
                                            c_vp]),
    "mocap_chunk_attn_append": (c_i32, [c_vp, c_vp, c_vp, c_i64, c_i64, c_i32, c_i32, c_i32, c_f32,
                                        c_vp, c_vp, c_vp, c_sz, ctypes.POINTER(AppendItem), c_i32,
                                        c_i64, c_vp]),
    "mocap_chunk_attn_varlen_append": (c_i32, [c_vp, c_vp, c_vp, ctypes.POINTER(VarlenItem), c_i32,
                                               c_i64, c_i64, c_i32, c_i32, c_i32, c_f32, c_vp,
                                               c_vp, c_vp, c_sz, ctypes.POINTER(AppendItem),
                                               c_i32, c_vp]),
    "mocap_last_row_attn_workspace_size": (c_sz, [ctypes.POINTER(c_i64), c_i32, c_i32, c_i32,
                                                   c_i32]),
    "mocap_last_row_attn": (c_i32, [c_vp, c_vp, c_vp, ctypes.POINTER(c_i64), ctypes.POINTER(c_i64),
                                    c_i32, c_i64, c_i32, c_i32, c_i32, c_f32, c_vp, c_vp, c_vp,
                                    c_sz, c_vp]),
    "mocap_last_device_status": (c_i32, [c_vp]),
    "mocap_selftest_bounded_wait": (c_i32, [ctypes.c_uint32, c_vp]),
    "mocap_status_string": (ctypes.c_char_p, [c_i32]),
}


def load(path: str | None = None):
    """Build (if stale) and load libmocap.so; raises if it cannot be built."""
    global _LIB
    with _LOCK:
        if _LIB is not None and path is None:
            return _LIB
        lib_path = path or _build.build()
        if not os.path.exists(lib_path):
            raise RuntimeError(f"libmocap.so not found at {lib_path}")
        lib = ctypes.CDLL(lib_path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        if path is None:
            _LIB = lib
        return lib
