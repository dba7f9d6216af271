"""Loader of libdamp.so (ctypes) with the C signatures of include/damp.h.

There is no fallback: if the library is missing or cannot be loaded, every
entry point raises DampLibraryError.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libdamp.so")


class DampLibraryError(RuntimeError):
    """libdamp.so is not built or cannot be loaded."""


class DampLayout(ctypes.Structure):
    _fields_ = [("num_heads", ctypes.c_int32), ("num_qk_heads", ctypes.c_int32), ("d_k", ctypes.c_int32),
                ("d_v", ctypes.c_int32), ("k_hi", ctypes.c_int32), ("lo_format", ctypes.c_int32),
                ("model_heads", ctypes.c_int32), ("head_map", ctypes.c_void_p)]


_P = ctypes.c_void_p
_L = ctypes.POINTER(DampLayout)
_i32, _i64 = ctypes.c_int32, ctypes.c_int64
_status = ctypes.c_int

_STEP = [_L, _P, _i64, _P, _i32, _P, _P, _P, _P, _P, _P, _P, _i32, _P]
_FP32_STEP = [_L, _P, _i64, _P, _i32, _P, _P, _P, _P, _P, _P, _i32, _P]
_GROUP_STEP = [_L, _i32, _P, _P, _P, _P, _i32, _P, _P, _P, _P, _P, _P, _i32, _P]

SIGNATURES = {
    "damp_validate_layout": (_status, [_L]),
    "damp_record_bytes": (ctypes.c_size_t, [_L]),
    "damp_slot_bytes": (ctypes.c_size_t, [_L]),
    "damp_bits_per_value": (ctypes.c_double, [_L]),
    "damp_gdn_decode_step": (_status, _STEP),
    "damp_kda_decode_step": (_status, _STEP),
    "damp_gdn_decode_step_groups": (_status, _GROUP_STEP),
    "damp_kda_decode_step_groups": (_status, _GROUP_STEP),
    "damp_test_kda_wait_timeout": (_status, _STEP),
    "damp_u8_gdn_decode_step": (_status, _STEP),
    "damp_u8_kda_decode_step": (_status, _STEP),
    "damp_fp32_gdn_decode_step": (_status, _FP32_STEP),
    "damp_fp32_kda_decode_step": (_status, _FP32_STEP),
    "damp_gdn_prefill_chunk": (_status, [_L, _P, _i64, _P, _i32, _i32, _P, _P, _P, _P, _P, _P, _P, _P, _i32, _P]),
    "damp_kda_prefill_chunk": (_status, [_L, _P, _i64, _P, _i32, _i32, _P, _P, _P, _P, _P, _P, _P, _P, _i32, _P]),
    "damp_calib_error_energy": (_status, [_L, _P, _i32, _P, _P]),
    "damp_calib_log_decay": (_status, [_L, _P, _i32, _i32, _P, _P]),
    "damp_calib_select": (_status, [_L, _P, _i64, _P, _i64, ctypes.c_float, _P, _P, _P]),
    "damp_calib_accumulate": (_status, [_L, _P, _i32, _i32, _P, _P, _P, _P, _P, _i32, _i32, _i32, _P, _P, _P]),
    "damp_quantize_state": (_status, [_L, _P, _P, _P, _i64, _P, _i32, _P]),
    "damp_dequantize_state": (_status, [_L, _P, _i64, _P, _i32, _P, _P, _P]),
    "damp_pack_tiers": (_status, [_L, _P, _P, _P, _P, _i64, _P, _i32, _P]),
    "damp_unpack_tiers": (_status, [_L, _P, _i64, _P, _i32, _P, _P, _P, _P]),
    "damp_device_status": (_status, [ctypes.POINTER(ctypes.c_uint32)]),
    "damp_status_string": (ctypes.c_char_p, [_status]),
    "damp_version": (_i32, []),
}

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (built beforehand by paper_2608_27513_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise DampLibraryError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2608_27513_gb300.build` "
                "(libdamp has no CPU fallback)")
        try:
            handle = ctypes.CDLL(LIB_PATH)
        except OSError as e:
            raise DampLibraryError(f"cannot load {LIB_PATH}: {e}") from e
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(handle, name)
            fn.restype = res
            fn.argtypes = args
        _lib = handle
    return _lib
