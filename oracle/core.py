"""ctypes wrapper over the plain-C oracle (damp_oracle.c).  Test infrastructure only.

Array conventions (all dense, C order):
  perm  uint8  [n, d_k]           packed row i holds natural key channel perm[i]
  hi    uint16 [n, K, d_v]        binary16 bit patterns of the FP16 tier S_hi
  codes uint8  [n, d_k-K, d_v]    UINT8 codes Q_lo (int8 for the row-absmax format; E4M3
        bit patterns for FP8; [n, d_k-K, d_v/2] two UINT4 codes per byte, even value
        index in the low nibble, for the 4-bit formats)
  meta  uint16 [n, d_k-K, d_v/32, 2]  binary16 (s, z) per 32-group (M_lo);
        float32 [n, d_k-K] scales for the row-absmax format,
        float32 [n, d_k-K, d_v/32] scales for FP8
  S     float32 [n, d_k, d_v]     natural-order state
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import build as _build

FMT_U8_H32 = 0
FMT_U8 = 1
FMT_S8_ROW = 2
FMT_U4_H32 = 3
FMT_U4 = 4
FMT_E4M3 = 5
KINDS = {"gdn": 0, "kda": 1}

_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(_build.build())
        P = ctypes.c_void_p
        i64, i32, f32 = ctypes.c_int64, ctypes.c_int, ctypes.c_float
        sig = {
            "dor_f32_to_f16": (ctypes.c_uint16, [f32]),
            "dor_f16_to_f32": (f32, [ctypes.c_uint16]),
            "dor_f32_to_f16_array": (None, [P, P, i64]),
            "dor_f16_to_f32_array": (None, [P, P, i64]),
            "dor_hadamard32": (None, [P, P]),
            "dor_quant_group_u8": (None, [P, P, P]),
            "dor_dequant_group_u8": (None, [P, P, P]),
            "dor_quant_row_s8": (None, [P, i32, P, P]),
            "dor_quant_group_u4": (None, [P, P, P]),
            "dor_dequant_group_u4": (None, [P, P, P]),
            "dor_e4m3_to_f32": (f32, [ctypes.c_uint8]),
            "dor_f32_to_e4m3": (ctypes.c_uint8, [f32]),
            "dor_quant_group_e4m3": (None, [P, P, P]),
            "dor_dequant_group_e4m3": (None, [P, f32, P]),
            "dor_dequant_row_s8": (None, [P, i32, f32, P]),
            "dor_qdq_rows": (None, [i64, i32, i32, P, P]),
            "dor_delta_step": (None, [i32, i32, P, P, P, P, P, f32, P]),
            "dor_delta_step_heads": (None, [i64, i32, i32, i32, P, P, P, P, P, P, P]),
            "dor_mixed_step_heads": (i32, [i64, i32, i32, i32, i32, i32, P, P, P, P, P, P, P, P, P, P]),
            "dor_prefill_chunk_heads": (i32, [i64, i32, i32, i32, i32, i32, P, P, P, P, i32, P, P, P, P, P, P, P]),
            "dor_pack_heads": (i32, [i64, i32, i32, i32, i32, P, P, P, P, P]),
            "dor_unpack_heads": (i32, [i64, i32, i32, i32, i32, P, P, P, P, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(_lib, name)
            fn.restype = res
            fn.argtypes = args
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


# ----------------------------------------------------------------------------
# element-level pieces
# ----------------------------------------------------------------------------

def f32_to_f16(x) -> np.ndarray:
    x = _f32(x)
    h = np.empty(x.shape, np.uint16)
    lib().dor_f32_to_f16_array(_p(x), _p(h), x.size)
    return h


def f16_to_f32(h) -> np.ndarray:
    h = np.ascontiguousarray(h, dtype=np.uint16)
    x = np.empty(h.shape, np.float32)
    lib().dor_f16_to_f32_array(_p(h), _p(x), h.size)
    return x


def hadamard32(x) -> np.ndarray:
    """Normalized block-32 Hadamard transform of every length-32 vector on the last axis."""
    x = _f32(x)
    assert x.shape[-1] == 32
    flat = x.reshape(-1, 32)
    out = np.empty_like(flat)
    for i in range(flat.shape[0]):
        lib().dor_hadamard32(_p(flat[i]), _p(out[i]))
    return out.reshape(x.shape)


def quant_group_u8(x):
    """UINT8 affine quantizer of one 32-group: returns (codes uint8[32], sz uint16[2])."""
    x = _f32(x).reshape(32)
    q = np.empty(32, np.uint8)
    sz = np.empty(2, np.uint16)
    lib().dor_quant_group_u8(_p(x), _p(q), _p(sz))
    return q, sz


def dequant_group_u8(q, sz) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8).reshape(32)
    sz = np.ascontiguousarray(sz, dtype=np.uint16).reshape(2)
    x = np.empty(32, np.float32)
    lib().dor_dequant_group_u8(_p(q), _p(sz), _p(x))
    return x


def quant_group_u4(x):
    """UINT4 affine quantizer of one 32-group: returns (codes uint8[16] nibble pairs, sz uint16[2])."""
    x = _f32(x).reshape(32)
    q = np.empty(16, np.uint8)
    sz = np.empty(2, np.uint16)
    lib().dor_quant_group_u4(_p(x), _p(q), _p(sz))
    return q, sz


def dequant_group_u4(q, sz) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8).reshape(16)
    sz = np.ascontiguousarray(sz, dtype=np.uint16).reshape(2)
    x = np.empty(32, np.float32)
    lib().dor_dequant_group_u4(_p(q), _p(sz), _p(x))
    return x


def e4m3_to_f32(b: int) -> float:
    return float(lib().dor_e4m3_to_f32(int(b)))


def f32_to_e4m3(x: float) -> int:
    return int(lib().dor_f32_to_e4m3(float(x)))


def quant_group_e4m3(x):
    """FP8 E4M3 group quantizer: returns (codes uint8[32] E4M3 bits, s float)."""
    x = _f32(x).reshape(32)
    q = np.empty(32, np.uint8)
    s = np.empty(1, np.float32)
    lib().dor_quant_group_e4m3(_p(x), _p(q), _p(s))
    return q, float(s[0])


def dequant_group_e4m3(q, s: float) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8).reshape(32)
    x = np.empty(32, np.float32)
    lib().dor_dequant_group_e4m3(_p(q), float(s), _p(x))
    return x


def quant_row_s8(x):
    x = _f32(x).reshape(-1)
    q = np.empty(x.size, np.int8)
    s = np.empty(1, np.float32)
    lib().dor_quant_row_s8(_p(x), x.size, _p(q), _p(s))
    return q, float(s[0])


def qdq_rows(x, fmt: int) -> np.ndarray:
    """Q_lo (quantize then reconstruct) applied to every row of the last axis (d_v)."""
    x = _f32(x)
    dv = x.shape[-1]
    flat = x.reshape(-1, dv)
    out = np.empty_like(flat)
    lib().dor_qdq_rows(flat.shape[0], dv, fmt, _p(flat), _p(out))
    return out.reshape(x.shape)


# ----------------------------------------------------------------------------
# packed tiers of n heads
# ----------------------------------------------------------------------------

def tier_arrays(n: int, d_k: int, d_v: int, k_hi: int, fmt: int):
    """Empty (hi, codes, meta) arrays for n heads."""
    lo = d_k - k_hi
    hi = np.zeros((n, k_hi, d_v), np.uint16)
    if fmt == FMT_S8_ROW:
        codes = np.zeros((n, lo, d_v), np.int8)
        meta = np.zeros((n, lo), np.float32)
    elif fmt in (FMT_U4_H32, FMT_U4):
        codes = np.zeros((n, lo, d_v // 2), np.uint8)
        meta = np.zeros((n, lo, d_v // 32, 2), np.uint16)
    elif fmt == FMT_E4M3:
        codes = np.zeros((n, lo, d_v), np.uint8)
        meta = np.zeros((n, lo, d_v // 32), np.float32)
    else:
        codes = np.zeros((n, lo, d_v), np.uint8)
        meta = np.zeros((n, lo, d_v // 32, 2), np.uint16)
    return hi, codes, meta


def pack_heads(perm, S, k_hi: int, fmt: int):
    perm = np.ascontiguousarray(perm, dtype=np.uint8)
    S = _f32(S)
    n, d_k, d_v = S.shape
    hi, codes, meta = tier_arrays(n, d_k, d_v, k_hi, fmt)
    rc = lib().dor_pack_heads(n, d_k, d_v, k_hi, fmt, _p(perm), _p(S), _p(hi), _p(codes), _p(meta))
    if rc:
        raise ValueError("oracle pack: invalid permutation or sizes")
    return hi, codes, meta


def unpack_heads(perm, hi, codes, meta, k_hi: int, fmt: int, d_k: int, d_v: int) -> np.ndarray:
    perm = np.ascontiguousarray(perm, dtype=np.uint8)
    n = perm.shape[0]
    S = np.empty((n, d_k, d_v), np.float32)
    rc = lib().dor_unpack_heads(n, d_k, d_v, k_hi, fmt, _p(perm), _p(np.ascontiguousarray(hi)),
                                _p(np.ascontiguousarray(codes)), _p(np.ascontiguousarray(meta)), _p(S))
    if rc:
        raise ValueError("oracle unpack: invalid permutation or sizes")
    return S


# ----------------------------------------------------------------------------
# steps over n independent heads
# ----------------------------------------------------------------------------

def delta_step_heads(S, q, k, v, g, beta, kind: str) -> np.ndarray:
    """FP32 delta-rule step on natural-order states S [n, d_k, d_v] (updated in place); returns o."""
    assert S.dtype == np.float32 and S.flags["C_CONTIGUOUS"]
    n, d_k, d_v = S.shape
    q, k, v, g, beta = _f32(q), _f32(k), _f32(v), _f32(g), _f32(beta)
    o = np.empty((n, d_v), np.float32)
    lib().dor_delta_step_heads(n, d_k, d_v, KINDS[kind], _p(S), _p(q), _p(k), _p(v), _p(g), _p(beta), _p(o))
    return o


def mixed_step_heads(perm, hi, codes, meta, q, k, v, g, beta, k_hi: int, fmt: int, kind: str) -> np.ndarray:
    """Quantized recurrence step on packed tiers (updated in place); returns o [n, d_v]."""
    for a in (hi, codes, meta):
        assert a.flags["C_CONTIGUOUS"]
    perm = np.ascontiguousarray(perm, dtype=np.uint8)
    n, d_k = perm.shape
    d_v = np.shape(v)[-1]
    q, k, v, g, beta = _f32(q), _f32(k), _f32(v), _f32(g), _f32(beta)
    o = np.empty((n, d_v), np.float32)
    rc = lib().dor_mixed_step_heads(n, d_k, d_v, k_hi, fmt, KINDS[kind], _p(perm), _p(hi), _p(codes), _p(meta),
                                    _p(q), _p(k), _p(v), _p(g), _p(beta), _p(o))
    if rc:
        raise ValueError("oracle mixed step: invalid permutation or sizes")
    return o


def prefill_chunk_heads(perm, hi, codes, meta, q, k, v, g, beta, k_hi: int, fmt: int, kind: str,
                        lengths=None) -> np.ndarray:
    """One prefill chunk per head on packed tiers (updated in place; App. A.5 prefill path).

    q, k [n, T, d_k]; v [n, T, d_v]; g [n, T] (GDN) or [n, T, d_k] (KDA); beta [n, T];
    lengths [n] (default T) = tokens of each head's chunk.  Returns o [n, T, d_v]
    (rows past a head's length are zero)."""
    for a in (hi, codes, meta):
        assert a.flags["C_CONTIGUOUS"]
    perm = np.ascontiguousarray(perm, dtype=np.uint8)
    n, d_k = perm.shape
    q, k, v, g, beta = _f32(q), _f32(k), _f32(v), _f32(g), _f32(beta)
    T = q.shape[1]
    d_v = v.shape[-1]
    lens = np.full(n, T, np.int32) if lengths is None else np.ascontiguousarray(lengths, dtype=np.int32)
    o = np.zeros((n, T, d_v), np.float32)
    rc = lib().dor_prefill_chunk_heads(n, d_k, d_v, k_hi, fmt, KINDS[kind], _p(perm), _p(hi), _p(codes), _p(meta),
                                       T, _p(lens), _p(q), _p(k), _p(v), _p(g), _p(beta), _p(o))
    if rc:
        raise ValueError("oracle prefill: invalid permutation, sizes or lengths")
    return o


def bits_per_value(d_k: int, d_v: int, k_hi: int, fmt: int) -> float:
    """Storage bits per state value counted from the tier arrays' bytes."""
    hi, codes, meta = tier_arrays(1, d_k, d_v, k_hi, fmt)
    return 8.0 * (hi.nbytes + codes.nbytes + meta.nbytes) / (d_k * d_v)
