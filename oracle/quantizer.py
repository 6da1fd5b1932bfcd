"""Affine per-token group quantiser and integer packing (App. C.4).

The paper's quantiser, for bit width b and m = 2^b - 1, on one group of 64
coordinates with extrema x_min, x_max:

    s = max(x_max - x_min, 1e-8) / m
    z = clip(round(-x_min / s), 0, m)
    q = clip(round(x / s + z), 0, m)
    x_hat = s (q - z)

with round-half-to-even and no special case for constant groups. Native
execution dequantises with the *stored* scale.

The paper gives the real-number formula only. This library stores the scale
and the zero point as fp16, so the oracle fixes how the stored scale is
staged (the readings are listed in the design notes):

* d   = RN_f32(x_max - x_min)                     (inputs are bf16, so the
                                                    difference is exact before
                                                    this single rounding)
* s32 = RN_f32(max(d, RN_f32(1e-8)) / m)          (IEEE single division)
* s   = RN_f16(s32); s = 2^-24 if that is 0, 65504 if it overflows
* z and q are computed from the stored s, in fp64, with round-half-to-even,
  adding z before rounding.

Everything else is fp64.
"""
from __future__ import annotations

import numpy as np

GROUP = 64
_FLOOR_F32 = np.float32(1e-8)
_F16_MIN_SUB = 2.0 ** -24
_F16_MAX = 65504.0


def levels(bits: int) -> int:
    """m = 2^b - 1, the largest code (App. C.4)."""
    if bits not in (2, 4):
        raise ValueError("bit width must be 2 or 4")
    return (1 << bits) - 1


def stored_scale(xmin: np.ndarray, xmax: np.ndarray, bits: int) -> np.ndarray:
    """Stored fp16 scale s for groups with extrema (xmin, xmax), as float64."""
    m = levels(bits)
    d = (np.asarray(xmax, np.float64) - np.asarray(xmin, np.float64)).astype(np.float32)
    s32 = np.maximum(d, _FLOOR_F32) / np.float32(m)
    with np.errstate(over="ignore"):
        s16 = s32.astype(np.float16).astype(np.float64)
    s16 = np.where(s16 == 0.0, _F16_MIN_SUB, s16)
    s16 = np.where(np.isinf(s16), _F16_MAX, s16)
    return s16


def quantize_groups(x: np.ndarray, bits: int):
    """Quantise groups along the last axis (length 64).

    Returns (q, s, z): integer codes with x's shape (int64), and the stored
    scale and zero point with the leading shape (float64 holding fp16 values,
    int64).
    """
    x = np.asarray(x, dtype=np.float64)
    if x.shape[-1] != GROUP:
        raise ValueError("last axis must hold one 64-coordinate group")
    m = levels(bits)
    xmin = x.min(axis=-1)
    xmax = x.max(axis=-1)
    s = stored_scale(xmin, xmax, bits)
    z = np.clip(np.rint(-xmin / s), 0, m)
    q = np.clip(np.rint(x / s[..., None] + z[..., None]), 0, m)
    return q.astype(np.int64), s, z.astype(np.int64)


def dequantize(q: np.ndarray, s: np.ndarray, z: np.ndarray) -> np.ndarray:
    """x_hat = s (q - z), exact in fp64; s and z broadcast over the last axis."""
    return np.asarray(s, np.float64)[..., None] * (np.asarray(q, np.float64) - np.asarray(z, np.float64)[..., None])


def dequantize_fp16(q: np.ndarray, s: np.ndarray, z: np.ndarray) -> np.ndarray:
    """RN_f16(s (q - z)): the dequantised value rounded once to fp16."""
    return dequantize(q, s, z).astype(np.float16)


def pack(q: np.ndarray, bits: int) -> np.ndarray:
    """Pack codes along the last axis, low bits first within each byte.

    INT4: byte j = q[2j] | q[2j+1] << 4.
    INT2: byte j = q[4j] | q[4j+1] << 2 | q[4j+2] << 4 | q[4j+3] << 6.
    """
    q = np.asarray(q, dtype=np.int64)
    per = 8 // bits
    if q.shape[-1] % per:
        raise ValueError("code count must fill whole bytes")
    r = q.reshape(q.shape[:-1] + (q.shape[-1] // per, per))
    out = np.zeros(r.shape[:-1], dtype=np.int64)
    for k in range(per):
        out |= r[..., k] << (bits * k)
    return out.astype(np.uint8)


def unpack(b: np.ndarray, bits: int) -> np.ndarray:
    """Inverse of ``pack``: bytes along the last axis to codes (int64)."""
    b = np.asarray(b, dtype=np.int64)
    per = 8 // bits
    mask = (1 << bits) - 1
    parts = [(b >> (bits * k)) & mask for k in range(per)]
    return np.stack(parts, axis=-1).reshape(b.shape[:-1] + (b.shape[-1] * per,))
