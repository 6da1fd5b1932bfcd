"""The paper's own C4R4 page format, in fp64. App. C.4: the native kernels keep
each content group's scale as bf16 and the RoPE group's scale as fp32, and
dequantise with those stored values. App. C.5, storage layout: 20,480 bytes per
64-token page, 320 bytes per token. Test infrastructure: used by tests/ only.

Quantiser (App. C.4: s = max(x_max - x_min, 1e-8) / m, z = clip(rne(-x_min / s), 0, m),
q = clip(rne(x / s + z), 0, m), x_hat = s (q - z), m = 15 for 4-bit groups), with the
staging this format fixes (the paper gives the real-number formula only):

* content groups: d = RN_f32(x_max - x_min); s = RN_bf16(RN_f32(max(d, RN_f32(1e-8)) / 15));
  z and q in exact arithmetic. x (bf16) and s (bf16) both have 8 significant bits,
  so an fp32 quotient x / s is either exactly a half-integer or far (>> 2^-24
  relative) from one: exact and fp32 evaluation agree.
* the RoPE group: d = RN_f32(x_max - x_min); s = RN_f32(max(d, RN_f32(1e-8)) / 15);
  z and q evaluated in fp32 as written: z = clip(rne(RN_f32(-x_min / s)), 0, 15),
  q = clip(rne(RN_f32(RN_f32(x / s) + z)), 0, 15). (With a 24-bit scale an exact
  quotient could sit within fp32 rounding of a half-integer, so the fp32 steps are
  part of the definition.)

Values the decode's fp16 tiles hold: RN_f16(s (q - z)) for content (the product of
a 4-bit integer and an 8-bit-mantissa scale is exact in fp32) and
RN_f16(RN_f32(s (q - z))) for the RoPE key.

Page (64 token slots, little-endian):

    0       content codes   [8 groups][64 slots][32 bytes]   16384
    16384   RoPE codes      [64 slots][32 bytes]              2048
    18432   content scales  [8 groups][64 slots] bf16         1024
    19456   RoPE scales     [64 slots] fp32                    256
    19712   zero points     [9 groups][64 slots] uint8         576   (group 8: RoPE)
    20288   padding (zero)                                     192
            total                                             20480

Codes are packed low nibble first (as in this library's own format).
"""
from __future__ import annotations

import numpy as np

from .quantizer import pack, unpack

PAGE_TOKENS = 64
PAGE_BYTES = 20480
OFF_PE_CODES = 16384
OFF_C_SCALE = 18432
OFF_PE_SCALE = 19456
OFF_ZERO = 19712
_FLOOR_F32 = np.float32(1e-8)
M = 15


def rn_bf16(x) -> np.ndarray:
    """Round float32 values to bf16 (round half to even on the 16 dropped bits);
    returns float32 holding bf16 values."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def content_scale(xmin, xmax) -> np.ndarray:
    d = (np.asarray(xmax, np.float64) - np.asarray(xmin, np.float64)).astype(np.float32)
    return rn_bf16(np.maximum(d, _FLOOR_F32) / np.float32(M)).astype(np.float64)


def rope_scale(xmin, xmax) -> np.ndarray:
    d = (np.asarray(xmax, np.float64) - np.asarray(xmin, np.float64)).astype(np.float32)
    return (np.maximum(d, _FLOOR_F32) / np.float32(M)).astype(np.float64)


def quantize_content(x: np.ndarray):
    """Groups along the last axis (64): (q int64, s float64 bf16 values, z int64)."""
    x = np.asarray(x, np.float64)
    s = content_scale(x.min(-1), x.max(-1))
    z = np.clip(np.rint(-x.min(-1) / s), 0, M)
    q = np.clip(np.rint(x / s[..., None] + z[..., None]), 0, M)
    return q.astype(np.int64), s, z.astype(np.int64)


def quantize_rope(x: np.ndarray):
    """The RoPE group in fp32 arithmetic: (q int64, s float64 fp32 values, z int64)."""
    x32 = np.asarray(x, np.float32)
    s32 = rope_scale(x32.min(-1), x32.max(-1)).astype(np.float32)
    z = np.clip(np.rint(np.float32(-1) * x32.min(-1) / s32), 0, M).astype(np.float32)
    t = (x32 / s32[..., None]).astype(np.float32)
    u = (t + z[..., None]).astype(np.float32)
    q = np.clip(np.rint(u), 0, M)
    return q.astype(np.int64), s32.astype(np.float64), z.astype(np.int64)


def quantize_tokens(latent, k_pe):
    """latent [n,512], k_pe [n,64] (bf16 values) -> q [n,576], s [n,9], z [n,9]."""
    latent = np.asarray(latent, np.float64)
    n = latent.shape[0]
    qc, sc, zc = quantize_content(latent.reshape(n, 8, 64))
    qp, sp, zp = quantize_rope(np.asarray(k_pe, np.float64).reshape(n, 1, 64))
    return (np.concatenate([qc.reshape(n, 512), qp.reshape(n, 64)], 1), np.concatenate([sc, sp], 1),
            np.concatenate([zc, zp], 1))


def dequantize_tokens(q, s, z):
    """x_hat = s (q - z) exactly: (C [n,512], K [n,64])."""
    n = q.shape[0]
    x = np.asarray(s, np.float64)[:, :, None] * (np.asarray(q, np.float64).reshape(n, 9, 64)
                                                  - np.asarray(z, np.float64)[:, :, None])
    x = x.reshape(n, 576)
    return x[:, :512], x[:, 512:]


def tile_values(q, s, z):
    """The fp16 values the decode's tiles hold (as float64): (C [n,512], K [n,64])."""
    n = q.shape[0]
    d = np.asarray(q, np.float64).reshape(n, 9, 64) - np.asarray(z, np.float64)[:, :, None]
    c = (np.asarray(s[:, :8], np.float64)[:, :, None] * d[:, :8]).astype(np.float16)
    k = (np.asarray(s[:, 8:], np.float32)[:, :, None] * d[:, 8:].astype(np.float32)).astype(np.float32)
    k = k.astype(np.float16)
    return c.reshape(n, 512).astype(np.float64), k.reshape(n, 64).astype(np.float64)


def write_tokens(pool: np.ndarray, latent, k_pe, seq_ids, positions, table) -> None:
    """Slot-mapped insertion into pool [num_pages, 20480] uint8."""
    q, s, z = quantize_tokens(latent, k_pe)
    for i, (b, p) in enumerate(zip(np.asarray(seq_ids), np.asarray(positions))):
        page = pool[int(table[int(b), int(p) // PAGE_TOKENS])]
        slot = int(p) % PAGE_TOKENS
        for g in range(8):
            page[(g * 64 + slot) * 32:(g * 64 + slot + 1) * 32] = pack(q[i, 64 * g:64 * g + 64], 4)
            hi = (np.array([s[i, g]], np.float32).view(np.uint32) >> 16).astype(np.uint16)  # bf16 bits
            page[OFF_C_SCALE + (g * 64 + slot) * 2:OFF_C_SCALE + (g * 64 + slot) * 2 + 2] = hi.view(np.uint8)
            page[OFF_ZERO + g * 64 + slot] = z[i, g]
        page[OFF_PE_CODES + slot * 32:OFF_PE_CODES + slot * 32 + 32] = pack(q[i, 512:], 4)
        page[OFF_PE_SCALE + slot * 4:OFF_PE_SCALE + slot * 4 + 4] = np.frombuffer(np.float32(s[i, 8]).tobytes(),
                                                                                   np.uint8)
        page[OFF_ZERO + 8 * 64 + slot] = z[i, 8]


def read_sequence(pool: np.ndarray, table_row, length: int):
    """Codes and metadata of tokens [0, length) of one sequence: q [L,576], s [L,9], z [L,9]."""
    q = np.zeros((length, 576), np.int64)
    s = np.zeros((length, 9), np.float64)
    z = np.zeros((length, 9), np.int64)
    for p in range(length):
        page = pool[int(table_row[p // PAGE_TOKENS])]
        slot = p % PAGE_TOKENS
        for g in range(8):
            q[p, 64 * g:64 * g + 64] = unpack(page[(g * 64 + slot) * 32:(g * 64 + slot + 1) * 32], 4)
            hi = page[OFF_C_SCALE + (g * 64 + slot) * 2:OFF_C_SCALE + (g * 64 + slot) * 2 + 2].view(np.uint16)[0]
            s[p, g] = np.array([np.uint32(hi) << 16], np.uint32).view(np.float32)[0]
            z[p, g] = page[OFF_ZERO + g * 64 + slot]
        q[p, 512:] = unpack(page[OFF_PE_CODES + slot * 32:OFF_PE_CODES + slot * 32 + 32], 4)
        s[p, 8] = page[OFF_PE_SCALE + slot * 4:OFF_PE_SCALE + slot * 4 + 4].view(np.float32)[0]
        z[p, 8] = page[OFF_ZERO + 8 * 64 + slot]
    return q, s, z
