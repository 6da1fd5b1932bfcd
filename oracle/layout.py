"""This library's paged cache block layout, written and read byte by byte.

The paper stores packed copies of every token in 64-token pages written by
"slot-mapped page insertion" (App. C.5, cache update). The byte layout below is
this library's own (the paper's C4R4 page keeps BF16 content scales and FP32
RoPE scales, App. C.5 storage layout; here both are fp16 with an fp16 integer
zero point). A block holds 64 token slots; slot = position mod 64 and the block
is block_table[seq][position div 64].

Block of 64 tokens, content at ``c_bits`` in {4, 2}, RoPE key at 4 bits,
cb = 64 * c_bits / 8 bytes of content codes per token and group:

    offset 0                   content codes  [8 groups][64 slots][cb bytes]
    offset 8*64*cb             RoPE-key codes [64 slots][32 bytes]
    offset 8*64*cb + 2048      scale/zero     [9 groups][64 slots][fp16 s, fp16 z]
                                              (group 8 is the RoPE key)

    INT4 content: 16384 + 2048 + 2304 = 20736 bytes per block (324 B/token)
    INT2 content:  8192 + 2048 + 2304 = 12544 bytes per block (196 B/token)

Group g of the content covers channels [64 g, 64 g + 64). All multi-byte
values are little-endian.
"""
from __future__ import annotations

import numpy as np

from .quantizer import pack, quantize_groups, unpack

BLOCK_TOKENS = 64
D_C = 512
D_R = 64
N_GROUPS = 9  # 8 content groups + 1 RoPE-key group
PE_BITS = 4


def content_code_bytes(c_bits: int) -> int:
    """Bytes of packed content codes per token and 64-channel group."""
    return 64 * c_bits // 8


def offsets(c_bits: int) -> dict:
    cb = content_code_bytes(c_bits)
    pe_codes = 8 * BLOCK_TOKENS * cb
    sz = pe_codes + BLOCK_TOKENS * 32
    total = sz + N_GROUPS * BLOCK_TOKENS * 4
    return {"cb": cb, "pe_codes": pe_codes, "sz": sz, "block_bytes": total}


def block_bytes(c_bits: int) -> int:
    return offsets(c_bits)["block_bytes"]


def quantize_tokens(latent: np.ndarray, k_pe: np.ndarray, c_bits: int):
    """Quantise tokens: latent [n,512] and k_pe [n,64] (bf16 values as float64).

    Returns q [n,576] (content codes then RoPE codes), s [n,9], z [n,9].
    """
    latent = np.asarray(latent, np.float64)
    k_pe = np.asarray(k_pe, np.float64)
    n = latent.shape[0]
    qc, sc, zc = quantize_groups(latent.reshape(n, 8, 64), c_bits)
    qp, sp, zp = quantize_groups(k_pe.reshape(n, 1, 64), PE_BITS)
    q = np.concatenate([qc.reshape(n, 512), qp.reshape(n, 64)], axis=1)
    s = np.concatenate([sc, sp], axis=1)
    z = np.concatenate([zc, zp], axis=1)
    return q, s, z


def write_tokens(pool: np.ndarray, c_bits: int, latent, k_pe, seq_ids, positions, table) -> None:
    """Quantise tokens and insert them into ``pool`` (uint8 [num_blocks, block_bytes]).

    Token i goes to block table[seq_ids[i], positions[i] // 64], slot
    positions[i] % 64.
    """
    o = offsets(c_bits)
    cb = o["cb"]
    seq_ids = np.asarray(seq_ids, np.int64)
    positions = np.asarray(positions, np.int64)
    table = np.asarray(table, np.int64)
    n = seq_ids.shape[0]
    if n == 0:
        return
    q, s, z = quantize_tokens(latent, k_pe, c_bits)
    blk = table[seq_ids, positions // BLOCK_TOKENS]
    if (blk < 0).any() or (blk >= pool.shape[0]).any():
        raise IndexError("block id out of range")
    slot = positions % BLOCK_TOKENS
    codes_c = pack(q[:, :512].reshape(n, 8, 64), c_bits)       # [n, 8, cb]
    codes_p = pack(q[:, 512:], PE_BITS)                          # [n, 32]
    for g in range(8):
        cols = g * BLOCK_TOKENS * cb + slot[:, None] * cb + np.arange(cb)[None, :]
        pool[blk[:, None], cols] = codes_c[:, g, :]
    cols = o["pe_codes"] + slot[:, None] * 32 + np.arange(32)[None, :]
    pool[blk[:, None], cols] = codes_p
    sz = np.stack([s.astype(np.float16), z.astype(np.float16)], axis=-1)  # [n, 9, 2]
    sz_bytes = sz.view(np.uint8).reshape(n, 9, 4)
    for g in range(N_GROUPS):
        cols = o["sz"] + (g * BLOCK_TOKENS + slot[:, None]) * 4 + np.arange(4)[None, :]
        pool[blk[:, None], cols] = sz_bytes[:, g, :]


def read_sequence(pool: np.ndarray, c_bits: int, table_row, length: int):
    """Read tokens 0..length-1 of one sequence back as (q [L,576], s [L,9], z [L,9])."""
    o = offsets(c_bits)
    cb = o["cb"]
    table_row = np.asarray(table_row, np.int64)
    pos = np.arange(length, dtype=np.int64)
    blk = table_row[pos // BLOCK_TOKENS]
    if (blk < 0).any() or (blk >= pool.shape[0]).any():
        raise IndexError("block id out of range")
    slot = pos % BLOCK_TOKENS
    qc = np.empty((length, 8, 64), np.int64)
    for g in range(8):
        cols = g * BLOCK_TOKENS * cb + slot[:, None] * cb + np.arange(cb)[None, :]
        qc[:, g, :] = unpack(pool[blk[:, None], cols], c_bits)
    cols = o["pe_codes"] + slot[:, None] * 32 + np.arange(32)[None, :]
    qp = unpack(pool[blk[:, None], cols], PE_BITS)
    sz = np.empty((length, N_GROUPS, 4), np.uint8)
    for g in range(N_GROUPS):
        cols = o["sz"] + (g * BLOCK_TOKENS + slot[:, None]) * 4 + np.arange(4)[None, :]
        sz[:, g, :] = pool[blk[:, None], cols]
    sz16 = np.ascontiguousarray(sz).view(np.float16).reshape(length, N_GROUPS, 2).astype(np.float64)
    q = np.concatenate([qc.reshape(length, 512), qp], axis=1)
    return q, sz16[..., 0], sz16[..., 1].astype(np.int64)


def bf16_block_bytes() -> int:
    """The unquantised comparison cache: 64 tokens x 576 bf16 = 73728 bytes."""
    return BLOCK_TOKENS * (D_C + D_R) * 2
