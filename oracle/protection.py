"""Sink/recent BF16 protection of the packed cache (App. C.5, "BF16 protection
and cache lifecycle"), in fp64. Test infrastructure: used by tests/ only.

For L cached tokens with zero-based positions the protected set is (Eq. in
App. C.5)

    P_L = {0, ..., min(4, L) - 1}  U  {max(0, L - 128), ..., L - 1},

the union counting shared positions once. Attention uses the pre-quantisation
BF16 content and RoPE-key values for positions in P_L and the values
reconstructed from the packed cache for every other position; a packed copy
exists for every token, and all tokens share one softmax normalisation.

Protection buffer of this library (per request, 132 rows x 576 bf16 = the
paper's 152,064 bytes): a row holds a token's 512 latent values then its 64
RoPE-key values. Rows 0..3 hold the sink positions 0..3; row 4 + (p mod 128)
holds recent position p. The writer stores position p of a request whose
length after the write is L into row p when p < 4, and into row 4 + (p mod 128)
when p >= L - 128 (positions older than the recent window are not written,
so one bulk write cannot put two positions into one row).
"""
from __future__ import annotations

import numpy as np

from .attention import attend, quantized_cache

SINK = 4
RECENT = 128
ROWS = SINK + RECENT
ROW_VALUES = 576


def protected_positions(L: int) -> np.ndarray:
    """Sorted positions of P_L."""
    L = int(L)
    sink = set(range(0, min(SINK, L)))
    recent = set(range(max(0, L - RECENT), L))
    return np.array(sorted(sink | recent), dtype=np.int64)


def row_of(p: int, L: int) -> int:
    """Buffer row attention reads for protected position p of a length-L request."""
    if p < SINK:
        return p
    if p >= L - RECENT:
        return SINK + p % RECENT
    raise ValueError("position is not protected")


def write_protection(prot: np.ndarray, latent, k_pe, seq_ids, positions, final_lens) -> None:
    """The writer rule: prot [S, 132, 576] (any dtype holding bf16 values),
    token i of request seq_ids[i] at positions[i], final_lens[seq] = the
    request's length after this write."""
    latent = np.asarray(latent)
    k_pe = np.asarray(k_pe)
    for i, (s, p) in enumerate(zip(np.asarray(seq_ids), np.asarray(positions))):
        row = np.concatenate([latent[i], k_pe[i]])
        L = int(final_lens[s])
        if p < SINK:
            prot[s, p] = row
        if p >= L - RECENT:
            prot[s, SINK + p % RECENT] = row


def protected_cache(latent, k_pe, c_bits: int):
    """Values one request's decode attends over (L = number of rows of latent):
    the original values for positions in P_L, the dequantised packed copy
    otherwise. Returns (C [L, 512], K [L, 64]) in fp64."""
    latent = np.asarray(latent, np.float64)
    k_pe = np.asarray(k_pe, np.float64)
    L = latent.shape[0]
    C, K = quantized_cache(latent, k_pe, c_bits)
    C = np.array(C, np.float64)
    K = np.array(K, np.float64)
    P = protected_positions(L)
    C[P] = latent[P]
    K[P] = k_pe[P]
    return C, K


def attend_protected(q_lat, q_pe, latent, k_pe, c_bits: int, tau: float):
    """Decode attention of one request under sink4/local128 protection:
    (out [H, 512], lse [H]) in fp64."""
    C, K = protected_cache(latent, k_pe, c_bits)
    return attend(q_lat, q_pe, C, K, tau)


def attend_from_buffer(q_lat, q_pe, pool_C, pool_K, prot_row, L: int, tau: float):
    """The same attention, reading protected positions from a protection buffer
    row array prot_row [132, 576] and the others from the dequantised pool
    (pool_C [L, 512], pool_K [L, 64]): the kernel's data path restated."""
    C = np.array(pool_C, np.float64)
    K = np.array(pool_K, np.float64)
    for p in protected_positions(L):
        r = np.asarray(prot_row[row_of(int(p), L)], np.float64)
        C[p] = r[:512]
        K[p] = r[512:]
    return attend(q_lat, q_pe, C, K, tau)
