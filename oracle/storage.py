"""Persistent cache storage per request and layer (App. C.5, Eq. physical_cache_storage).

For a request of L tokens with 64-token pages, the paper's packed C4R4 format
takes ceil(L/64) (20480 + 8) + 152064 bytes (packed pages, an 8-byte reverse
page map per page, and 132 x 576 BF16 protection rows), against
ceil(L/64) * 73728 bytes for a BF16 cache.

This library's format has no protection buffers or reverse map; a page is
``block_bytes`` (20736 B for INT4 content, 12544 B for INT2 content).
"""
from __future__ import annotations

PAGE = 64
PAPER_C4R4_PAGE = 20480
PAPER_REVERSE_MAP = 8
PAPER_PROTECTION = 132 * 576 * 2
BF16_PAGE = PAGE * 1152


def pages(L: int) -> int:
    return -(-int(L) // PAGE)


def paper_c4r4_bytes(L: int) -> int:
    return pages(L) * (PAPER_C4R4_PAGE + PAPER_REVERSE_MAP) + PAPER_PROTECTION


def bf16_bytes(L: int) -> int:
    return pages(L) * BF16_PAGE


def paper_ratio(L: int) -> float:
    return bf16_bytes(L) / paper_c4r4_bytes(L)


def packed_bytes(L: int, block_bytes: int) -> int:
    """This library's persistent bytes for L tokens: whole blocks only."""
    return pages(L) * block_bytes
