"""Pins of the paper-format oracle (BF16 content scales, FP32 RoPE scales,
integer zero points, 20,480-byte pages): the page size and storage ratios
against the paper's printed figures, bf16 rounding against torch, a
hand-worked group with its exact bytes, the round-trip bound, brute-force
code optimality, the claim that exact and fp32 content quantisation agree,
and a write/read round trip."""
import os

import numpy as np
import pytest
import torch

from oracle import paper_format as F
from oracle import protection as Pr
from oracle import storage as St

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_storage.txt")


def _golden():
    d = {}
    for line in open(GOLDEN):
        line = line.split("#")[0].strip()
        if line:
            k, v = (t.strip() for t in line.split("="))
            d[k] = float(v)
    return d


def _bf16(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).float().numpy()


def test_page_size_is_the_papers():
    g = _golden()
    assert F.PAGE_BYTES == g["c4r4_page_bytes"]
    assert F.PAGE_BYTES // F.PAGE_TOKENS == g["c4r4_bytes_per_token"]
    # every region inside the page, no overlap: codes, scales, zeros, padding
    assert F.OFF_PE_CODES == 8 * 64 * 32 and F.OFF_C_SCALE == F.OFF_PE_CODES + 64 * 32
    assert F.OFF_PE_SCALE == F.OFF_C_SCALE + 8 * 64 * 2 and F.OFF_ZERO == F.OFF_PE_SCALE + 64 * 4
    assert F.OFF_ZERO + 9 * 64 <= F.PAGE_BYTES


@pytest.mark.parametrize("L,key", [(4096, "ratio_4k"), (131072, "ratio_128k")])
def test_storage_ratio_with_real_pages(L, key):
    # Eq. physical_cache_storage with this format's page, the 8-byte reverse map and
    # the protection buffer: reproduces the printed 3.22x / 3.59x.
    pages = -(-L // 64)
    c4r4 = pages * (F.PAGE_BYTES + 8) + Pr.ROWS * Pr.ROW_VALUES * 2
    assert round(St.bf16_bytes(L) / c4r4, 2) == _golden()[key]


def test_rn_bf16_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10.0 ** rng.integers(-8, 5, 100000),
                        np.array([1.0, 1.00390625, 1.01171875, 0.0, -0.0, 3.0e-39, 1e-8], np.float32)]).astype(np.float32)
    assert np.array_equal(F.rn_bf16(x), _bf16(x))


def test_hand_worked_group_and_bytes():
    # x_k = (k mod 16 - 4) / 4: d = 3.75, s = 0.25 exactly (bf16 and fp32), z = 4,
    # q = k mod 16, x_hat = x; content codes 0x10, 0x32, ..., 0xFE.
    x = ((np.arange(64) % 16) - 4) / 4.0
    lat = np.tile(x, 8)[None, :]
    kpe = x[None, :]
    q, s, z = F.quantize_tokens(lat, kpe)
    assert np.all(s == 0.25) and np.all(z == 4) and np.array_equal(q[0], np.tile(np.arange(64) % 16, 9))
    C, K = F.dequantize_tokens(q, s, z)
    assert np.array_equal(C[0], lat[0]) and np.array_equal(K[0], kpe[0])
    pool = np.zeros((1, F.PAGE_BYTES), np.uint8)
    F.write_tokens(pool, lat, kpe, [0], [5], np.zeros((1, 1), np.int64))
    page = pool[0]
    assert list(page[5 * 32:5 * 32 + 8]) == [0x10, 0x32, 0x54, 0x76, 0x98, 0xBA, 0xDC, 0xFE]
    assert page[F.OFF_C_SCALE + 5 * 2:F.OFF_C_SCALE + 5 * 2 + 2].view(np.uint16)[0] == 0x3E80   # bf16 0.25
    assert page[F.OFF_PE_SCALE + 5 * 4:F.OFF_PE_SCALE + 5 * 4 + 4].view(np.uint32)[0] == 0x3E800000  # fp32 0.25
    assert page[F.OFF_ZERO + 5] == 4 and page[F.OFF_ZERO + 8 * 64 + 5] == 4
    assert not page[F.OFF_ZERO + 9 * 64:].any()  # padding untouched


def _groups(rng, n):
    g = rng.standard_normal((n, 64)) * np.exp(0.5 * rng.standard_normal((n, 1)))
    return _bf16(g).astype(np.float64)


@pytest.mark.parametrize("path", ["content", "rope"])
def test_round_trip_bound_and_brute_force(path):
    rng = np.random.default_rng(1 if path == "content" else 2)
    x = _groups(rng, 400)
    q, s, z = (F.quantize_content if path == "content" else F.quantize_rope)(x)
    xh = s[:, None] * (q - z[:, None])
    interior = (q > 0) & (q < 15)
    assert np.all(np.abs(x - xh)[interior] <= s[:, None].repeat(64, 1)[interior] * (0.5 + 1e-6))
    # brute force: no other code gives a strictly closer reconstruction for interior
    # elements. The RoPE codes are decided in fp32 (two roundings of a quotient below
    # 32, each at most 2^-19 of s), so there a neighbour may win by up to 2^-17 s.
    cand = s[:, None, None] * (np.arange(16)[None, None, :] - z[:, None, None])
    best = np.abs(x[:, :, None] - cand).min(-1)
    slack = 1e-12 if path == "content" else 2.0 ** -17 * s[:, None].repeat(64, 1)[interior]
    assert np.all(np.abs(x - xh)[interior] <= best[interior] + slack)
    if path == "rope":
        # and exact-arithmetic codes differ only where the exact x / s + z lies
        # within 2^-18 of a half-integer
        qe = np.clip(np.rint(x / s[:, None] + z[:, None]), 0, 15)
        frac = np.abs((x / s[:, None] + z[:, None]) % 1.0 - 0.5)
        assert np.all(frac[qe != q] <= 2.0 ** -18)


def test_content_exact_and_fp32_agree():
    # x and s carry 8 significant bits, so evaluating rne(x / s + z) with an fp32
    # quotient gives the same codes as exact arithmetic.
    rng = np.random.default_rng(3)
    x = _groups(rng, 3000)
    q, s, z = F.quantize_content(x)
    x32, s32 = x.astype(np.float32), s.astype(np.float32)
    z32 = np.clip(np.rint((-x32.min(-1)) / s32), 0, 15)
    q32 = np.clip(np.rint((x32 / s32[:, None]).astype(np.float32) + z32[:, None].astype(np.float32)), 0, 15)
    assert np.array_equal(q, q32.astype(np.int64)) and np.array_equal(z, z32.astype(np.int64))


def test_write_read_round_trip():
    rng = np.random.default_rng(4)
    L = 150
    lat = _bf16(rng.standard_normal((L, 512)) * 3).astype(np.float64)
    kpe = _bf16(rng.standard_normal((L, 64))).astype(np.float64)
    table = np.array([[2, 0, 1]], np.int64)
    pool = np.zeros((3, F.PAGE_BYTES), np.uint8)
    order = rng.permutation(L)
    F.write_tokens(pool, lat[order], kpe[order], np.zeros(L, np.int64), order, table)
    q, s, z = F.read_sequence(pool, table[0], L)
    q2, s2, z2 = F.quantize_tokens(lat, kpe)
    assert np.array_equal(q, q2) and np.array_equal(s, s2) and np.array_equal(z, z2)
    # fp16 tile values: content is one rounding of the exact product
    C, _ = F.dequantize_tokens(q, s, z)
    Ct, _ = F.tile_values(q, s, z)
    assert np.array_equal(Ct, C.astype(np.float16).astype(np.float64))
