"""Pins of the oracle's block writer/reader against the documented byte layout."""
import numpy as np

from oracle import layout as Lo
from oracle import quantizer as Q


def test_block_sizes():
    # INT4: 8*64*32 + 64*32 + 9*64*4 = 16384 + 2048 + 2304; INT2: 8192 + 2048 + 2304.
    assert Lo.block_bytes(4) == 20736 and Lo.block_bytes(4) // 64 == 324
    assert Lo.block_bytes(2) == 12544 and Lo.block_bytes(2) // 64 == 196
    assert Lo.bf16_block_bytes() == 73728


def _token(k_offset=0.0):
    # content channel c has value ((c mod 16) - 4)/4 + k_offset*(c//64): every group has
    # s = 0.25, z = 4 - 4*k_offset... keep k_offset = 0 for exact hand values.
    c = np.arange(512)
    lat = ((c % 16) - 4) / 4.0
    r = np.arange(64)
    kpe = (r % 16) - 8.0          # x_min = -8, x_max = 7: s = 1, z = 8, q = r mod 16
    return lat[None, :], kpe[None, :]


def test_slot_mapped_insertion_bytes():
    # Sequence 1, position 69 -> logical block 1, slot 5 -> physical block table[1][1] = 2.
    table = np.array([[0, 3], [1, 2]], np.int32)
    for bits in (4, 2):
        pool = np.full((4, Lo.block_bytes(bits)), 0xAB, np.uint8)
        lat, kpe = _token()
        if bits == 2:
            lat = (np.arange(512) % 4 - 1.0)[None, :]   # s = 1, z = 1, q = c mod 4
        Lo.write_tokens(pool, bits, lat, kpe, [1], [69], table)
        cb = 64 * bits // 8
        blk = pool[2]
        # untouched blocks keep their poison
        assert np.all(pool[[0, 1, 3]] == 0xAB)
        code_byte = 0x10 if bits == 4 else 0xE4
        for g in range(8):
            off = g * 64 * cb + 5 * cb
            if bits == 4:
                assert list(blk[off:off + 8]) == [0x10, 0x32, 0x54, 0x76, 0x98, 0xBA, 0xDC, 0xFE]
            else:
                assert np.all(blk[off:off + cb] == code_byte)
            # neighbouring slots untouched
            assert np.all(blk[off - cb:off] == 0xAB) and np.all(blk[off + cb:off + 2 * cb] == 0xAB)
        pe_off = 8 * 64 * cb + 5 * 32
        assert list(blk[pe_off:pe_off + 8]) == [0x10, 0x32, 0x54, 0x76, 0x98, 0xBA, 0xDC, 0xFE]
        sz_off = 8 * 64 * cb + 2048
        for g in range(9):
            o = sz_off + (g * 64 + 5) * 4
            s, z = np.frombuffer(blk[o:o + 4].tobytes(), dtype="<f2")
            if g < 8:
                assert (s, z) == ((0.25, 4.0) if bits == 4 else (1.0, 1.0))
            else:
                assert (s, z) == (1.0, 8.0)


def test_write_read_round_trip():
    rng = np.random.default_rng(3)
    for bits in (4, 2):
        n = 150
        lat = rng.standard_normal((n, 512)).astype(np.float32).astype(np.float64)
        kpe = rng.standard_normal((n, 64)).astype(np.float32).astype(np.float64)
        table = np.array([[5, 0, 3]], np.int32)
        pool = np.zeros((6, Lo.block_bytes(bits)), np.uint8)
        Lo.write_tokens(pool, bits, lat, kpe, np.zeros(n, np.int64), np.arange(n), table)
        q, s, z = Lo.read_sequence(pool, bits, table[0], n)
        q2, s2, z2 = Lo.quantize_tokens(lat, kpe, bits)
        assert np.array_equal(q, q2) and np.array_equal(s, s2) and np.array_equal(z, z2)
        # the two unused blocks stay zero
        assert not pool[[1, 2, 4]].any()


def test_quantize_tokens_groups():
    # Group g of the content is channels [64g, 64g+64); the RoPE key is group 8 at 4 bits.
    rng = np.random.default_rng(4)
    lat = rng.standard_normal((3, 512))
    kpe = rng.standard_normal((3, 64))
    q, s, z = Lo.quantize_tokens(lat, kpe, 2)
    for g in range(8):
        qg, sg, zg = Q.quantize_groups(lat[:, 64 * g:64 * g + 64], 2)
        assert np.array_equal(q[:, 64 * g:64 * g + 64], qg) and np.array_equal(s[:, g], sg)
    qp, sp, zp = Q.quantize_groups(kpe, 4)
    assert np.array_equal(q[:, 512:], qp) and np.array_equal(z[:, 8], zp)
