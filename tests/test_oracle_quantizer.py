"""Pins of the oracle quantiser and packer (App. C.4) against hand-derived facts."""
import itertools

import numpy as np
import pytest

from oracle import quantizer as Q


def _bf16(x):
    """Round float64 values to bf16 (round-half-even on the top 16 bits)."""
    import torch
    return torch.tensor(np.asarray(x, np.float64)).to(torch.bfloat16).to(torch.float64).numpy()


def test_worked_int4_group():
    # x_k = (k mod 16 - 4) / 4: x_min = -1, x_max = 2.75, so s = 3.75 / 15 = 0.25
    # exactly, z = round(1 / 0.25) = 4 and q_k = k mod 16; dequantisation is exact.
    k = np.arange(64)
    x = (k % 16 - 4) / 4.0
    q, s, z = Q.quantize_groups(x, 4)
    assert s == 0.25 and z == 4
    assert np.array_equal(q, k % 16)
    assert np.array_equal(Q.dequantize(q, s, z), x)
    packed = Q.pack(q, 4)
    assert list(packed[:8]) == [0x10, 0x32, 0x54, 0x76, 0x98, 0xBA, 0xDC, 0xFE]
    assert np.array_equal(packed, np.tile(packed[:8], 4))


def test_worked_int2_group():
    # x_k = (k mod 4) - 1: s = 3 / 3 = 1, z = 1, q_k = k mod 4, byte = 0b11_10_01_00.
    k = np.arange(64)
    x = (k % 4) - 1.0
    q, s, z = Q.quantize_groups(x, 2)
    assert s == 1.0 and z == 1
    assert np.array_equal(q, k % 4)
    assert set(Q.pack(q, 2).tolist()) == {0xE4}


def test_ties_round_half_even():
    # x_min = 0, x_max = 15: s = 1, z = 0. 2.5 -> 2 and 3.5 -> 4, 0.5 -> 0, 1.5 -> 2.
    x = np.zeros(64)
    x[1] = 15.0
    x[2:6] = [2.5, 3.5, 0.5, 1.5]
    q, s, z = Q.quantize_groups(x, 4)
    assert s == 1.0 and z == 0
    assert list(q[2:6]) == [2, 4, 0, 2]


def test_zero_point_added_before_rounding():
    # x_min = -1, x_max = 14: s = 1, z = 1 (odd). x = 1.5 gives x/s + z = 2.5 -> 2,
    # whereas rounding first and adding z would give 3; 0.5 -> 2 (not 1).
    x = np.zeros(64)
    x[0], x[1] = -1.0, 14.0
    x[2], x[3] = 1.5, 0.5
    q, s, z = Q.quantize_groups(x, 4)
    assert s == 1.0 and z == 1
    assert q[2] == 2 and q[3] == 2


def test_scale_is_fp16_rounded_quotient():
    # d = 1, m = 15: 1/15 = 0.0666..., the nearest fp16 is 0.066650390625
    # (its neighbours are 0.0666503906 - 2^-14 and 0.066711425781).
    x = np.zeros(64)
    x[1] = 1.0
    _, s, _ = Q.quantize_groups(x, 4)
    assert s == 0.066650390625
    # m = 3: 1/3 -> fp16 0.333251953125
    _, s2, _ = Q.quantize_groups(x, 2)
    assert s2 == 0.333251953125


def test_constant_group_no_special_case():
    # A constant group has d = 0 -> s = max(0, 1e-8) / m, which underflows fp16; the
    # stored scale is then the smallest fp16 subnormal 2^-24.
    for c, qexp in [(0.0, 0), (0.5, 15), (-0.5, 0)]:
        x = np.full(64, c)
        q, s, z = Q.quantize_groups(x, 4)
        assert s == 2.0 ** -24
        assert np.all(q == qexp)
    q, s, z = Q.quantize_groups(np.full(64, -0.5), 4)
    assert z == 15  # -x_min / s is huge and clips to m


def test_round_trip_bound_random():
    rng = np.random.default_rng(0)
    for bits in (4, 2):
        m = Q.levels(bits)
        x = _bf16(rng.standard_normal((2000, 64)) * np.exp(rng.standard_normal((2000, 1))))
        q, s, z = Q.quantize_groups(x, bits)
        err = np.abs(x - Q.dequantize(q, s, z))
        t = x / s[:, None] + z[:, None]
        unclipped = (t >= -0.5) & (t <= m + 0.5)
        # Unclipped coordinates: |x - x_hat| <= s/2 (up to fp64 evaluation error).
        slack = 1e-13 * np.abs(x).max()
        assert np.all((err - s[:, None] / 2)[unclipped] <= slack)
        # Groups straddling zero: clipping at the top adds at most m * 2^-11 * s
        # (the fp16 rounding of the scale), so err <= s (1/2 + m 2^-11).
        straddle = (x.min(1) <= 0) & (x.max(1) >= 0)
        bound = s[:, None] * (0.5 + m * 2.0 ** -11) * (1 + 1e-9)
        assert np.all(err[straddle] <= bound[straddle])
        assert unclipped.mean() > 0.99


def test_codes_minimise_error_exhaustive():
    # For unclipped coordinates the chosen code is the nearest reconstruction
    # among all m+1 codes (brute force), given the stored s and z.
    rng = np.random.default_rng(1)
    for bits in (4, 2):
        m = Q.levels(bits)
        x = _bf16(rng.standard_normal((200, 64)))
        q, s, z = Q.quantize_groups(x, bits)
        cand = s[:, None, None] * (np.arange(m + 1)[None, None, :] - z[:, None, None])
        best = np.abs(x[:, :, None] - cand).min(axis=2)
        got = np.abs(x - Q.dequantize(q, s, z))
        assert np.all(got <= best + 1e-15)
        # and the zero point is the nearest integer to -x_min / s (when not clipped)
        r = -x.min(1) / s
        inside = (r > 0.5) & (r < m - 0.5)
        assert np.all(np.abs(r - z)[inside] <= 0.5)


@pytest.mark.parametrize("bits", [4, 2])
def test_pack_unpack_identity_exhaustive(bits):
    per = 8 // bits
    allbytes = np.arange(256, dtype=np.uint8)
    assert np.array_equal(Q.pack(Q.unpack(allbytes, bits), bits), allbytes)
    codes = np.array(list(itertools.product(range(1 << bits), repeat=per)), dtype=np.int64)
    assert np.array_equal(Q.unpack(Q.pack(codes, bits), bits), codes)
    # low bits first: code k of a byte sits at bits [bits*k, bits*(k+1))
    one = np.zeros(per, np.int64)
    one[1] = 1
    assert Q.pack(one, bits)[0] == 1 << bits
