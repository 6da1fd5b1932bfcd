"""Decode with several query tokens per sequence (qmla_mla_decode_multi) against
the oracle of Eq. mla_compact with its causal mask: ragged lengths whose query
window crosses tile edges, rows with no admissible key, splits whose pieces see
no key for some query tokens, protection, a multi-token decode loop, T = 1
against the single-token entry point, and a full-size DeepSeek-V3-shaped case."""
import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import TAU, Case, rel_l2
from workloads import synthetic as W

pytestmark = pytest.mark.gpu

MAX_ABS = 2e-3
REL_L2 = 1e-3
LSE_ABS = 1e-3

LENS = (1, 2, 3, 63, 64, 65, 127, 128, 129, 130, 131, 300, 1000)


def _check(c: Case, lens, step, T, out, lse, seqs=None, tile=False):
    for b in (range(c.w.batch) if seqs is None else seqs):
        ref, rlse = c.oracle_decode_multi(b, lens[b], step, T, fp16_tiles=tile)
        for t in range(T):
            n = lens[b] - T + t + 1
            if n <= 0:
                assert np.all(out[b, t] == 0) and np.all(np.isneginf(lse[b, t])), f"seq {b} token {t}: no key"
                continue
            assert np.isfinite(out[b, t]).all(), f"seq {b} token {t}"
            if tile:
                scale = max(1.0, float(np.abs(ref[t]).max()))
                assert np.max(np.abs(out[b, t] - ref[t])) <= 1e-3 * scale, f"seq {b} token {t} (L={lens[b]})"
            else:
                assert np.max(np.abs(out[b, t] - ref[t])) <= MAX_ABS, f"seq {b} token {t} (L={lens[b]})"
            assert rel_l2(out[b, t], ref[t]) <= REL_L2, f"seq {b} token {t} (L={lens[b]})"
            assert np.max(np.abs(lse[b, t] - rlse[t])) <= LSE_ABS, f"seq {b} token {t} (L={lens[b]})"


def _case(name, lengths, heads, seed, c_bits=4, protect=False):
    w = W.small_workload(name, batch=len(lengths), heads=heads, lengths=lengths, c_bits=c_bits, seed=seed,
                         latent_dist="gauss_gain_outlier" if c_bits == 4 else "t4_gain")
    c = Case(w, protect=protect)
    c.prefill_all()
    return c


@pytest.mark.parametrize("T,heads", [(2, 16), (3, 16), (4, 64), (8, 16), (2, 128), (5, 20)])
def test_ragged_lengths_and_query_windows(T, heads):
    c = _case(f"mq{T}_{heads}", LENS, heads, seed=10 * T + heads)
    out, lse = c.decode_multi(0, T, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, T, out, lse, tile=True)
    _check(c, c.prefill, 0, T, out, lse, seqs=[b for b in range(c.w.batch) if c.prefill[b] >= 256])


def test_int2_content():
    c = _case("mq_int2", LENS, 64, seed=91, c_bits=2)
    out, lse = c.decode_multi(0, 3, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, 3, out, lse, tile=True)


def test_split_pieces_that_see_no_key():
    # 150 sequences of 129 tokens, T = 2: the second tile of each holds only
    # position 128, which query token 0 may not see. With ~2 tiles per CTA many
    # CTA ranges start on such a tile, so their partial for token 0 is empty
    # (m = -inf, l = 0) and the merge must ignore it.
    lens = (129,) * 150
    c = _case("mq_split", lens, 16, seed=5)
    out, lse = c.decode_multi(0, 2, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, 2, out, lse, seqs=range(0, 150, 7), tile=True)


def test_long_sequence_split_across_ctas():
    c = _case("mq_long", (40000, 300), 64, seed=6)
    out, lse = c.decode_multi(0, 4, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, 4, out, lse)


def test_protected():
    lens = (1, 4, 5, 131, 132, 133, 134, 260, 1000)
    c = _case("mq_prot", lens, 16, seed=8, protect=True)
    out, lse = c.decode_multi(0, 3, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, 3, out, lse, tile=True)


def test_multi_token_decode_loop():
    # Each step appends T = 3 tokens per sequence and scores all three.
    T = 3
    w = W.small_workload("mq_loop", batch=3, heads=16, lengths=(61, 126, 500), c_bits=4, seed=12, append=T,
                         steps=4)
    c = Case(w)
    c.prefill_all()
    for step in range(w.steps):
        c.append_step(step)
        out, lse = c.decode_multi(step, T)
        assert c.dev_error() == 0
        _check(c, c.lengths_at(step), step, T, out, lse, tile=True)


def test_one_token_is_the_single_token_decode():
    c = _case("mq_t1", (5, 129, 1000, 4097), 64, seed=13)
    out1, lse1 = c.decode_multi(0, 1, lens=c.prefill)
    ql, qp = W.queries_multi(c.w, 0, 1)
    out, lse = c.decode(0, lens=c.prefill, queries=(ql[:, 0], qp[:, 0]))
    assert np.array_equal(out1[:, 0], out) and np.array_equal(lse1[:, 0], lse)


def test_full_size_dsv3_two_tokens():
    # DeepSeek-V3 shape with multi-token prediction depth 1: two query tokens per
    # sequence, 64 sequences of 4096 + 2 tokens, 128 heads (256 query rows).
    w = W.small_workload("dsv3_mtp2", batch=64, heads=128, lengths=(4096,), c_bits=4, seed=1, append=2)
    c = Case(w)
    c.prefill_all()
    c.append_step(0)
    out, lse = c.decode_multi(0, 2)
    assert c.dev_error() == 0
    _check(c, c.lengths_at(0), 0, 2, out, lse, seqs=[0, 31, 63])


def test_few_units_with_an_empty_piece():
    # One sequence of 151 * 128 + 1 tokens: 152 tiles, one per CTA on a 152-SM
    # GPU, so the last CTA's piece holds only position 19328, which query token 0
    # may not see. A single unit takes the wide merge, which must skip that piece.
    c = _case("mq_wide", (151 * 128 + 1,), 16, seed=15)
    out, lse = c.decode_multi(0, 2, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, 0, 2, out, lse)
