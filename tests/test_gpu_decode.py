"""Parity of qmla_mla_decode (and its BF16-cache variant) with the fp64 oracle.

Bar (on every workload): max |out - oracle| <= 2e-3 and
||out - oracle|| / ||oracle|| <= 1e-3, with the oracle attending over the exact
dequantised cache s (q - z). Edge cases whose outputs are dominated by a few
large tokens are additionally checked against the oracle evaluated on the
fp16-rounded reconstruction RN_f16(s (q - z)) that the kernel's tiles hold,
where the only remaining differences are the fp16 rounding of the softmax
weights (relative 2^-11 each, so at most ~5e-4 of the largest |value|) and fp32
accumulation: there the bar is max-abs <= 1e-3 * max(1, max|ref|) and
rel-L2 <= 1e-3. Very short contexts (a handful of tokens) are checked only
that way: their output is a few reconstructed tokens, whose fp16 rounding alone
can exceed 2e-3 on the x8 outlier channels.
"""
import math

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


def check(case: Case, step: int, seqs, got_out, got_lse, max_abs=MAX_ABS, rel=REL_L2, fp16_tiles=False,
          queries=None):
    lens = case.lengths_at(step)
    outs, refs, lses, rlses = [], [], [], []
    for b in seqs:
        ref, rlse = case.oracle_decode(b, lens[b], step, fp16_tiles=fp16_tiles, queries=queries)
        outs.append(got_out[b]); refs.append(ref); lses.append(got_lse[b]); rlses.append(rlse)
    o, r = np.stack(outs), np.stack(refs)
    assert np.isfinite(o).all()
    err = np.max(np.abs(o - r))
    rl = rel_l2(o, r)
    assert err <= max_abs, f"max-abs {err:.3e}"
    assert rl <= rel, f"rel-L2 {rl:.3e}"
    assert np.max(np.abs(np.stack(lses) - np.stack(rlses))) <= LSE_ABS
    return err, rl


def check_tile(case: Case, step: int, seqs, got_out, got_lse, queries=None):
    """Against the oracle on the fp16-rounded reconstruction (tile-exact)."""
    lens = case.lengths_at(step)
    for b in seqs:
        ref, rlse = case.oracle_decode(b, lens[b], step, fp16_tiles=True, queries=queries)
        if lens[b] == 0:
            continue
        scale = max(1.0, float(np.abs(ref).max()))
        assert np.max(np.abs(got_out[b] - ref)) <= 1e-3 * scale, f"seq {b}"
        assert rel_l2(got_out[b], ref) <= 1e-3, f"seq {b}"
        assert np.max(np.abs(got_lse[b] - rlse)) <= LSE_ABS


def run_case(w, bf16=False):
    c = Case(w, bf16_cache=bf16)
    c.prefill_all()
    c.append_step(0)
    out, lse = c.decode(0)
    assert c.dev_error() == 0
    return c, out, lse


def test_tiny_workload_full():
    c, out, lse = run_case(W.WORKLOADS["tiny_b1_h16_l256_int4"])
    check(c, 0, [0], out, lse)


@pytest.mark.parametrize("bits", [4, 2])
@pytest.mark.parametrize("heads", [1, 16, 20, 64, 100, 128])
def test_shapes_and_ragged_tails(bits, heads):
    lengths = (1, 2, 63, 64, 65, 127, 128, 129, 300, 1000)
    w = W.small_workload("s", batch=len(lengths), heads=heads, lengths=lengths, c_bits=bits, seed=21 + heads,
                         latent_dist="gauss_gain_outlier" if bits == 4 else "t4_gain")
    c, out, lse = run_case(w)
    check_tile(c, 0, range(w.batch), out, lse)
    check(c, 0, [b for b in range(w.batch) if c.prefill[b] >= 256], out, lse)


def test_bf16_cache_variant():
    w = W.small_workload("b", batch=5, heads=64, lengths=(1, 64, 129, 700, 2000), seed=31)
    c, out, lse = run_case(w, bf16=True)
    check_tile(c, 0, range(w.batch), out, lse)
    check(c, 0, [3, 4], out, lse)
    w2 = W.small_workload("b2", batch=3, heads=128, lengths=(5, 4097, 200), seed=32)
    c2, out2, lse2 = run_case(w2, bf16=True)
    check_tile(c2, 0, range(w2.batch), out2, lse2)
    check(c2, 0, [1], out2, lse2)


def test_split_units_and_combine():
    # Far more tiles than SMs: every (sequence, head group) is split across
    # several CTAs and merged by the combine kernel.
    w = W.small_workload("split", batch=3, heads=128, lengths=(20000, 9000, 130), seed=41)
    c, out, lse = run_case(w)
    check(c, 0, range(w.batch), out, lse)


def test_same_answer_at_any_split():
    # The same sequence decoded alone (few splits) and next to long neighbours
    # (many splits) agrees to fp32 accumulation-order noise.
    w_many = W.small_workload("a", batch=4, heads=64, lengths=(5000, 60000, 60000, 60000), seed=51)
    w_alone = W.small_workload("a", batch=1, heads=64, lengths=(5000,), seed=51)
    ql, qp = W.queries(w_many, 0)
    c1 = Case(w_alone)
    c1.prefill_all()
    out1, _ = c1.decode(0, queries=(ql[:1].contiguous(), qp[:1].contiguous()))
    c2 = Case(w_many)
    c2.prefill_all()
    out2, _ = c2.decode(0, queries=(ql, qp))
    assert c1.dev_error() == 0 and c2.dev_error() == 0
    assert np.max(np.abs(out1[0] - out2[0])) <= 1e-4


def test_empty_and_single_token_sequences():
    w = W.small_workload("e", batch=4, heads=16, lengths=(0, 1, 0, 65), seed=61)
    c = Case(w)
    c.prefill_all()
    out, lse = c.decode(0, lens=[0, 1, 0, 65])
    assert np.all(out[0] == 0) and np.all(out[2] == 0)
    assert np.all(np.isneginf(lse[0])) and np.all(np.isneginf(lse[2]))
    # one token: every head's output is that token's reconstruction RN_f16(s (q - z))
    Cf, _ = c.oracle_cache(1, 1, fp16_tiles=True)
    assert np.array_equal(out[1], np.repeat(Cf[:1].astype(np.float32), 16, axis=0))
    check_tile(c, 0, [3], out, lse)
    assert c.dev_error() == 0


def test_rescale_path_growing_scores():
    # Scores that grow along the sequence force the reference max to move by far
    # more than 2^8 between tiles, exercising the O rescaling.
    w = W.small_workload("r", batch=2, heads=64, lengths=(1500, 700), seed=71)
    c = Case(w)
    for b in range(w.batch):
        lat, kp = c.tokens(b)
        ramp = torch.linspace(0.2, 3.0, lat.shape[0], dtype=torch.float64)[:, None]
        c._tok[b] = ((lat.double() * ramp).to(torch.bfloat16), kp)
    c.prefill_all()
    ql, qp = W.queries(w, 0)
    ql = (ql.double() * 40.0).to(torch.bfloat16)
    out, lse = c.decode(0, queries=(ql, qp))
    assert c.dev_error() == 0
    assert np.isfinite(out).all()
    # Largest score gap along the sequence, in log2 units, must exceed the threshold.
    S = []
    for b in range(w.batch):
        C, K = c.oracle_cache(b, c.prefill[b])
        s = TAU * (ql[b].double().numpy() @ C.T + qp[b].double().numpy() @ K.T) / math.log(2)
        S.append(s[:, -128:].max() - s[:, :128].max())
    assert max(S) > 16
    lens = c.prefill
    for b in range(w.batch):
        ref, rlse = c.oracle_decode(b, lens[b], 0, fp16_tiles=True, queries=(ql, qp))
        scale = np.abs(ref).max()
        assert np.max(np.abs(out[b] - ref)) <= 2e-3 * scale
        assert rel_l2(out[b], ref) <= 1e-3
        assert np.max(np.abs(lse[b] - rlse)) <= 1e-3 * max(1.0, np.abs(rlse).max())


def test_bad_block_id_flags_error_and_stays_finite():
    w = W.small_workload("bad", batch=2, heads=16, lengths=(200, 200), seed=81)
    c = Case(w)
    c.prefill_all()
    t = c.table.clone()
    t[1, 1] = 1 << 20
    c.table_d = t.cuda()
    out, lse = c.decode(0)
    assert c.dev_error() & Q.DEVERR_BAD_BLOCK
    assert np.isfinite(out).all()
    # sequence 0 is unaffected
    check_tile(c, 0, [0], out, lse)


def test_seq_len_beyond_table_flags_error():
    w = W.small_workload("over", batch=2, heads=16, lengths=(64, 64), seed=82)
    c = Case(w)
    c.prefill_all()
    out, lse = c.decode(0, lens=[64, 64 * 50])
    assert c.dev_error() & Q.DEVERR_BAD_POSITION
    assert np.all(out[1] == 0) and np.all(np.isneginf(lse[1]))


@pytest.mark.parametrize("name", ["dsv3_b64_h128_l4096_int4", "int2_b32_h128_l32768", "long_b4_h64_l128k"])
def test_full_size_workloads(name):
    w = W.WORKLOADS[name]
    c, out, lse = run_case(w)
    seqs = sorted({0, w.batch // 2, w.batch - 1})
    check(c, 0, seqs, out, lse)


def test_serving_mix_256_steps():
    w = W.WORKLOADS["serve_b128_h16_mix"]
    c = Case(w)
    c.prefill_all()
    seqs = [0, 77, 127]
    for step in range(w.steps):
        c.append_step(step)
        if step % 32 == 0 or step in (1, w.steps - 1):  # 10 of the 256 steps, spread over the run
            out, lse = c.decode(step)
            check(c, step, seqs, out, lse)
    assert c.dev_error() == 0


def test_many_units_split_over_many_pieces():
    # 40 units of ragged length: one long sequence spans dozens of CTAs, most
    # units are split over several; empty, one-token and too-long sequences sit
    # between split ones.
    rng = np.random.default_rng(7)
    lengths = [int(x) for x in rng.integers(100, 3000, size=40)]
    lengths[3], lengths[11], lengths[20], lengths[33] = 30000, 0, 1, 0
    w = W.small_workload("fuse", batch=40, heads=64, lengths=lengths, seed=93)
    c = Case(w)
    c.prefill_all()
    lens = list(lengths)
    lens[35] = 64 * (c.table_d.shape[1] + 3)  # beyond its table: an error bit, then out 0 / lse -inf
    out, lse = c.decode(0, lens=lens)
    assert c.dev_error() & Q.DEVERR_BAD_POSITION
    for b in (11, 33, 35):
        assert np.all(out[b] == 0) and np.all(np.isneginf(lse[b]))
    check_tile(c, 0, [20], out, lse)
    seqs = [0, 3, 7, 19, 21, 39]
    lens_ok = c.lengths_at(0)
    outs, refs = [], []
    for b in seqs:
        ref, rlse = c.oracle_decode(b, lens_ok[b], 0)
        outs.append(out[b]); refs.append(ref)
        assert np.max(np.abs(lse[b] - rlse)) <= LSE_ABS
    o, r = np.stack(outs), np.stack(refs)
    assert np.max(np.abs(o - r)) <= MAX_ABS and rel_l2(o, r) <= REL_L2


def test_decode_ex_matches_entry_points():
    # qmla_mla_decode_ex with a descriptor is the same computation as the
    # per-variant entry points: identical bits for the INT4 block and the BF16 cache.
    for bf16 in (False, True):
        w = W.small_workload("ex", batch=5, heads=64, lengths=(1, 200, 4097, 900, 64), seed=95)
        c = Case(w, bf16_cache=bf16)
        c.prefill_all()
        ref_out, ref_lse = c.decode(0)
        ql, qp = W.queries(w, 0)
        out = torch.full((w.batch, w.heads, 512), float("nan"), dtype=torch.float32, device="cuda")
        lse = torch.full((w.batch, w.heads), float("nan"), dtype=torch.float32, device="cuda")
        ws = Q.workspace_for(w.batch, w.heads, "cuda")
        sl = torch.tensor(c.lengths_at(0), dtype=torch.int32, device="cuda")
        Q.mla_decode_ex(c.pool, "bf16" if bf16 else 4, ql.cuda(), qp.cuda(), c.table_d, sl, TAU, out, lse, ws,
                        c.dev_err)
        torch.cuda.synchronize()
        assert np.array_equal(out.cpu().numpy(), ref_out) and np.array_equal(lse.cpu().numpy(), ref_lse)
        assert c.dev_error() == 0


def test_decode_ex_events_are_per_call():
    # Events given to one call bracket that call's main kernel only: a call in
    # between without events leaves them alone (no state survives the call).
    w = W.small_workload("evt", batch=8, heads=128, lengths=(4000,), seed=97)
    c = Case(w)
    c.prefill_all()
    ql, qp = W.queries(w, 0)
    ql, qp = ql.cuda(), qp.cuda()
    out = torch.empty((w.batch, w.heads, 512), dtype=torch.float32, device="cuda")
    lse = torch.empty((w.batch, w.heads), dtype=torch.float32, device="cuda")
    ws = Q.workspace_for(w.batch, w.heads, "cuda")
    sl = torch.tensor(c.lengths_at(0), dtype=torch.int32, device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    for e in ev:
        e.record()
    torch.cuda.synchronize()
    Q.mla_decode_ex(c.pool, 4, ql, qp, c.table_d, sl, TAU, out, lse, ws, c.dev_err, events=(ev[0], ev[1]))
    Q.mla_decode(c.pool, 4, ql, qp, c.table_d, sl, TAU, out, lse, ws, c.dev_err)
    Q.mla_decode_ex(c.pool, 4, ql, qp, c.table_d, sl, TAU, out, lse, ws, c.dev_err, events=(ev[2], ev[3]))
    torch.cuda.synchronize()
    first, second = ev[0].elapsed_time(ev[1]), ev[2].elapsed_time(ev[3])
    between = ev[1].elapsed_time(ev[2])
    assert first > 0 and second > 0
    # the middle call's main kernel runs between the two brackets
    assert between > 0.5 * min(first, second), (first, between, second)
    assert c.dev_error() == 0
