"""qmla_mla_decode_pair (units of 128 query rows on CTA pairs) against the fp64
oracle at the spec bar (max-abs <= 2e-3, rel-L2 <= 1e-3), against the
oracle on the fp16-rounded reconstruction for short contexts (max-abs <= 1e-3 *
max(1, max|ref|)), and against qmla_mla_decode on the same inputs: ragged
lengths across tile edges, INT2 content, empty sequences, units split over
many pairs and merged, the rescale path, several query tokens per sequence,
and the DeepSeek-V3-shaped workload at full size."""
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
LENS = (1, 2, 63, 64, 65, 127, 128, 129, 300, 1000)


def decode_pair(c: Case, lens, queries=None, q_tokens=1):
    """(out, lse) of qmla_mla_decode_pair on the host."""
    if q_tokens == 1:
        ql, qp = queries if queries is not None else W.queries(c.w, 0)
        shape = (c.w.batch, c.w.heads)
    else:
        ql, qp = W.queries_multi(c.w, 0, q_tokens)
        shape = (c.w.batch, q_tokens, c.w.heads)
    out = torch.full(shape + (512,), float("nan"), dtype=torch.float32, device="cuda")
    lse = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
    ws = Q.workspace_for(c.w.batch, q_tokens * c.w.heads, "cuda")
    ws.fill_(0x7F)
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    Q.mla_decode_pair(c.pool, c.w.c_bits, ql.contiguous().cuda(), qp.contiguous().cuda(), c.table_d, sl, TAU, out,
                      lse, ws, c.dev_err)
    torch.cuda.synchronize()
    return out.cpu().numpy(), lse.cpu().numpy()


def check(c: Case, lens, out, lse, seqs, tile=False, queries=None):
    for b in seqs:
        if lens[b] == 0:
            assert np.all(out[b] == 0) and np.all(np.isneginf(lse[b])), f"seq {b}: empty"
            continue
        ref, rlse = c.oracle_decode(b, lens[b], 0, fp16_tiles=tile, queries=queries)
        assert np.isfinite(out[b]).all(), f"seq {b}"
        if tile:
            assert np.max(np.abs(out[b] - ref)) <= 1e-3 * max(1.0, float(np.abs(ref).max())), f"seq {b}"
        else:
            assert np.max(np.abs(out[b] - ref)) <= MAX_ABS, f"seq {b} (L={lens[b]})"
        assert rel_l2(out[b], ref) <= REL_L2, f"seq {b} (L={lens[b]})"
        assert np.max(np.abs(lse[b] - rlse)) <= LSE_ABS, f"seq {b} (L={lens[b]})"


def _case(name, lengths, seed, c_bits=4, heads=128):
    w = W.small_workload(name, batch=len(lengths), heads=heads, lengths=lengths, c_bits=c_bits, seed=seed,
                         latent_dist="gauss_gain_outlier" if c_bits == 4 else "t4_gain")
    c = Case(w)
    c.prefill_all()
    return c


@pytest.mark.parametrize("bits", [4, 2])
def test_ragged_lengths(bits):
    c = _case(f"pair{bits}", LENS, seed=300 + bits, c_bits=bits)
    out, lse = decode_pair(c, c.prefill)
    assert c.dev_error() == 0
    check(c, c.prefill, out, lse, range(c.w.batch), tile=True)
    check(c, c.prefill, out, lse, [b for b in range(c.w.batch) if c.prefill[b] >= 256])
    # the single-CTA kernel on the same cache and queries
    out1, lse1 = c.decode(0, lens=c.prefill)
    assert np.max(np.abs(out - out1)) <= 1e-3 * max(1.0, float(np.abs(out1).max()))
    assert np.max(np.abs(lse - lse1)) <= 1e-4 * max(1.0, float(np.abs(lse1).max()))


def test_empty_sequences_and_split_units():
    # one long unit over many pairs (merged), empty sequences next to it
    c = _case("pair_split", (0, 40000, 0, 700), seed=311)
    out, lse = decode_pair(c, c.prefill)
    assert c.dev_error() == 0
    check(c, c.prefill, out, lse, range(c.w.batch))


def test_rescale_path_growing_scores():
    w = W.small_workload("pair_r", batch=2, heads=128, lengths=(1500, 700), seed=321)
    c = Case(w)
    for b in range(w.batch):
        lat, kp = c.tokens(b)
        ramp = torch.linspace(0.2, 3.0, lat.shape[0], dtype=torch.float64)[:, None]
        c._tok[b] = ((lat.double() * ramp).to(torch.bfloat16), kp)
    c.prefill_all()
    ql, qp = W.queries(w, 0)
    ql = (ql.double() * 40.0).to(torch.bfloat16)
    out, lse = decode_pair(c, c.prefill, queries=(ql, qp))
    assert c.dev_error() == 0
    S = []
    for b in range(w.batch):
        C, K = c.oracle_cache(b, c.prefill[b])
        s = TAU * (ql[b].double().numpy() @ C.T + qp[b].double().numpy() @ K.T) / math.log(2)
        S.append(s[:, -128:].max() - s[:, :128].max())
    assert max(S) > 16
    for b in range(w.batch):
        ref, rlse = c.oracle_decode(b, c.prefill[b], 0, fp16_tiles=True, queries=(ql, qp))
        assert np.max(np.abs(out[b] - ref)) <= 2e-3 * np.abs(ref).max()
        assert rel_l2(out[b], ref) <= 1e-3
        assert np.max(np.abs(lse[b] - rlse)) <= 1e-3 * max(1.0, np.abs(rlse).max())


def test_two_query_tokens():
    c = _case("pair_mq", (1, 2, 129, 300, 1000, 2000), seed=331)
    out, lse = decode_pair(c, c.prefill, q_tokens=2)
    assert c.dev_error() == 0
    for b in range(c.w.batch):
        ref, rlse = c.oracle_decode_multi(b, c.prefill[b], 0, 2, fp16_tiles=True)
        for t in range(2):
            if c.prefill[b] - 2 + t + 1 <= 0:
                assert np.all(out[b, t] == 0) and np.all(np.isneginf(lse[b, t]))
                continue
            assert np.max(np.abs(out[b, t] - ref[t])) <= 1e-3 * max(1.0, float(np.abs(ref[t]).max())), (b, t)
            assert rel_l2(out[b, t], ref[t]) <= REL_L2, (b, t)
            assert np.max(np.abs(lse[b, t] - rlse[t])) <= LSE_ABS, (b, t)


def test_unsupported_head_count():
    c = _case("pair_h64", (100,), seed=341, heads=64)
    with pytest.raises(Q.QmlaError):
        decode_pair(c, c.prefill)


def test_dsv3_full_size():
    w = W.WORKLOADS["dsv3_b64_h128_l4096_int4"]
    c = Case(w)
    c.prefill_all()
    c.append_step(0)
    lens = c.lengths_at(0)
    out, lse = decode_pair(c, lens)
    assert c.dev_error() == 0
    check(c, lens, out, lse, [0, 31, 63])
