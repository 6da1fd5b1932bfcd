"""The seeded generators are deterministic and have the documented shapes and spread."""
import math

import torch

from workloads import synthetic as W


def test_deterministic_and_shapes():
    w = W.WORKLOADS["tiny_b1_h16_l256_int4"]
    a = W.latent_for_seq(w, 0, 256)
    b = W.latent_for_seq(w, 0, 256)
    assert a.dtype == torch.bfloat16 and a.shape == (256, 512)
    assert torch.equal(a, b)
    # a prefix of a longer draw is the same tokens
    assert torch.equal(W.latent_for_seq(w, 0, 100), a[:100])
    kp = W.kpe_for_seq(w, 0, 256)
    assert kp.shape == (256, 64) and torch.equal(kp[:10], W.kpe_for_seq(w, 0, 10))
    ql, qp = W.queries(w)
    assert ql.shape == (1, 16, 512) and qp.shape == (1, 16, 64)
    assert abs(ql.double().std().item() - 1 / math.sqrt(512)) < 0.005
    assert abs(qp.double().std().item() - 1 / 8) < 0.02


def test_rope_preserves_pair_norms():
    w = W.WORKLOADS["tiny_b1_h16_l256_int4"]
    kp = W.kpe_for_seq(w, 0, 256).double()
    g = W._gen(w.seed, W._S_KPE_BASE + 0)
    raw = torch.randn(256, 64, generator=g, dtype=torch.float64)
    n_rot = kp[:, :32] ** 2 + kp[:, 32:] ** 2
    n_raw = raw[:, :32] ** 2 + raw[:, 32:] ** 2
    assert torch.allclose(n_rot, n_raw, rtol=2e-2, atol=1e-2)
    assert torch.allclose(kp[0], raw[0].to(torch.bfloat16).double())  # position 0: no rotation


def test_block_tables():
    w = W.WORKLOADS["dsv3_b64_h128_l4096_int4"]
    t, total = W.block_table(w)
    assert t.shape == (64, 65) and total == 64 * 65
    assert sorted(t.flatten().tolist()) == list(range(total))
    wc = W.WORKLOADS["tiny_b1_h16_l256_int4"]
    tc, tot = W.block_table(wc)
    assert tc.tolist() == [[0, 1, 2, 3]] and tot == 4
    ws = W.WORKLOADS["serve_b128_h16_mix"]
    lens = W.seq_lengths(ws)
    assert len(lens) == 128 and min(lens) >= 1024 and max(lens) <= 16384
    t4, tot4 = W.block_table(ws)
    assert tot4 == sum(-(-(n + 256) // 64) for n in lens)


def test_outliers_and_heavy_tails():
    w = W.WORKLOADS["tiny_b1_h16_l256_int4"]
    g = W.channel_gains(w)
    assert (g > 8 * 0.2).sum() >= 4 and g.max() > 8 * 0.5
    w2 = W.WORKLOADS["int2_b32_h128_l32768"]
    x = W.latent_for_seq(w2, 0, 512).double() / W.channel_gains(w2)
    kurt = ((x - x.mean()) ** 4).mean() / x.var() ** 2
    assert kurt > 4.0   # Student-t(4) is heavy-tailed (normal: 3)
