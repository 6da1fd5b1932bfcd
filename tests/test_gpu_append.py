"""The packed cache written by qmla_quant_append is byte-identical to the oracle's."""
import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import Case
from workloads import synthetic as W

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("bits", [4, 2])
@pytest.mark.parametrize("lengths", [(1,), (63, 64, 65), (300, 7, 129, 128)])
def test_small_pools_bit_exact(bits, lengths):
    w = W.small_workload("t", batch=len(lengths), heads=16, lengths=lengths, c_bits=bits, seed=11,
                         latent_dist="gauss_gain_outlier" if bits == 4 else "t4_gain")
    c = Case(w)
    c.prefill_all()
    torch.cuda.synchronize()
    blocks, want = c.oracle_pool_blocks(range(w.batch), c.prefill)
    got = c.pool.cpu().numpy()
    assert np.array_equal(got[blocks], want)
    # blocks not referenced keep their poison bytes
    assert np.all(np.delete(got, blocks, axis=0) == 0xAB)
    assert c.dev_error() == 0


def test_edge_values_bit_exact():
    # constant groups, exact ties, huge and tiny magnitudes, negative zero.
    n = 8
    lat = torch.zeros(n, 512, dtype=torch.float64)
    lat[1] = 0.5                                    # constant group -> s = 2^-24
    lat[2, :64] = torch.arange(64) % 16 - 4.0       # s = 1, z = 4 exact
    lat[3] = torch.linspace(-300, 300, 512)
    lat[4] = torch.linspace(-1e-3, 1e-3, 512)
    lat[5, ::2] = -0.0
    lat[6, :64] = torch.tensor([0.0, 15.0] + [2.5, 3.5, 0.5, 1.5] * 15 + [7.0, 8.0])
    lat[7] = torch.randn(512, generator=torch.Generator().manual_seed(5)) * 1e4
    kpe = torch.randn(n, 64, generator=torch.Generator().manual_seed(6), dtype=torch.float64)
    kpe[0] = 0.0
    lat_b, kpe_b = lat.to(torch.bfloat16), kpe.to(torch.bfloat16)
    from oracle import layout as OL
    for bits in (4, 2):
        table = torch.arange(2, dtype=torch.int32)[None, :]
        pool = torch.full((2, Q.block_bytes(bits)), 0xAB, dtype=torch.uint8, device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        pos = torch.tensor([0, 1, 2, 63, 64, 65, 100, 127], dtype=torch.int32)
        Q.quant_append(pool, bits, lat_b.cuda(), kpe_b.cuda(), torch.zeros(n, dtype=torch.int32, device="cuda"),
                       pos.cuda(), table.cuda(), err)
        want = np.full((2, Q.block_bytes(bits)), 0xAB, np.uint8)
        OL.write_tokens(want, bits, lat_b.double().numpy(), kpe_b.double().numpy(), np.zeros(n, np.int64),
                        pos.numpy(), table.numpy())
        assert np.array_equal(pool.cpu().numpy(), want)
        assert Q.read_dev_err(err) == 0


@pytest.mark.parametrize("name", list(W.WORKLOADS))
def test_workload_pools_bit_exact(name):
    w = W.WORKLOADS[name]
    c = Case(w)
    c.prefill_all()
    c.append_step(0)
    torch.cuda.synchronize()
    upto = c.lengths_at(0)
    seqs = sorted({0, w.batch // 2, w.batch - 1})
    blocks, want = c.oracle_pool_blocks(seqs, upto)
    got = c.pool[torch.tensor(blocks, device="cuda")].cpu().numpy()
    assert np.array_equal(got, want)
    assert c.dev_error() == 0


def test_bad_destinations_flag_and_skip():
    w = W.small_workload("t", batch=2, heads=16, lengths=(64,), seed=3)
    c = Case(w)
    lat, kp = c.tokens(0)
    table = c.table.clone()
    table[1, 0] = 10_000                       # block id out of range
    c.table_d = table.cuda()
    before = c.pool.clone()
    c.append(lat[:3], kp[:3], [1, 5, 0], [0, 0, 10_000])   # bad block, bad seq, bad position
    torch.cuda.synchronize()
    err = c.dev_error()
    assert err & Q.DEVERR_BAD_BLOCK and err & Q.DEVERR_BAD_SEQ and err & Q.DEVERR_BAD_POSITION
    assert torch.equal(c.pool, before)
