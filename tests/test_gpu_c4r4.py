"""The paper's own INT4 page (App. C.5 storage layout: bf16 content scales,
fp32 RoPE scale, uint8 zero points, 20,480 bytes per 64 tokens) on the GPU
against the oracle: the writer's pages byte for byte, and the decode within
the parity bar, on the exact reconstruction s (q - z) and tile-exact on the
fp16 values the kernel's tiles hold, with and without sink4/local128
protection."""
import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import POISON, Case, rel_l2
from oracle import paper_format as OF
from workloads import synthetic as W

pytestmark = pytest.mark.gpu

MAX_ABS = 2e-3
REL_L2 = 1e-3
LSE_ABS = 1e-3


def _case(name, lengths, heads=16, seed=5, protect=False, dist="gauss_gain_outlier"):
    w = W.small_workload(name, batch=len(lengths), heads=heads, lengths=lengths, c_bits=4, seed=seed,
                         latent_dist=dist)
    c = Case(w, c4r4=True, protect=protect)
    c.prefill_all()
    return c


def _check(c: Case, lens, out, lse, seqs=None, tile=False, step=0):
    for b in (range(c.w.batch) if seqs is None else seqs):
        ref, rlse = c.oracle_decode(b, lens[b], step, fp16_tiles=tile)
        if lens[b] == 0:
            continue
        assert np.isfinite(out[b]).all(), f"seq {b}"
        if tile:
            scale = max(1.0, float(np.abs(ref).max()))
            assert np.max(np.abs(out[b] - ref)) <= 1e-3 * scale, f"seq {b} (L={lens[b]})"
        else:
            assert np.max(np.abs(out[b] - ref)) <= MAX_ABS, f"seq {b} (L={lens[b]})"
        assert rel_l2(out[b], ref) <= REL_L2, f"seq {b} (L={lens[b]})"
        assert np.max(np.abs(lse[b] - rlse)) <= LSE_ABS, f"seq {b} (L={lens[b]})"


@pytest.mark.parametrize("lengths", [(1,), (63, 64, 65), (300, 7, 129, 128)])
@pytest.mark.parametrize("dist", ["gauss_gain_outlier", "t4_gain"])
def test_writer_pages_bit_exact(lengths, dist):
    c = _case("c4w", lengths, dist=dist)
    torch.cuda.synchronize()
    assert c.dev_error() == 0
    blocks, want = c.oracle_pool_blocks(range(c.w.batch), c.prefill)
    got = c.pool.cpu().numpy()
    assert got.shape[1] == OF.PAGE_BYTES == Q.c4r4_page_bytes()
    assert np.array_equal(got[blocks], want)          # padding included: never written
    assert np.all(np.delete(got, blocks, axis=0) == POISON)


def _edge_tokens():
    # constant groups (the 1e-8 floor: s far below fp16's normal range, so the
    # decode takes its fp32 path), exact ties, huge and tiny ranges, -0.0
    n = 8
    lat = torch.zeros(n, 512, dtype=torch.float64)
    lat[1] = 0.5
    lat[2, :64] = torch.arange(64) % 16 - 4.0
    lat[3] = torch.linspace(-300, 300, 512)
    lat[4] = torch.linspace(-1e-3, 1e-3, 512)
    lat[5, ::2] = -0.0
    lat[6, :64] = torch.tensor([0.0, 15.0] + [2.5, 3.5, 0.5, 1.5] * 15 + [7.0, 8.0])
    lat[7] = torch.randn(512, generator=torch.Generator().manual_seed(5)) * 1e4
    kpe = torch.randn(n, 64, generator=torch.Generator().manual_seed(6), dtype=torch.float64)
    kpe[0] = 0.0
    kpe[3] *= 1e3
    kpe[4] *= 1e-5
    return lat.to(torch.bfloat16), kpe.to(torch.bfloat16)


def test_writer_edge_values_bit_exact():
    lat, kpe = _edge_tokens()
    n = lat.shape[0]
    table = torch.arange(2, dtype=torch.int32)[None, :]
    pool = torch.full((2, Q.c4r4_page_bytes()), POISON, dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    pos = torch.tensor([0, 1, 2, 63, 64, 65, 100, 127], dtype=torch.int32)
    Q.quant_append_c4r4(pool, lat.cuda(), kpe.cuda(), torch.zeros(n, dtype=torch.int32, device="cuda"), pos.cuda(),
                        table.cuda(), err)
    want = np.full((2, OF.PAGE_BYTES), POISON, np.uint8)
    OF.write_tokens(want, lat.double().numpy(), kpe.double().numpy(), np.zeros(n, np.int64), pos.numpy(),
                    table.numpy())
    assert np.array_equal(pool.cpu().numpy(), want)
    assert Q.read_dev_err(err) == 0


def test_decode_edge_values_tile_exact():
    # The edge tokens of the writer test as a 8-token context, checked on the fp16
    # tile values (content fp16 path, content fp32 path, RoPE fp32 path).
    lat, kpe = _edge_tokens()
    n = lat.shape[0]
    table = torch.zeros((1, 1), dtype=torch.int32)
    pool = torch.full((1, Q.c4r4_page_bytes()), POISON, dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    Q.quant_append_c4r4(pool, lat.cuda(), kpe.cuda(), torch.zeros(n, dtype=torch.int32, device="cuda"),
                        torch.arange(n, dtype=torch.int32, device="cuda"), table.cuda(), err)
    g = torch.Generator().manual_seed(9)
    ql = (torch.randn(1, 16, 512, generator=g) * 1e-3).to(torch.bfloat16)
    qp = (torch.randn(1, 16, 64, generator=g) * 1e-3).to(torch.bfloat16)
    out = torch.empty((1, 16, 512), dtype=torch.float32, device="cuda")
    lse = torch.empty((1, 16), dtype=torch.float32, device="cuda")
    ws = Q.workspace_for(1, 16, "cuda")
    tau = 1.0 / np.sqrt(192.0)
    Q.mla_decode_c4r4(pool, ql.cuda(), qp.cuda(), table.cuda(), torch.tensor([n], dtype=torch.int32, device="cuda"),
                      tau, out, lse, ws, err)
    torch.cuda.synchronize()
    assert Q.read_dev_err(err) == 0
    q, s, z = OF.quantize_tokens(lat.double().numpy(), kpe.double().numpy())
    C, K = OF.tile_values(q, s, z)
    from oracle import attention as OA
    ref, rlse = OA.attend(ql[0].double().numpy(), qp[0].double().numpy(), C, K, tau)
    got = out[0].cpu().numpy()
    scale = max(1.0, float(np.abs(ref).max()))
    assert np.max(np.abs(got - ref)) <= 1e-3 * scale
    assert np.max(np.abs(lse[0].cpu().numpy() - rlse)) <= LSE_ABS


@pytest.mark.parametrize("heads", [1, 16, 64, 100, 128])
def test_decode_shapes_and_ragged_tails(heads):
    lengths = (1, 2, 63, 64, 65, 127, 128, 129, 300, 1000)
    c = _case("c4d", lengths, heads=heads, seed=40 + heads)
    out, lse = c.decode(0, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, out, lse, tile=True)
    _check(c, c.prefill, out, lse, seqs=[b for b in range(c.w.batch) if c.prefill[b] >= 256])


@pytest.mark.parametrize("heads", [16, 128])
def test_decode_protected(heads):
    lengths = (1, 4, 5, 131, 132, 133, 260, 1000, 4097)
    c = _case("c4p", lengths, heads=heads, seed=60 + heads, protect=True)
    out, lse = c.decode(0, lens=c.prefill)
    assert c.dev_error() == 0
    _check(c, c.prefill, out, lse, tile=True)
    _check(c, c.prefill, out, lse, seqs=[b for b in range(c.w.batch) if c.prefill[b] >= 256])


def test_decode_loop_appends_one_token_per_step():
    w = W.small_workload("c4loop", batch=3, heads=16, lengths=(62, 127, 500), c_bits=4, seed=71, append=1, steps=6)
    c = Case(w, c4r4=True)
    c.prefill_all()
    for step in range(w.steps):
        c.append_step(step)
        out, lse = c.decode(step)
        assert c.dev_error() == 0
        _check(c, c.lengths_at(step), out, lse, tile=True, step=step)


@pytest.mark.parametrize("name", ["dsv3_b64_h128_l4096_int4", "long_b4_h64_l128k"])
def test_full_size_sampled(name):
    w = W.WORKLOADS[name]
    c = Case(w, c4r4=True)
    c.prefill_all()
    c.append_step(0)
    out, lse = c.decode(0)
    assert c.dev_error() == 0
    _check(c, c.lengths_at(0), out, lse, seqs=sorted({0, w.batch // 2, w.batch - 1}))
