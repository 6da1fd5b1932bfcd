"""The fp16 tiles the decode kernel reconstructs, bit for bit. qmla_debug_tile
runs the decode's own row loaders (packed rows dequantised, protected and BF16
rows converted) into its swizzled shared-memory chunks and writes the tile out in
channel order; every element must equal the oracle's single rounding
RN_f16(s (q - z)) of the same codes (this library's block and the paper's page),
RN_f16 of the bf16 value for BF16 and protected rows, and zero past the end."""
import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import Case
from oracle import layout as OL
from oracle import paper_format as OF
from oracle import protection as OP
from oracle import quantizer as OQ
from workloads import synthetic as W

pytestmark = pytest.mark.gpu

LENS = (300, 1000, 129, 1, 64)


def _expected(c: Case, b: int, kind: str) -> np.ndarray:
    """[L, 576] fp16 values of sequence b's tile rows (all L positions)."""
    lat, kp = c.tokens(b)
    L = c.prefill[b]
    latf, kpf = lat[:L].double().numpy(), kp[:L].double().numpy()
    if kind == "bf16":
        return np.concatenate([latf, kpf], 1).astype(np.float16)
    if kind == "c4r4":
        q, s, z = OF.quantize_tokens(latf, kpf)
        C, K = OF.tile_values(q, s, z)
        x = np.concatenate([C, K], 1).astype(np.float16)
    else:
        q, s, z = OL.quantize_tokens(latf, kpf, c.w.c_bits)
        x = OQ.dequantize_fp16(q.reshape(L, 9, 64), s, z).reshape(L, 576)
    if c.protect:
        P = OP.protected_positions(L)
        x[P] = np.concatenate([latf[P], kpf[P]], 1).astype(np.float16)
    return x


def _dump(c: Case, kind_code: int, b: int, j: int) -> np.ndarray:
    tile = torch.full((128, 576), 0x7E00, dtype=torch.int16, device="cuda")   # fp16 NaN: unwritten shows
    sl = torch.tensor(c.prefill, dtype=torch.int32, device="cuda")
    Q.debug_tile(c.pool, kind_code, c.table_d, sl, b, j, tile, c.dev_err, prot=c.prot if c.protect else None)
    torch.cuda.synchronize()
    assert c.dev_error() == 0
    return tile.cpu().numpy()


@pytest.mark.parametrize("kind", ["int4", "int2", "c4r4", "bf16", "int4_protected", "c4r4_protected"])
def test_tiles_bit_exact(kind):
    bits = 2 if kind == "int2" else 4
    w = W.small_workload(f"tile_{kind}", batch=len(LENS), heads=16, lengths=LENS, c_bits=bits, seed=77,
                         latent_dist="t4_gain" if bits == 2 else "gauss_gain_outlier")
    c = Case(w, bf16_cache=kind == "bf16", c4r4=kind.startswith("c4r4"), protect=kind.endswith("protected"))
    c.prefill_all()
    code = {"int4": 4, "int2": 2, "c4r4": Q.CACHE_C4R4, "bf16": Q.CACHE_BF16}[kind.split("_")[0]]
    for b, L in enumerate(c.prefill):
        want = _expected(c, b, kind.split("_")[0])
        for j in sorted({0, (L - 1) // 256, (L - 1) // 128}):
            got = _dump(c, code, b, j)
            n = min(128, L - 128 * j)
            ref = np.zeros((128, 576), np.float16)
            ref[:n] = want[128 * j:128 * j + n]
            bad = np.argwhere(got != ref.view(np.int16))
            assert bad.size == 0, f"seq {b} tile {j}: {len(bad)} elements differ, first at {bad[:3].tolist()}"


def test_rejects_bad_arguments():
    w = W.small_workload("tile_bad", batch=1, heads=16, lengths=(10,), seed=1)
    c = Case(w)
    c.prefill_all()
    sl = torch.tensor(c.prefill, dtype=torch.int32, device="cuda")
    tile = torch.zeros((128, 576), dtype=torch.int16, device="cuda")
    for kind, b, j in ((3, 0, 0), (4, 1, 0), (4, -1, 0), (4, 0, -1), (4, 0, 5)):
        with pytest.raises(Q.QmlaError):
            Q.debug_tile(c.pool, kind, c.table_d, sl, b, j, tile, c.dev_err)
