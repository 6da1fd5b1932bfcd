"""Test harness: drives the CUDA library and the CPU oracle on the same seeded inputs.

The oracle sees only the generator's bf16 inputs (never anything the GPU
produced); the GPU sees the same bytes through the library's C ABI.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import paper_2609_36760_gb300 as Q
from oracle import attention as OA
from oracle import layout as OL
from oracle import multi_query as OM
from oracle import paper_format as OF
from oracle import protection as OP
from oracle import quantizer as OQ
from workloads import synthetic as W

TAU = 1.0 / math.sqrt(192.0)
POISON = 0xAB


def rel_l2(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


class Case:
    """A workload materialised on the GPU (packed or BF16 cache) plus its inputs on the host.
    c4r4=True stores the packed cache in the paper's page format (INT4 only)."""

    def __init__(self, w: W.Workload, bf16_cache: bool = False, device: str = "cuda", protect: bool = False,
                 c4r4: bool = False):
        assert not c4r4 or (w.c_bits == 4 and not bf16_cache)
        self.w = w
        self.bf16 = bf16_cache
        self.c4r4 = c4r4
        self.protect = protect
        self.dev = device
        self.prefill = W.seq_lengths(w)
        self.final = W.final_lengths(w)
        table, nblocks = W.block_table(w)
        self.table = table
        self.nblocks = nblocks
        self.gains = W.channel_gains(w)
        bb = Q.bf16_block_bytes() if bf16_cache else (Q.c4r4_page_bytes() if c4r4 else Q.block_bytes(w.c_bits))
        self.pool = torch.full((nblocks, bb), POISON, dtype=torch.uint8, device=device)
        self.table_d = table.to(device)
        self.dev_err = torch.zeros(1, dtype=torch.int32, device=device)
        self._tok = {}
        # sink4/local128 protection rows, poisoned with bf16 NaN so that a row read
        # before the writer filled it shows up in the output
        self.prot = (torch.full((w.batch, 132, 576), 0xFFFF, dtype=torch.int32, device=device)
                     .to(torch.int16).view(torch.bfloat16) if protect else None)

    # host-side inputs, cached per sequence (bf16 tensors up to the final length)
    def tokens(self, b: int):
        if b not in self._tok:
            n = self.final[b]
            self._tok[b] = (W.latent_for_seq(self.w, b, n, self.gains), W.kpe_for_seq(self.w, b, n))
        return self._tok[b]

    def append(self, lat: torch.Tensor, kpe: torch.Tensor, seq_ids, positions, lens_after=None) -> None:
        lat_d = lat.contiguous().to(self.dev)
        kpe_d = kpe.contiguous().to(self.dev)
        sid = None if seq_ids is None else torch.as_tensor(seq_ids, dtype=torch.int32).to(self.dev)
        pos = torch.as_tensor(positions, dtype=torch.int32).to(self.dev)
        if self.c4r4:
            la = torch.as_tensor(lens_after, dtype=torch.int32).to(self.dev) if self.protect else None
            Q.quant_append_c4r4(self.pool, lat_d, kpe_d, sid, pos, self.table_d, self.dev_err, seq_lens=la,
                                prot=self.prot)
        elif self.protect:
            la = torch.as_tensor(lens_after, dtype=torch.int32).to(self.dev)
            Q.quant_append_protected(self.pool, self.w.c_bits, lat_d, kpe_d, sid, pos, self.table_d, la, self.prot,
                                     self.dev_err)
        elif self.bf16:
            Q.bf16_append(self.pool, lat_d, kpe_d, sid, pos, self.table_d, self.dev_err)
        else:
            Q.quant_append(self.pool, self.w.c_bits, lat_d, kpe_d, sid, pos, self.table_d, self.dev_err)

    def prefill_all(self, chunk_tokens: int = 1 << 20) -> None:
        """Writes tokens [0, prefill_b) of every sequence."""
        lats, kps, sids, poss = [], [], [], []
        pending = 0
        for b in range(self.w.batch):
            n = self.prefill[b]
            if n == 0:
                continue
            lat, kp = self.tokens(b)
            lats.append(lat[:n]); kps.append(kp[:n])
            sids.append(torch.full((n,), b, dtype=torch.int32)); poss.append(torch.arange(n, dtype=torch.int32))
            pending += n
            if pending >= chunk_tokens:
                self.append(torch.cat(lats), torch.cat(kps), torch.cat(sids), torch.cat(poss), self.prefill)
                lats, kps, sids, poss, pending = [], [], [], [], 0
        if pending:
            self.append(torch.cat(lats), torch.cat(kps), torch.cat(sids), torch.cat(poss), self.prefill)

    def lengths_at(self, step: int) -> list[int]:
        return [n + self.w.append * (step + 1) for n in self.prefill]

    def append_step(self, step: int) -> None:
        """Writes the ``append`` tokens of every sequence for decode step ``step``."""
        if self.w.append == 0:
            return
        lats, kps, sids, poss = [], [], [], []
        for b in range(self.w.batch):
            lat, kp = self.tokens(b)
            a0 = self.prefill[b] + self.w.append * step
            for k in range(self.w.append):
                lats.append(lat[a0 + k:a0 + k + 1]); kps.append(kp[a0 + k:a0 + k + 1])
                sids.append(b); poss.append(a0 + k)
        self.append(torch.cat(lats), torch.cat(kps), sids, poss, self.lengths_at(step))

    def decode(self, step: int, lens: list[int] | None = None, queries=None):
        ql, qp = queries if queries is not None else W.queries(self.w, step)
        lens = self.lengths_at(step) if lens is None else lens
        B, H = self.w.batch, self.w.heads
        out = torch.full((B, H, 512), float("nan"), dtype=torch.float32, device=self.dev)
        lse = torch.full((B, H), float("nan"), dtype=torch.float32, device=self.dev)
        ws = Q.workspace_for(B, H, self.dev)
        ws.fill_(0x7F)
        sl = torch.tensor(lens, dtype=torch.int32, device=self.dev)
        ql_d, qp_d = ql.contiguous().to(self.dev), qp.contiguous().to(self.dev)
        if self.c4r4:
            Q.mla_decode_c4r4(self.pool, ql_d, qp_d, self.table_d, sl, TAU, out, lse, ws, self.dev_err,
                              prot=self.prot if self.protect else None)
        elif self.protect:
            Q.mla_decode_protected(self.pool, self.w.c_bits, ql_d, qp_d, self.table_d, sl, self.prot, TAU, out, lse,
                                   ws, self.dev_err)
        elif self.bf16:
            Q.mla_decode_bf16cache(self.pool, ql_d, qp_d, self.table_d, sl, TAU, out, lse, ws, self.dev_err)
        else:
            Q.mla_decode(self.pool, self.w.c_bits, ql_d, qp_d, self.table_d, sl, TAU, out, lse, ws, self.dev_err)
        torch.cuda.synchronize()
        return out.cpu().numpy(), lse.cpu().numpy()

    def decode_multi(self, step: int, q_tokens: int, lens: list[int] | None = None):
        """mla_decode_multi with T = q_tokens query tokens per sequence (the last
        T positions of each sequence): (out [B,T,H,512], lse [B,T,H]) on the host."""
        ql, qp = W.queries_multi(self.w, step, q_tokens)
        lens = self.lengths_at(step) if lens is None else lens
        B, H = self.w.batch, self.w.heads
        out = torch.full((B, q_tokens, H, 512), float("nan"), dtype=torch.float32, device=self.dev)
        lse = torch.full((B, q_tokens, H), float("nan"), dtype=torch.float32, device=self.dev)
        ws = Q.workspace_for(B, q_tokens * H, self.dev)
        ws.fill_(0x7F)
        sl = torch.tensor(lens, dtype=torch.int32, device=self.dev)
        Q.mla_decode_multi(self.pool, self.w.c_bits, ql.contiguous().to(self.dev), qp.contiguous().to(self.dev),
                           self.table_d, sl, TAU, out, lse, ws, self.dev_err,
                           prot=self.prot if self.protect else None)
        torch.cuda.synchronize()
        return out.cpu().numpy(), lse.cpu().numpy()

    def oracle_decode_multi(self, b: int, L: int, step: int, q_tokens: int, fp16_tiles: bool = False):
        ql, qp = W.queries_multi(self.w, step, q_tokens)
        C, K = self.oracle_cache(b, L, fp16_tiles)
        return OM.attend_multi(ql[b].double().numpy(), qp[b].double().numpy(), C, K, TAU)

    def dev_error(self) -> int:
        return Q.read_dev_err(self.dev_err)

    # ---------------------------------------------------------------- oracle side
    def oracle_cache(self, b: int, L: int, fp16_tiles: bool = False):
        lat, kp = self.tokens(b)
        latf = lat[:L].double().numpy()
        kpf = kp[:L].double().numpy()
        if self.bf16:
            return latf, kpf
        if self.c4r4:
            q, s, z = OF.quantize_tokens(latf, kpf)
            C, K = OF.tile_values(q, s, z) if fp16_tiles else OF.dequantize_tokens(q, s, z)
        elif fp16_tiles:
            q, s, z = OL.quantize_tokens(latf, kpf, self.w.c_bits)
            x = OQ.dequantize_fp16(q.reshape(L, 9, 64), s, z).astype(np.float64).reshape(L, 576)
            C, K = x[:, :512], x[:, 512:]
        else:
            q, s, z = OL.quantize_tokens(latf, kpf, self.w.c_bits)
            C, K = OA.dequantize_tokens(q, s, z)
        if self.protect:
            # protected positions attend with the original values (rounded to fp16
            # in the tile-exact variant, as the kernel's tiles hold them)
            C, K = np.array(C), np.array(K)
            P = OP.protected_positions(L)
            rnd = (lambda a: a.astype(np.float16).astype(np.float64)) if fp16_tiles else (lambda a: a)
            C[P] = rnd(latf[P])
            K[P] = rnd(kpf[P])
        return C, K

    def oracle_decode(self, b: int, L: int, step: int = 0, heads=None, fp16_tiles: bool = False, queries=None):
        ql, qp = queries if queries is not None else W.queries(self.w, step)
        C, K = self.oracle_cache(b, L, fp16_tiles)
        hs = slice(None) if heads is None else heads
        return OA.attend(ql[b, hs].double().numpy(), qp[b, hs].double().numpy(), C, K, TAU)

    def oracle_pool_blocks(self, seqs, upto: list[int]):
        """Oracle-written bytes of the blocks owned by ``seqs`` (tokens [0, upto[b]))."""
        bb = OF.PAGE_BYTES if self.c4r4 else OL.block_bytes(self.w.c_bits)
        pool = np.full((self.nblocks, bb), POISON, np.uint8)
        for b in seqs:
            lat, kp = self.tokens(b)
            n = upto[b]
            if self.c4r4:
                OF.write_tokens(pool, lat[:n].double().numpy(), kp[:n].double().numpy(), np.full(n, b),
                                np.arange(n), self.table.numpy())
            else:
                OL.write_tokens(pool, self.w.c_bits, lat[:n].double().numpy(), kp[:n].double().numpy(),
                                np.full(n, b), np.arange(n), self.table.numpy())
        blocks = sorted({int(x) for b in seqs for x in self.table[b].tolist() if x >= 0})
        return blocks, pool[blocks]

    def oracle_prot_rows(self, b: int, L: int) -> np.ndarray:
        """Expected protection rows of request b at length L: [132, 576] fp64, NaN where unused."""
        lat, kp = self.tokens(b)
        buf = np.full((1, 132, 576), np.nan)
        OP.write_protection(buf, lat[:L].double().numpy(), kp[:L].double().numpy(), np.zeros(L, int), np.arange(L), [L])
        return buf[0]
