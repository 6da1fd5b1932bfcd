"""Seeded synthetic workloads shaped like the paper's native-attention study.

The paper measures its native backend on synthetic BF16 queries and cache
values (App. F.1) with d_c = 512, d_r = 64, 64-token pages and one query token
per sequence (``queries_multi`` gives several, for multi-token decoding). The five workloads below fix batch, heads, context lengths,
bit widths and value distributions; every tensor is drawn from a
``torch.Generator`` on the CPU, so a given (workload, sequence) pair always
yields the same bytes on any machine.

Distributions (the readings are listed in the design notes):

* content latent: N(0, 1) per element times a per-channel gain exp(0.5 N(0,1)),
  with four seeded outlier channels scaled by 8 ("gauss_gain_outlier"), or a
  Student-t (nu = 4) variate times the same gains without outliers ("t4_gain");
* RoPE key: N(0, 1) vectors rotated by RoPE(position, theta = 10000) with the
  half-split pairing (i, i + 32) and inverse frequency theta^(-2i/64);
* queries: q_latent ~ N(0, 1/512), q_pe ~ N(0, 1/64), all bf16.

Per-sequence tensors are seeded by (workload seed, sequence index), so a test
can regenerate one sequence of a large workload without drawing the others.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
import math

import torch

D_C = 512
D_R = 64
BLOCK_TOKENS = 64

# Stream ids: each independent draw gets its own generator so that adding a
# draw never shifts another one.
_S_GAIN, _S_OUTLIER, _S_QUERY, _S_TABLE, _S_LENGTHS = 1, 2, 3, 4, 5
_S_LATENT_BASE, _S_KPE_BASE = 1_000_000, 2_000_000


@dataclass(frozen=True)
class Workload:
    """One synthetic decode workload.

    ``lengths`` are the prefill context lengths; ``append`` tokens per
    sequence are written by ``quant_append`` right before each decode step, so
    the decode attends over ``lengths[b] + append`` tokens at step 0 and the
    lengths grow by ``append`` every further step.
    """

    name: str
    batch: int
    heads: int
    c_bits: int
    latent_dist: str
    seed: int
    lengths: tuple = field(default=())
    length_range: tuple | None = None  # (lo, hi) inclusive, seeded uniform draw
    contiguous: bool = False
    append: int = 0
    steps: int = 1

    @property
    def n_heads_padded(self) -> int:
        return self.heads


def _gen(seed: int, stream: int, device=None) -> torch.Generator:
    """The seeded generator of one stream. On the CPU (the default) it gives the
    values every test and the oracle use; on a CUDA device the same recipe gives
    other values from the same distributions (bench.py's secondary workloads,
    whose inputs are too large to draw quickly on the host)."""
    g = torch.Generator(device="cpu" if device is None else device)
    g.manual_seed(seed * 10_000_019 + stream)
    return g


def seq_lengths(w: Workload) -> list[int]:
    """Prefill lengths of the workload (before any appended token)."""
    if w.length_range is not None:
        lo, hi = w.length_range
        g = _gen(w.seed, _S_LENGTHS)
        return [int(v) for v in torch.randint(lo, hi + 1, (w.batch,), generator=g)]
    if len(w.lengths) == 1:
        return [int(w.lengths[0])] * w.batch
    assert len(w.lengths) == w.batch
    return [int(v) for v in w.lengths]


def final_lengths(w: Workload) -> list[int]:
    """Context length of every sequence after all steps' appends."""
    return [n + w.append * w.steps for n in seq_lengths(w)]


def channel_gains(w: Workload) -> torch.Tensor:
    """Per-channel gains exp(0.5 N(0,1)), times 8 on four seeded outlier channels."""
    gain = torch.exp(0.5 * torch.randn(D_C, generator=_gen(w.seed, _S_GAIN), dtype=torch.float64))
    if w.latent_dist == "gauss_gain_outlier":
        idx = torch.randperm(D_C, generator=_gen(w.seed, _S_OUTLIER))[:4]
        gain[idx] *= 8.0
    elif w.latent_dist != "t4_gain":
        raise ValueError(f"unknown latent distribution {w.latent_dist!r}")
    return gain


def latent_for_seq(w: Workload, b: int, n_tokens: int, gains: torch.Tensor | None = None,
                   device=None) -> torch.Tensor:
    """Content latent rows 0..n_tokens-1 of sequence ``b`` as bf16 [n, 512]
    (drawn on ``device``, see _gen)."""
    g = _gen(w.seed, _S_LATENT_BASE + b, device)
    if gains is None:
        gains = channel_gains(w)
    gains = gains.to(g.device)
    if w.latent_dist == "gauss_gain_outlier":
        x = torch.randn(n_tokens, D_C, generator=g, dtype=torch.float64, device=g.device)
    else:  # Student-t with 4 degrees of freedom: N / sqrt(chi2_4 / 4),
        # chi2_4 = -2 ln(U1 U2) (a sum of two exponentials with mean 2)
        z = torch.randn(n_tokens, D_C, generator=g, dtype=torch.float64, device=g.device)
        u = 1.0 - torch.rand(2, n_tokens, D_C, generator=g, dtype=torch.float64, device=g.device)
        chi = -2.0 * (torch.log(u[0]) + torch.log(u[1]))
        x = z / torch.sqrt(chi / 4.0)
    return (x * gains).to(torch.bfloat16)


def kpe_for_seq(w: Workload, b: int, n_tokens: int, theta: float = 10000.0, device=None) -> torch.Tensor:
    """RoPE key rows 0..n_tokens-1 of sequence ``b`` as bf16 [n, 64].

    Token i sits at position i; the pair (j, j + 32) is rotated by the angle
    i * theta^(-2j/64).
    """
    g = _gen(w.seed, _S_KPE_BASE + b, device)
    x = torch.randn(n_tokens, D_R, generator=g, dtype=torch.float64, device=g.device)
    half = D_R // 2
    inv_freq = theta ** (-2.0 * torch.arange(half, dtype=torch.float64, device=g.device) / D_R)
    ang = torch.arange(n_tokens, dtype=torch.float64, device=g.device)[:, None] * inv_freq[None, :]
    cos, sin = torch.cos(ang), torch.sin(ang)
    x1, x2 = x[:, :half], x[:, half:]
    out = torch.cat([x1 * cos - x2 * sin, x1 * sin + x2 * cos], dim=1)
    return out.to(torch.bfloat16)


def queries(w: Workload, step: int = 0, device=None) -> tuple[torch.Tensor, torch.Tensor]:
    """(q_latent [B,H,512], q_pe [B,H,64]) as bf16 for decode step ``step``."""
    g = _gen(w.seed, _S_QUERY + 7919 * step, device)
    ql = torch.randn(w.batch, w.heads, D_C, generator=g, dtype=torch.float64, device=g.device) / math.sqrt(D_C)
    qp = torch.randn(w.batch, w.heads, D_R, generator=g, dtype=torch.float64, device=g.device) / math.sqrt(D_R)
    return ql.to(torch.bfloat16), qp.to(torch.bfloat16)


def queries_multi(w: Workload, step: int, q_tokens: int) -> tuple[torch.Tensor, torch.Tensor]:
    """(q_latent [B,T,H,512], q_pe [B,T,H,64]) bf16 for a step that scores T new
    tokens per sequence: query token t is the single-token query of step
    step * T + t, so T = 1 gives queries(w, step)."""
    qs = [queries(w, step * q_tokens + t) for t in range(q_tokens)]
    return torch.stack([q[0] for q in qs], 1), torch.stack([q[1] for q in qs], 1)


def block_table(w: Workload) -> tuple[torch.Tensor, int]:
    """Block table [B, max_blocks] (int32, unused entries -1) and the pool size.

    Every sequence owns ceil(final_length / 64) blocks. With ``contiguous`` the
    blocks are numbered in order; otherwise the physical ids are a seeded random
    permutation of the pool, so logically adjacent blocks are scattered.
    """
    lens = final_lengths(w)
    nblk = [(n + BLOCK_TOKENS - 1) // BLOCK_TOKENS for n in lens]
    total = sum(nblk)
    max_blocks = max(nblk) if nblk else 1
    if w.contiguous:
        phys = torch.arange(total, dtype=torch.int64)
    else:
        phys = torch.randperm(total, generator=_gen(w.seed, _S_TABLE))
    table = torch.full((w.batch, max_blocks), -1, dtype=torch.int32)
    k = 0
    for b, nb in enumerate(nblk):
        table[b, :nb] = phys[k:k + nb].to(torch.int32)
        k += nb
    return table, total


def small_workload(name: str, batch: int, heads: int, lengths, c_bits: int = 4,
                   latent_dist: str = "gauss_gain_outlier", seed: int = 100,
                   contiguous: bool = False, append: int = 0, steps: int = 1) -> Workload:
    """A test-sized workload with the same distributions as the named ones."""
    lengths = tuple(lengths) if isinstance(lengths, (list, tuple)) else (int(lengths),)
    return Workload(name=name, batch=batch, heads=heads, c_bits=c_bits, latent_dist=latent_dist,
                    seed=seed, lengths=lengths, contiguous=contiguous, append=append, steps=steps)


# The five named workloads.
WORKLOADS: dict[str, Workload] = {
    # Tiny INT4/INT4 decode: B=1, 16 heads, 256 tokens, contiguous cache.
    "tiny_b1_h16_l256_int4": Workload(
        name="tiny_b1_h16_l256_int4", batch=1, heads=16, c_bits=4,
        latent_dist="gauss_gain_outlier", seed=0, lengths=(256,), contiguous=True),
    # DeepSeek-V3-shaped: B=64, 128 heads, context 4096 plus one appended token.
    "dsv3_b64_h128_l4096_int4": Workload(
        name="dsv3_b64_h128_l4096_int4", batch=64, heads=128, c_bits=4,
        latent_dist="gauss_gain_outlier", seed=1, lengths=(4096,), append=1),
    # INT2 content + INT4 RoPE key, heavy-tailed latent: B=32, 128 heads, 32768 tokens.
    "int2_b32_h128_l32768": Workload(
        name="int2_b32_h128_l32768", batch=32, heads=128, c_bits=2,
        latent_dist="t4_gain", seed=2, lengths=(32768,)),
    # Long context with skewed lengths: B=4, 64 heads.
    "long_b4_h64_l128k": Workload(
        name="long_b4_h64_l128k", batch=4, heads=64, c_bits=4,
        latent_dist="gauss_gain_outlier", seed=3, lengths=(131072, 98304, 65536, 16384)),
    # Cache-pressure serving mix: B=128, 16 heads, lengths U[1024, 16384],
    # 256 steps of (append one token per sequence, decode).
    "serve_b128_h16_mix": Workload(
        name="serve_b128_h16_mix", batch=128, heads=16, c_bits=4,
        latent_dist="gauss_gain_outlier", seed=4, length_range=(1024, 16384), append=1, steps=256),
}


def with_steps(w: Workload, steps: int) -> Workload:
    return replace(w, steps=steps)
