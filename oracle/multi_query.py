"""Decode with several query tokens per sequence, in fp64. Test infrastructure:
used by tests/ only.

Eq. (mla_compact) with its additive causal mask M_attn. A step that scores T
new tokens at once (multi-token prediction, speculative verification) has, for
a sequence of L cached tokens whose last T are those new tokens, query rows at
positions L - T, ..., L - 1. Query row t may attend to key positions
p <= L - T + t, so

    M_attn[t, p] = 0 if p <= L - T + t else -inf,
    S_{t,h} = tau (Qbar_{C,t,h} C^T + Q_{P,t,h} K_P^T) + M_attn[t, :],
    A_{t,h} = softmax(S_{t,h}),   out_{t,h} = A_{t,h} C.

A row with no admissible key (L - T + t < 0) has out = 0 and lse = -inf, the
convention of the single-token decode for an empty sequence.

The split-result merge of App. C.5 extends to masked rows: a partial over a key
set with no admissible key for a row carries (m, s, o) = (-inf, 0, 0) for that
row and contributes nothing.
"""
from __future__ import annotations

import numpy as np


def causal_mask(L: int, T: int) -> np.ndarray:
    """M_attn [T, L]: 0 where key p is admissible for query row t, -inf elsewhere."""
    t = np.arange(T)[:, None]
    p = np.arange(L)[None, :]
    return np.where(p <= L - T + t, 0.0, -np.inf)


def masked_scores(q_lat, q_pe, C, K, tau: float, L_total: int | None = None, key_pos=None) -> np.ndarray:
    """S [T, H, n] for query rows q_lat [T, H, 512], q_pe [T, H, 64] against keys
    C [n, 512], K [n, 64] at positions key_pos (default 0..n-1) of a sequence of
    L_total tokens (default n), with M_attn added."""
    q_lat = np.asarray(q_lat, np.float64)
    q_pe = np.asarray(q_pe, np.float64)
    C = np.asarray(C, np.float64)
    K = np.asarray(K, np.float64)
    n = C.shape[0]
    L = n if L_total is None else int(L_total)
    pos = np.arange(n) if key_pos is None else np.asarray(key_pos)
    T = q_lat.shape[0]
    S = tau * (np.einsum("thc,pc->thp", q_lat, C) + np.einsum("thr,pr->thp", q_pe, K))
    return S + causal_mask(L, T)[:, None, :][..., pos]


def attend_multi(q_lat, q_pe, C, K, tau: float):
    """All T query rows of one sequence over its L cached tokens (C [L, 512],
    K [L, 64]): (out [T, H, 512], lse [T, H])."""
    C = np.asarray(C, np.float64)
    T, H = np.asarray(q_lat).shape[:2]
    out = np.zeros((T, H, C.shape[1] if C.ndim == 2 else 512))
    lse = np.full((T, H), -np.inf)
    if C.shape[0] == 0:
        return out, lse
    S = masked_scores(q_lat, q_pe, C, K, tau)
    for t in range(T):
        for h in range(H):
            row = S[t, h]
            if not np.isfinite(row).any():
                continue
            mx = row.max()
            e = np.exp(row - mx)
            den = e.sum()
            out[t, h] = (e / den) @ C
            lse[t, h] = mx + np.log(den)
    return out, lse


def partial_multi(q_lat, q_pe, C, K, tau: float, L_total: int, key_pos):
    """Unnormalised partial (m, s, o) [T, H], [T, H], [T, H, 512] over the keys
    at key_pos of a sequence of L_total tokens; rows with no admissible key in
    this set get (-inf, 0, 0)."""
    C = np.asarray(C, np.float64)
    S = masked_scores(q_lat, q_pe, C, K, tau, L_total, key_pos)
    T, H = S.shape[:2]
    m = np.full((T, H), -np.inf)
    s = np.zeros((T, H))
    o = np.zeros((T, H, C.shape[1]))
    for t in range(T):
        for h in range(H):
            row = S[t, h]
            if row.size == 0 or not np.isfinite(row).any():
                continue
            m[t, h] = row.max()
            e = np.exp(row - m[t, h])
            s[t, h] = e.sum()
            o[t, h] = e @ C
    return m, s, o


def merge_multi(parts):
    """App. C.5 merge of masked partials; a row that is empty in every part
    gives out = 0, lse = -inf."""
    m = np.max(np.stack([p[0] for p in parts]), axis=0)
    finite = np.isfinite(m)
    mm = np.where(finite, m, 0.0)
    s = sum(np.where(np.isfinite(p[0]), np.exp(np.where(np.isfinite(p[0]), p[0], 0.0) - mm), 0.0) * p[1]
            for p in parts)
    o = sum((np.where(np.isfinite(p[0]), np.exp(np.where(np.isfinite(p[0]), p[0], 0.0) - mm), 0.0))[..., None] * p[2]
            for p in parts)
    out = np.where(finite[..., None], o / np.where(s > 0, s, 1.0)[..., None], 0.0)
    lse = np.where(finite, mm + np.log(np.where(s > 0, s, 1.0)), -np.inf)
    return out, lse
