"""Absorbed MLA decode attention over the dequantised cache, in fp64.

Eq. (mla_compact), for one query token and head h, with the cached content
latent C (n x d_c) and the decoupled RoPE key K_P (n x d_r):

    S_h = tau (Qbar_{C,h} C^T + Q_{P,h} K_P^T)
    A_h = softmax(S_h)
    output_h = A_h C            (the value/output map B_h is applied by the caller)

Decode attends to every cached position, so the causal mask adds nothing.
Here C and K_P are the dequantised cache s (q - z) (App. C.4). The log-sum-exp
of S_h is returned alongside.

The split-result merge follows App. C.5 (global attention normalisation): for
partial results (m_j, s_j, o_j) over disjoint token sets,

    m = max_j m_j,  s = sum_j e^{m_j - m} s_j,  o = sum_j e^{m_j - m} o_j,  O = o / s.
"""
from __future__ import annotations

import numpy as np

from .layout import quantize_tokens
from .quantizer import dequantize


def dequantize_tokens(q: np.ndarray, s: np.ndarray, z: np.ndarray):
    """Codes [n,576] with per-group s, z [n,9] -> (C_hat [n,512], K_hat [n,64]) in fp64."""
    n = q.shape[0]
    x = dequantize(q.reshape(n, 9, 64), s, z).reshape(n, 576)
    return x[:, :512], x[:, 512:]


def quantized_cache(latent, k_pe, c_bits: int):
    """Dequantised cache (C_hat, K_hat) the decode kernel must attend over."""
    q, s, z = quantize_tokens(latent, k_pe, c_bits)
    return dequantize_tokens(q, s, z)


def scores(q_lat: np.ndarray, q_pe: np.ndarray, C: np.ndarray, K: np.ndarray, tau: float) -> np.ndarray:
    """S [H, n] = tau (q_lat C^T + q_pe K^T)."""
    q_lat = np.asarray(q_lat, np.float64)
    q_pe = np.asarray(q_pe, np.float64)
    return tau * (q_lat @ np.asarray(C, np.float64).T + q_pe @ np.asarray(K, np.float64).T)


def softmax_rows(S: np.ndarray) -> np.ndarray:
    mx = S.max(axis=-1, keepdims=True)
    e = np.exp(S - mx)
    return e / e.sum(axis=-1, keepdims=True)


def attend(q_lat, q_pe, C, K, tau: float):
    """Decode attention for one sequence: (out [H, 512], lse [H]) in fp64.

    With no cached token the output is 0 and the log-sum-exp is -inf.
    """
    q_lat = np.asarray(q_lat, np.float64)
    H = q_lat.shape[0]
    if np.asarray(C).shape[0] == 0:
        return np.zeros((H, np.asarray(C).shape[1] if np.asarray(C).ndim == 2 else 512)), np.full(H, -np.inf)
    S = scores(q_lat, q_pe, C, K, tau)
    mx = S.max(axis=1)
    e = np.exp(S - mx[:, None])
    den = e.sum(axis=1)
    out = (e / den[:, None]) @ np.asarray(C, np.float64)
    return out, mx + np.log(den)


def partial(q_lat, q_pe, C, K, tau: float):
    """Unnormalised partial (m, s, o) over the given tokens (App. C.5 notation)."""
    S = scores(q_lat, q_pe, C, K, tau)
    m = S.max(axis=1)
    e = np.exp(S - m[:, None])
    return m, e.sum(axis=1), e @ np.asarray(C, np.float64)


def merge(parts):
    """Merge partials [(m_j, s_j, o_j)] into (O, lse) by the App. C.5 rule."""
    m = np.max(np.stack([p[0] for p in parts]), axis=0)
    s = sum(np.exp(p[0] - m) * p[1] for p in parts)
    o = sum(np.exp(p[0] - m)[:, None] * p[2] for p in parts)
    return o / s[:, None], m + np.log(s)
