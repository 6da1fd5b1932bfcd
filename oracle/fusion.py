"""Offline-fusion identities of the learned transformations, in fp64 (Sec. 3,
Eq. content_transform and Prop. 1; App. C.1 content-path fusion, App. C.2
RoPE-path fusion). Test infrastructure: used by tests/ only.

Content path. The cached latent is c = u Gamma with u = RMSNorm(x) (weightless)
and Gamma the normalisation scale. With an orthogonal R_C and a positive
diagonal S_C the cache stores z = u R_C S_C instead, and every consumer W_b of
the latent becomes W_b' = S_C^{-1} R_C^T Gamma W_b, so that z W_b' = c W_b. For
the absorbed decode the consumers are the key side of the content score and
the value/output map:

    Qbar c^T = (Qbar Gamma R_C S_C^{-1}) z^T      (query compensated)
    A c      = (A z) S_C^{-1} R_C^T Gamma         (output mapped back)

RoPE path (Prop. 1). R_P = blockdiag(R_i), R_i in SO(2) on each RoPE frequency
pair, S_P = blockdiag(s_i I_2): Q_P' = Q_P R_P S_P^{-1}, K_P' = K_P R_P S_P keep
Q_P K_P^T, and both commute with the positional rotation when R_P uses the same
pair layout as RoPE, so they can be applied before RoPE. The pair layout here is
the half-split one of the synthetic inputs: pair i = channels (i, i + 32),
inverse frequency theta^(-2i/64).
"""
from __future__ import annotations

import numpy as np

D_R = 64
HALF = D_R // 2


def cayley(a: np.ndarray) -> np.ndarray:
    """Orthogonal matrix (I - A)^{-1} (I + A) of the skew part A of a (the Cayley
    map the paper uses to parameterise content rotations)."""
    a = np.asarray(a, np.float64)
    skew = 0.5 * (a - a.T)
    eye = np.eye(a.shape[0])
    return np.linalg.solve(eye - skew, eye + skew)


def rmsnorm(x: np.ndarray, eps: float = 0.0) -> np.ndarray:
    """Weightless RMSNorm over the last axis."""
    x = np.asarray(x, np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def content_cache(u: np.ndarray, r_c: np.ndarray, s_c: np.ndarray) -> np.ndarray:
    """z = u R_C S_C for latent rows u [n, 512]."""
    return (np.asarray(u, np.float64) @ r_c) * np.asarray(s_c, np.float64)[None, :]


def consumer(w_b: np.ndarray, gamma: np.ndarray, r_c: np.ndarray, s_c: np.ndarray) -> np.ndarray:
    """W_b' = S_C^{-1} R_C^T Gamma W_b."""
    return (r_c.T @ (np.asarray(gamma, np.float64)[:, None] * w_b)) / np.asarray(s_c, np.float64)[:, None]


def content_query(q_bar: np.ndarray, gamma: np.ndarray, r_c: np.ndarray, s_c: np.ndarray) -> np.ndarray:
    """Qbar' = Qbar Gamma R_C S_C^{-1} (rows of absorbed content queries)."""
    return ((np.asarray(q_bar, np.float64) * gamma) @ r_c) / np.asarray(s_c, np.float64)


def content_output(out_z: np.ndarray, gamma: np.ndarray, r_c: np.ndarray, s_c: np.ndarray) -> np.ndarray:
    """A c from A z: (A z) S_C^{-1} R_C^T Gamma."""
    return ((np.asarray(out_z, np.float64) / s_c) @ r_c.T) * gamma


def pair_rotation(angles: np.ndarray, layout: str = "half") -> np.ndarray:
    """R_P [64, 64] rotating pair i by angles[i]. layout "half": pair i is
    channels (i, i + 32); "adjacent": channels (2i, 2i + 1)."""
    r = np.zeros((D_R, D_R))
    for i, th in enumerate(np.asarray(angles, np.float64)):
        a, b = (i, i + HALF) if layout == "half" else (2 * i, 2 * i + 1)
        c, s = np.cos(th), np.sin(th)
        # row-vector convention: [x_a, x_b] @ [[c, s], [-s, c]] rotates the pair by th
        r[a, a], r[a, b], r[b, a], r[b, b] = c, s, -s, c
    return r


def pair_scale(scales: np.ndarray, layout: str = "half") -> np.ndarray:
    """Diagonal of S_P: s_i on both channels of pair i."""
    d = np.zeros(D_R)
    for i, v in enumerate(np.asarray(scales, np.float64)):
        a, b = (i, i + HALF) if layout == "half" else (2 * i, 2 * i + 1)
        d[a] = d[b] = v
    return d


def rope(x: np.ndarray, positions, theta: float = 10000.0) -> np.ndarray:
    """Half-split RoPE of rows x [n, 64] at the given positions (pair i =
    (i, i + 32) rotated by pos * theta^(-2i/64)), as the synthetic keys use."""
    x = np.asarray(x, np.float64)
    pos = np.asarray(positions, np.float64)[:, None]
    inv = theta ** (-2.0 * np.arange(HALF) / D_R)
    ang = pos * inv[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[:, :HALF], x[:, HALF:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=1)


def rope_key(k_pre: np.ndarray, positions, r_p: np.ndarray, s_p: np.ndarray) -> np.ndarray:
    """K_P' = RoPE(k_pre R_P S_P): the transformation fused before RoPE."""
    return rope((np.asarray(k_pre, np.float64) @ r_p) * s_p, positions)


def rope_query(q_pre: np.ndarray, positions, r_p: np.ndarray, s_p: np.ndarray) -> np.ndarray:
    """Q_P' = RoPE(q_pre R_P S_P^{-1})."""
    return rope((np.asarray(q_pre, np.float64) @ r_p) / s_p, positions)
