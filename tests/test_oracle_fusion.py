"""Pins of the offline-fusion identities (Eq. content_transform, Prop. 1, App. C.1
and C.2): Cayley rotations are in SO(n); weightless RMSNorm is rotation
equivariant; a compensated consumer reproduces c W_b; Prop. 1's reciprocal
pair transform keeps Q_P K_P^T; the pair rotation commutes with RoPE in the
same pair layout and not in a different one; and the whole absorbed decode
over a fused cache, mapped back, equals the decode over the original cache
(the pinned single-token oracle on both sides)."""
import math

import numpy as np
import pytest

from oracle import attention as A
from oracle import fusion as F

TAU = 1.0 / math.sqrt(192.0)


def _transforms(rng, n=512):
    r_c = F.cayley(rng.standard_normal((n, n)) * 0.1)
    s_c = np.exp(np.clip(rng.standard_normal(n) * 0.5, -2, 2))    # log-space scales clipped to [-2, 2]
    ang = rng.uniform(-np.pi, np.pi, 32)
    s_p = np.exp(np.clip(rng.standard_normal(32) * 0.5, -2, 2))
    return r_c, s_c, F.pair_rotation(ang), F.pair_scale(s_p)


def test_cayley_is_a_rotation():
    rng = np.random.default_rng(0)
    for n in (2, 7, 64, 512):
        r = F.cayley(rng.standard_normal((n, n)))
        assert np.allclose(r @ r.T, np.eye(n), atol=1e-10)
        assert np.isclose(np.linalg.det(r), 1.0, atol=1e-8)
    assert np.allclose(F.cayley(np.zeros((5, 5))), np.eye(5))


def test_rmsnorm_is_rotation_equivariant():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((16, 512)) * 3
    r = F.cayley(rng.standard_normal((512, 512)) * 0.2)
    assert np.allclose(F.rmsnorm(x @ r), F.rmsnorm(x) @ r, atol=1e-12)
    # a non-orthogonal map breaks it (the identity is not vacuous)
    d = np.diag(np.linspace(0.5, 2.0, 512))
    assert np.max(np.abs(F.rmsnorm(x @ d) - F.rmsnorm(x) @ d)) > 1e-2


def test_compensated_consumer_reproduces_c_w():
    rng = np.random.default_rng(2)
    u = F.rmsnorm(rng.standard_normal((32, 512)))
    gamma = np.exp(rng.standard_normal(512) * 0.5)
    w_b = rng.standard_normal((512, 96))
    r_c, s_c, _, _ = _transforms(rng)
    z = F.content_cache(u, r_c, s_c)
    assert np.allclose(z @ F.consumer(w_b, gamma, r_c, s_c), (u * gamma) @ w_b, atol=1e-10)


def test_prop1_reciprocal_pair_transform_keeps_scores():
    rng = np.random.default_rng(3)
    q = rng.standard_normal((8, 64))
    k = rng.standard_normal((20, 64))
    _, _, r_p, s_p = _transforms(rng)
    assert np.allclose(((q @ r_p) / s_p) @ ((k @ r_p) * s_p).T, q @ k.T, atol=1e-12)
    assert np.allclose(r_p @ r_p.T, np.eye(64), atol=1e-14)


def test_pair_rotation_commutes_with_rope_only_in_its_layout():
    rng = np.random.default_rng(4)
    k = rng.standard_normal((50, 64))
    pos = rng.integers(0, 131072, 50)
    ang = rng.uniform(-np.pi, np.pi, 32)
    s = np.exp(rng.standard_normal(32) * 0.5)
    r_half, s_half = F.pair_rotation(ang, "half"), F.pair_scale(s, "half")
    assert np.allclose(F.rope((k @ r_half) * s_half, pos), (F.rope(k, pos) @ r_half) * s_half, atol=1e-10)
    # the same angles on adjacent pairs do not commute with half-split RoPE: a
    # pairing mistake is visible
    r_adj, s_adj = F.pair_rotation(ang, "adjacent"), F.pair_scale(s, "adjacent")
    assert np.max(np.abs(F.rope((k @ r_adj) * s_adj, pos) - (F.rope(k, pos) @ r_adj) * s_adj)) > 0.1


def test_positional_scores_survive_fusion_before_rope():
    rng = np.random.default_rng(5)
    q = rng.standard_normal((4, 64))
    k = rng.standard_normal((30, 64))
    pq = np.full(4, 1000)
    pk = np.arange(30) * 33
    _, _, r_p, s_p = _transforms(rng)
    fused = F.rope_query(q, pq, r_p, s_p) @ F.rope_key(k, pk, r_p, s_p).T
    assert np.allclose(fused, F.rope(q, pq) @ F.rope(k, pk).T, atol=1e-10)


@pytest.mark.parametrize("n", [1, 17, 300])
def test_decode_over_a_fused_cache_maps_back(n):
    rng = np.random.default_rng(100 + n)
    u = F.rmsnorm(rng.standard_normal((n, 512)))
    gamma = np.exp(rng.standard_normal(512) * 0.5)
    gamma[rng.permutation(512)[:4]] *= 8.0
    k_pre = rng.standard_normal((n, 64))
    pos = np.arange(n)
    q_bar = rng.standard_normal((6, 512)) / math.sqrt(512)
    q_pre = rng.standard_normal((6, 64)) / 8
    r_c, s_c, r_p, s_p = _transforms(rng)
    # original: c = u Gamma, K = RoPE(k_pre), query RoPE at position n - 1
    out, lse = A.attend(q_bar, F.rope(q_pre, np.full(6, n - 1)), u * gamma, F.rope(k_pre, pos), TAU)
    # fused: z, K', compensated queries; the output mapped back by S_C^{-1} R_C^T Gamma
    z = F.content_cache(u, r_c, s_c)
    kf = F.rope_key(k_pre, pos, r_p, s_p)
    qf = F.content_query(q_bar, gamma, r_c, s_c)
    qpf = F.rope_query(q_pre, np.full(6, n - 1), r_p, s_p)
    out_z, lse_z = A.attend(qf, qpf, z, kf, TAU)
    assert np.allclose(F.content_output(out_z, gamma, r_c, s_c), out, atol=1e-10)
    assert np.allclose(lse_z, lse, atol=1e-10)
