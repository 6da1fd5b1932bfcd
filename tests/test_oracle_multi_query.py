"""Pins of the multi-token decode oracle (Eq. mla_compact with the additive causal
mask): the mask against its closed form, one query row against the pinned
single-token oracle on the matching prefix, T = 1 against that oracle, scipy's
softmax / logsumexp on brute-force masked scores, hand-worked tiny cases, rows
with no admissible key, and the App. C.5 merge of masked partials over random
key partitions (including parts that are empty for some rows)."""
import math

import numpy as np
import pytest
from scipy.special import logsumexp, softmax

from oracle import attention as A
from oracle import multi_query as M

TAU = 1.0 / math.sqrt(192.0)


def _inputs(rng, L, T, H):
    C = rng.standard_normal((L, 512)) * 2.0
    K = rng.standard_normal((L, 64))
    ql = rng.standard_normal((T, H, 512)) / math.sqrt(512)
    qp = rng.standard_normal((T, H, 64)) / 8
    return ql, qp, C, K


@pytest.mark.parametrize("L", range(0, 12))
@pytest.mark.parametrize("T", range(1, 6))
def test_mask_closed_form(L, T):
    m = M.causal_mask(L, T)
    assert m.shape == (T, L)
    for t in range(T):
        n = max(0, L - T + t + 1)                       # admissible keys of row t
        assert np.all(m[t, :n] == 0.0) and np.all(np.isneginf(m[t, n:]))


@pytest.mark.parametrize("L", [1, 2, 7, 130, 300])
def test_single_query_is_the_decode_oracle(L):
    rng = np.random.default_rng(L)
    ql, qp, C, K = _inputs(rng, L, 1, 3)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    o1, l1 = A.attend(ql[0], qp[0], C, K, TAU)
    assert np.allclose(out[0], o1, atol=1e-12) and np.allclose(lse[0], l1, atol=1e-12)


@pytest.mark.parametrize("L,T", [(2, 2), (5, 3), (130, 4), (300, 2), (129, 3), (64, 8)])
def test_each_row_is_a_decode_over_its_prefix(L, T):
    rng = np.random.default_rng(100 * T + L)
    ql, qp, C, K = _inputs(rng, L, T, 4)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    for t in range(T):
        n = L - T + t + 1
        o1, l1 = A.attend(ql[t], qp[t], C[:n], K[:n], TAU)
        assert np.allclose(out[t], o1, atol=1e-12) and np.allclose(lse[t], l1, atol=1e-12)


def test_against_scipy_on_brute_force_scores():
    rng = np.random.default_rng(7)
    L, T, H = 9, 4, 2
    ql, qp, C, K = _inputs(rng, L, T, H)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    for t in range(T):
        for h in range(H):
            s = np.array([TAU * (ql[t, h] @ C[p] + qp[t, h] @ K[p]) if p <= L - T + t else -np.inf
                          for p in range(L)])
            w = softmax(s)
            assert np.allclose(out[t, h], w @ C, atol=1e-12)
            assert np.isclose(lse[t, h], logsumexp(s), atol=1e-12)


def test_hand_worked_two_by_two():
    # L = 2, T = 2: row 0 sees key 0 only (out = C[0], lse = its score); row 1 both.
    rng = np.random.default_rng(3)
    ql, qp, C, K = _inputs(rng, 2, 2, 1)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    s00 = TAU * (ql[0, 0] @ C[0] + qp[0, 0] @ K[0])
    assert np.array_equal(out[0, 0], C[0]) and np.isclose(lse[0, 0], s00, atol=1e-14)
    s10 = TAU * (ql[1, 0] @ C[0] + qp[1, 0] @ K[0])
    s11 = TAU * (ql[1, 0] @ C[1] + qp[1, 0] @ K[1])
    w1 = 1.0 / (1.0 + math.exp(s10 - s11))            # two-key logistic closed form
    assert np.allclose(out[1, 0], (1 - w1) * C[0] + w1 * C[1], atol=1e-12)


def test_rows_without_keys():
    # L = 1, T = 3: rows 0 and 1 would sit before position 0.
    rng = np.random.default_rng(5)
    ql, qp, C, K = _inputs(rng, 1, 3, 2)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    assert np.all(out[:2] == 0) and np.all(np.isneginf(lse[:2]))
    assert np.allclose(out[2], np.broadcast_to(C[0], (2, 512)), atol=1e-12)
    out0, lse0 = M.attend_multi(ql, qp, C[:0], K[:0], TAU)
    assert np.all(out0 == 0) and np.all(np.isneginf(lse0))


@pytest.mark.parametrize("L,T", [(130, 4), (257, 3), (5, 5)])
def test_merge_of_masked_partials(L, T):
    rng = np.random.default_rng(L + 17 * T)
    ql, qp, C, K = _inputs(rng, L, T, 3)
    out, lse = M.attend_multi(ql, qp, C, K, TAU)
    rest = np.arange(L - 1)
    for trial in range(4):
        # contiguous pieces as the kernel's splits make them, or a shuffled partition,
        # of keys 0..L-2; key L-1 alone forms a part that is empty for rows t < T-1
        if trial < 3:
            cuts = np.sort(rng.choice(np.arange(1, L - 1), size=min(trial + 1, L - 2), replace=False))
            pieces = np.split(rest, cuts)
        else:
            perm = rng.permutation(rest)
            pieces = [np.sort(perm[i::3]) for i in range(3)]
        pieces = [p for p in pieces if len(p)] + [np.array([L - 1])]
        parts = [M.partial_multi(ql, qp, C[p], K[p], TAU, L, p) for p in pieces]
        assert np.all(np.isneginf(parts[-1][0][:T - 1]))   # the lone last key is masked for them
        o2, l2 = M.merge_multi(parts)
        assert np.allclose(o2, out, atol=1e-12) and np.allclose(l2, lse, atol=1e-12)
