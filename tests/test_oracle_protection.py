"""Pins of the sink4/local128 protection oracle: the protected set against
closed forms and a hand-worked case, the buffer size against the paper's
figure, the writer's ring against two independent write orders, and protected
attention against a library softmax (all tokens protected) and against the
App. C.5 merge of the protected and packed regions."""
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import logsumexp, softmax

from oracle import attention as A
from oracle import protection as Pr

TAU = 1.0 / math.sqrt(192.0)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_storage.txt")


def _golden():
    d = {}
    for line in open(GOLDEN):
        line = line.split("#")[0].strip()
        if line:
            k, v = (t.strip() for t in line.split("="))
            d[k] = float(v)
    return d


@pytest.mark.parametrize("L", list(range(0, 300)) + [4096, 4097, 131072])
def test_protected_set_closed_forms(L):
    P = Pr.protected_positions(L)
    assert len(P) == min(L, 132)                      # 4 + 128 once the regions are disjoint
    assert len(np.unique(P)) == len(P)
    assert L == 0 or (P.min() == 0 and P.max() == L - 1)
    outside = np.setdiff1d(np.arange(L), P)
    if L > 132:
        assert np.array_equal(outside, np.arange(4, L - 128))  # one contiguous packed interval
    else:
        assert outside.size == 0


def test_protected_set_hand_worked():
    assert list(Pr.protected_positions(0)) == []
    assert list(Pr.protected_positions(3)) == [0, 1, 2]
    assert list(Pr.protected_positions(5)) == [0, 1, 2, 3, 4]
    # L = 133: the recent window is 5..132, the sinks 0..3, so only position 4 is packed.
    assert np.array_equal(np.setdiff1d(np.arange(133), Pr.protected_positions(133)), [4])


def test_buffer_size_is_the_papers():
    assert Pr.ROWS * Pr.ROW_VALUES * 2 == int(_golden()["protection_bytes"])


def _bf16(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).float().numpy()


def _tokens(rng, L):
    return _bf16(rng.standard_normal((L, 512))), _bf16(rng.standard_normal((L, 64)))


@pytest.mark.parametrize("L", [1, 3, 4, 5, 127, 128, 129, 131, 132, 133, 200, 300])
def test_writer_ring_two_orders(L):
    rng = np.random.default_rng(L)
    lat, kpe = _tokens(rng, L)
    # (a) one token per call, as in a decode loop (length after each call = p + 1)
    a = np.full((1, 132, 576), np.nan)
    for p in range(L):
        Pr.write_protection(a, lat[p:p + 1], kpe[p:p + 1], [0], [p], [p + 1])
    # (b) one bulk call with every position (length L), positions shuffled
    b = np.full((1, 132, 576), np.nan)
    order = rng.permutation(L)
    Pr.write_protection(b, lat[order], kpe[order], np.zeros(L, int), order, [L])
    for p in Pr.protected_positions(L):
        r = Pr.row_of(int(p), L)
        want = np.concatenate([lat[p], kpe[p]])
        assert np.array_equal(a[0, r], want) and np.array_equal(b[0, r], want)


@pytest.mark.parametrize("c_bits", [4, 2])
@pytest.mark.parametrize("L", [1, 7, 64, 128, 132])
def test_all_protected_is_exact_attention(c_bits, L):
    # Every token is protected: attention over the unquantised values, checked
    # against scipy's softmax / logsumexp.
    rng = np.random.default_rng(100 + L)
    lat, kpe = _tokens(rng, L)
    ql = rng.standard_normal((3, 512)) / math.sqrt(512)
    qp = rng.standard_normal((3, 64)) / 8
    out, lse = Pr.attend_protected(ql, qp, lat, kpe, c_bits, TAU)
    S = TAU * (ql @ lat.astype(np.float64).T + qp @ kpe.astype(np.float64).T)
    assert np.allclose(out, softmax(S, axis=1) @ lat.astype(np.float64), atol=1e-12)
    assert np.allclose(lse, logsumexp(S, axis=1), atol=1e-12)


@pytest.mark.parametrize("c_bits", [4, 2])
@pytest.mark.parametrize("L", [133, 140, 300, 700])
def test_protected_equals_merge_of_regions(c_bits, L):
    rng = np.random.default_rng(200 + L)
    lat, kpe = _tokens(rng, L)
    ql = rng.standard_normal((2, 512)) / math.sqrt(512)
    qp = rng.standard_normal((2, 64)) / 8
    out, lse = Pr.attend_protected(ql, qp, lat, kpe, c_bits, TAU)
    P = Pr.protected_positions(L)
    U = np.setdiff1d(np.arange(L), P)
    Cq, Kq = A.quantized_cache(lat, kpe, c_bits)
    parts = [A.partial(ql, qp, lat[P], kpe[P], TAU), A.partial(ql, qp, np.asarray(Cq)[U], np.asarray(Kq)[U], TAU)]
    o2, l2 = A.merge(parts)
    assert np.allclose(out, o2, atol=1e-12) and np.allclose(lse, l2, atol=1e-12)
    # and it differs from the unprotected answer (the protection is not a no-op)
    o3, _ = A.attend(ql, qp, Cq, Kq, TAU)
    assert np.max(np.abs(out - o3)) > 1e-6


@pytest.mark.parametrize("L", [5, 133, 400])
def test_buffer_path_equals_definition(L):
    rng = np.random.default_rng(300 + L)
    lat, kpe = _tokens(rng, L)
    ql = rng.standard_normal((2, 512)) / math.sqrt(512)
    qp = rng.standard_normal((2, 64)) / 8
    buf = np.zeros((1, 132, 576))
    Pr.write_protection(buf, lat, kpe, np.zeros(L, int), np.arange(L), [L])
    Cq, Kq = A.quantized_cache(lat, kpe, 4)
    o1, l1 = Pr.attend_from_buffer(ql, qp, Cq, Kq, buf[0], L, TAU)
    o2, l2 = Pr.attend_protected(ql, qp, lat, kpe, 4, TAU)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)
