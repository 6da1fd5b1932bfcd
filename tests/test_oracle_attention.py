"""Pins of the oracle attention, merge and storage against closed forms, a library
routine, brute force and the paper's Proposition 2."""
import math

import numpy as np
import pytest
import torch

from oracle import attention as A
from oracle import storage as St

TAU = 1.0 / math.sqrt(192.0)


def _rand(rng, H, n, scale_c=1.0):
    ql = rng.standard_normal((H, 512)) / math.sqrt(512)
    qp = rng.standard_normal((H, 64)) / 8.0
    C = rng.standard_normal((n, 512)) * scale_c
    K = rng.standard_normal((n, 64))
    return ql, qp, C, K


def test_single_token_returns_its_latent():
    rng = np.random.default_rng(0)
    ql, qp, C, K = _rand(rng, 4, 1)
    out, lse = A.attend(ql, qp, C, K, TAU)
    assert np.array_equal(out, np.repeat(C, 4, axis=0))
    s0 = TAU * (ql @ C[0] + qp @ K[0])
    assert np.allclose(lse, s0, rtol=0, atol=1e-14)


def test_equal_scores_give_mean_of_values():
    # With zero queries every score is 0, so the weights are uniform.
    rng = np.random.default_rng(1)
    _, _, C, K = _rand(rng, 2, 37)
    out, lse = A.attend(np.zeros((2, 512)), np.zeros((2, 64)), C, K, TAU)
    assert np.allclose(out, C.mean(0)[None, :], atol=1e-14)
    assert np.allclose(lse, math.log(37), atol=1e-14)
    # Same with equal RoPE keys and zero content query: q_pe . k is the same for all t.
    Keq = np.repeat(K[:1], 37, axis=0)
    out2, _ = A.attend(np.zeros((2, 512)), rng.standard_normal((2, 64)), C, Keq, TAU)
    assert np.allclose(out2, C.mean(0)[None, :], atol=1e-13)


def test_two_tokens_sigmoid_closed_form():
    # Tokens c_0 = 0 and c_1 = b e_0, query a e_0: S = (0, tau a b), so the weight on
    # token 1 is the logistic function of tau a b and out[0] = b * sigma(tau a b).
    a, b = 3.0, 2.5
    q = np.zeros((1, 512)); q[0, 0] = a
    C = np.zeros((2, 512)); C[1, 0] = b
    K = np.zeros((2, 64))
    out, lse = A.attend(q, np.zeros((1, 64)), C, K, TAU)
    w1 = 1.0 / (1.0 + math.exp(-TAU * a * b))
    assert out[0, 0] == pytest.approx(b * w1, rel=1e-14)
    assert lse[0] == pytest.approx(math.log(1.0 + math.exp(TAU * a * b)), rel=1e-14)
    # The RoPE path enters the scores the same way (q_pe = a e_0, k_1 = b e_0).
    qp = np.zeros((1, 64)); qp[0, 0] = a
    K2 = np.zeros((2, 64)); K2[1, 0] = b
    C2 = np.zeros((2, 512)); C2[1, 7] = 1.0
    out2, _ = A.attend(np.zeros((1, 512)), qp, C2, K2, TAU)
    assert out2[0, 7] == pytest.approx(w1, rel=1e-14)


def test_matches_library_sdpa():
    # Absorbed MLA decode is ordinary attention with key [C, K_P] (576 wide),
    # value C and scale tau; torch's reference SDPA in fp64 must agree.
    rng = np.random.default_rng(2)
    for H, n in [(16, 300), (3, 5), (128, 70)]:
        ql, qp, C, K = _rand(rng, H, n, scale_c=3.0)
        out, lse = A.attend(ql, qp, C, K, TAU)
        q = torch.tensor(np.concatenate([ql, qp], 1))[:, None, :]
        k = torch.tensor(np.concatenate([C, K], 1))[None].expand(H, n, 576)
        v = torch.tensor(C)[None].expand(H, n, 512)
        ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, scale=TAU)[:, 0, :].numpy()
        assert np.max(np.abs(out - ref)) < 1e-12
        S = (q @ k.transpose(1, 2) * TAU)[:, 0, :]
        assert np.allclose(lse, torch.logsumexp(S, dim=1).numpy(), atol=1e-12)


def test_brute_force_tiny():
    rng = np.random.default_rng(5)
    for H, n in [(1, 1), (2, 3), (2, 4)]:
        ql, qp, C, K = _rand(rng, H, n, scale_c=4.0)
        out, lse = A.attend(ql, qp, C, K, TAU)
        for h in range(H):
            s = []
            for t in range(n):
                acc = 0.0
                for c in range(512):
                    acc += ql[h, c] * C[t, c]
                for r in range(64):
                    acc += qp[h, r] * K[t, r]
                s.append(TAU * acc)
            mx = max(s)
            w = [math.exp(v - mx) for v in s]
            den = sum(w)
            for c in range(0, 512, 37):
                assert out[h, c] == pytest.approx(sum(w[t] * C[t, c] for t in range(n)) / den, rel=1e-12, abs=1e-13)
            assert lse[h] == pytest.approx(mx + math.log(den), rel=1e-13)


def test_softmax_rows_sum_to_one():
    rng = np.random.default_rng(6)
    ql, qp, C, K = _rand(rng, 8, 500, scale_c=20.0)
    P = A.softmax_rows(A.scores(ql, qp, C, K, TAU))
    assert np.all(np.abs(P.sum(1) - 1.0) <= 1e-12)


def test_merge_equals_unsplit():
    rng = np.random.default_rng(7)
    ql, qp, C, K = _rand(rng, 6, 1000, scale_c=10.0)
    full, lse = A.attend(ql, qp, C, K, TAU)
    for _ in range(5):
        cuts = np.sort(rng.choice(np.arange(1, 1000), size=rng.integers(1, 8), replace=False))
        parts = [A.partial(ql, qp, C[a:b], K[a:b], TAU) for a, b in zip([0, *cuts], [*cuts, 1000])]
        rng.shuffle(parts)
        merged, mlse = A.merge(parts)
        assert np.max(np.abs(merged - full)) <= 1e-12
        assert np.max(np.abs(mlse - lse)) <= 1e-12


def test_positional_qk_bound_prop2():
    # Prop. 2 with B_h = I and exact content: per head,
    # ||out(K_hat) - out(K)|| <= tau/2 * ||q_pe (K_hat - K)^T|| * ||C||_2.
    rng = np.random.default_rng(8)
    for trial in range(20):
        H, n = 4, 200
        ql, qp, C, K = _rand(rng, H, n, scale_c=2.0)
        Kh = K + rng.standard_normal(K.shape) * 10 ** rng.uniform(-3, 0.5)
        o1, _ = A.attend(ql, qp, C, K, TAU)
        o2, _ = A.attend(ql, qp, C, Kh, TAU)
        spec = np.linalg.norm(C, 2)
        for h in range(H):
            dz = qp[h] @ (Kh - K).T
            assert np.linalg.norm(o2[h] - o1[h]) <= TAU / 2 * np.linalg.norm(dz) * spec * (1 + 1e-12)


def _golden():
    import os
    vals = {}
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_storage.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                k, v = line.split("=")
                vals[k.strip()] = float(v)
    return vals


def test_storage_closed_form_matches_paper():
    g = _golden()
    assert St.PAPER_C4R4_PAGE == g["c4r4_page_bytes"] and St.PAPER_C4R4_PAGE / 64 == g["c4r4_bytes_per_token"]
    assert St.PAPER_PROTECTION == g["protection_bytes"]
    assert St.PAPER_REVERSE_MAP == g["reverse_map_bytes_per_page"]
    assert St.BF16_PAGE == g["bf16_page_bytes"]
    assert round(St.paper_ratio(4096), 2) == g["ratio_4k"]
    assert round(St.paper_ratio(131072), 2) == g["ratio_128k"]
    # this library's INT4 block: 20736 B per 64 tokens -> 3.556x against BF16 at 128K
    assert St.packed_bytes(131072, 20736) == 42467328
    assert St.bf16_bytes(131072) == 150994944
