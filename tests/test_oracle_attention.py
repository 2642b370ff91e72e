"""Pins for oracle.attention / oracle.cache against things other than the
oracle itself: scalar brute force, torch's float64 SDPA, scipy's logsumexp /
softmax, closed forms, and invariants of the softmax-attention definition
(Sec. 4.1: the drafter's cross-attention is plain self-attention over the
cache; Alg. 2 fixes which rows each draft / verify query sees)."""

import math

import numpy as np
import pytest
import scipy.special
import torch

from oracle import attention as A
from oracle import cache as C


def brute(q, K, V, scale):
    """Scalar pure-Python softmax attention (math.exp / math.fsum)."""
    s = [scale * math.fsum(float(q[d]) * float(K[j, d]) for d in range(len(q)))
         for j in range(K.shape[0])]
    m = max(s)
    e = [math.exp(x - m) for x in s]
    l = math.fsum(e)
    o = [math.fsum(e[j] / l * float(V[j, d]) for j in range(len(e))) for d in range(V.shape[1])]
    return np.array(o), m + math.log(l)


@pytest.mark.parametrize("seed", range(6))
def test_attend_matches_scalar_brute_force(seed):
    g = np.random.default_rng(seed)
    D = int(g.integers(1, 9))
    n = int(g.integers(1, 21))
    q, K, V = g.standard_normal(D), g.standard_normal((n, D)), g.standard_normal((n, D))
    scale = float(g.uniform(0.1, 2.0))
    o, lse, p = A.attend(q, K, V, scale)
    ob, lb = brute(q, K, V, scale)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    assert abs(lse - lb) < 1e-12
    assert abs(p.sum() - 1.0) < 1e-12


@pytest.mark.parametrize("seed", range(4))
def test_verify_matches_torch_sdpa_float64(seed):
    """Causal-among-new-rows verify attention with GQA vs torch SDPA (fp64)."""
    g = np.random.default_rng(100 + seed)
    Hkv, G, D = 2, 3, 8
    Hq = Hkv * G
    L = int(g.integers(0, 12))
    n_q = int(g.integers(1, 6))
    q = g.standard_normal((n_q, Hq, D))
    k = g.standard_normal((L + n_q, Hkv, D))
    v = g.standard_normal((L + n_q, Hkv, D))
    scale = 1 / math.sqrt(D)
    o, lse = A.verify_attention_seq(q, k, v, L, scale)

    tq = torch.from_numpy(q).permute(1, 0, 2)                 # [Hq, n_q, D]
    tk = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, dim=0)
    tv = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, dim=0)
    mask = torch.zeros(n_q, L + n_q, dtype=torch.bool)
    for j in range(n_q):
        mask[j, :L + j + 1] = True
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, attn_mask=mask, scale=scale)
    np.testing.assert_allclose(o, ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)
    # lse against scipy on explicitly built score rows
    for j in range(n_q):
        for h in range(Hq):
            s = scale * (k[:L + j + 1, h // G] @ q[j, h])
            assert abs(lse[j, h] - scipy.special.logsumexp(s)) < 1e-12


@pytest.mark.parametrize("seed", range(3))
def test_draft_matches_torch_sdpa_float64(seed):
    g = np.random.default_rng(200 + seed)
    Hkv, G, D = 2, 4, 16
    Hq = Hkv * G
    L, i = int(g.integers(0, 30)), int(g.integers(1, 5))
    q = g.standard_normal((Hq, D))
    ck, cv = g.standard_normal((L, Hkv, D)), g.standard_normal((L, Hkv, D))
    dk, dv = g.standard_normal((i, Hkv, D)), g.standard_normal((i, Hkv, D))
    o, lse = A.draft_attention_seq(q, ck, cv, dk, dv, 0.25)
    K = np.concatenate([ck, dk]).transpose(1, 0, 2).repeat(G, axis=0)
    V = np.concatenate([cv, dv]).transpose(1, 0, 2).repeat(G, axis=0)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[:, None], torch.from_numpy(K), torch.from_numpy(V), scale=0.25)
    np.testing.assert_allclose(o, ref[:, 0].numpy(), rtol=0, atol=1e-12)


def test_closed_form_single_row():
    g = np.random.default_rng(1)
    q, K, V = g.standard_normal(8), g.standard_normal((1, 8)), g.standard_normal((1, 8))
    o, lse, _ = A.attend(q, K, V, 0.5)
    np.testing.assert_allclose(o, V[0], rtol=0, atol=1e-15)
    assert abs(lse - 0.5 * float(K[0] @ q)) < 1e-14


def test_closed_form_identical_keys():
    g = np.random.default_rng(2)
    n = 7
    q = g.standard_normal(8)
    K = np.tile(g.standard_normal(8), (n, 1))
    V = g.standard_normal((n, 8))
    o, lse, _ = A.attend(q, K, V, 0.3)
    np.testing.assert_allclose(o, V.mean(axis=0), rtol=0, atol=1e-14)
    assert abs(lse - (0.3 * float(K[0] @ q) + math.log(n))) < 1e-13


def test_closed_form_one_hot_values_give_probabilities():
    g = np.random.default_rng(3)
    n = 6
    q, K = g.standard_normal(5), g.standard_normal((n, 5))
    o, _, _ = A.attend(q, K, np.eye(n), 0.7)
    np.testing.assert_allclose(o, scipy.special.softmax(0.7 * (K @ q)), rtol=0, atol=1e-15)


def test_closed_form_two_rows_is_a_sigmoid():
    """Scores s0 = scale*|q|^2 (key = q) and s1 = 0 (key orthogonal): the
    weight of row 0 is 1 / (1 + exp(-s0)); catches a dropped scale."""
    q = np.array([1.0, 2.0, 0.0, 0.0])
    K = np.array([q, [0.0, 0.0, 3.0, 1.0]])
    V = np.array([[1.0, 0, 0, 0], [0.0, 1, 0, 0]])
    scale = 0.5
    o, _, _ = A.attend(q, K, V, scale)
    w0 = 1.0 / (1.0 + math.exp(-scale * 5.0))
    np.testing.assert_allclose(o, [w0, 1 - w0, 0, 0], rtol=0, atol=1e-15)


def test_gqa_group_mapping():
    """Query head h reads KV head h // G: with V of KV head g constant g, the
    output of head h is exactly h // G (catches h % Hkv or other mappings)."""
    Hkv, G, D, L, i = 4, 3, 8, 9, 2
    g = np.random.default_rng(4)
    ck = g.standard_normal((L, Hkv, D))
    dk = g.standard_normal((i, Hkv, D))
    cv = np.broadcast_to(np.arange(Hkv, dtype=float)[None, :, None], (L, Hkv, D)).copy()
    dv = np.broadcast_to(np.arange(Hkv, dtype=float)[None, :, None], (i, Hkv, D)).copy()
    o, _ = A.draft_attention_seq(g.standard_normal((Hkv * G, D)), ck, cv, dk, dv, 0.2)
    for h in range(Hkv * G):
        np.testing.assert_allclose(o[h], h // G, rtol=0, atol=1e-14)


def test_verify_query_is_independent_causal_decode():
    """Verify query j equals one decode step over rows 0..L+j; the last query
    equals draft attention over the same rows (Alg. 2 masks)."""
    g = np.random.default_rng(5)
    Hkv, G, D, L, n_q = 2, 2, 8, 11, 4
    q = g.standard_normal((n_q, Hkv * G, D))
    k = g.standard_normal((L + n_q, Hkv, D))
    v = g.standard_normal((L + n_q, Hkv, D))
    o, lse = A.verify_attention_seq(q, k, v, L, 0.35)
    for j in range(n_q):
        for h in range(Hkv * G):
            oj, lj, _ = A.attend(q[j, h], k[:L + j + 1, h // G], v[:L + j + 1, h // G], 0.35)
            np.testing.assert_allclose(o[j, h], oj, rtol=0, atol=1e-13)
            assert abs(lse[j, h] - lj) < 1e-13
    od, _ = A.draft_attention_seq(q[n_q - 1], k[:L], v[:L], k[L:], v[L:], 0.35)
    np.testing.assert_allclose(o[n_q - 1], od, rtol=0, atol=1e-13)


def test_k0_verify_is_single_token_decode():
    """k = 0: one verify query over the L committed rows plus its own row is
    an ordinary autoregressive decode step (draft with one row, its own)."""
    g = np.random.default_rng(6)
    Hkv, G, D, L = 2, 4, 16, 20
    q = g.standard_normal((1, Hkv * G, D))
    k = g.standard_normal((L + 1, Hkv, D))
    v = g.standard_normal((L + 1, Hkv, D))
    o, lse = A.verify_attention_seq(q, k, v, L, 0.25)
    od, ld = A.draft_attention_seq(q[0], k[:L], v[:L], k[L:], v[L:], 0.25)
    np.testing.assert_allclose(o[0], od, rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse[0], ld, rtol=0, atol=1e-14)


@pytest.mark.parametrize("seed", range(4))
def test_split_merge_equals_unsplit(seed):
    g = np.random.default_rng(300 + seed)
    n, D = 50, 8
    q, K, V = g.standard_normal(D), 3 * g.standard_normal((n, D)), g.standard_normal((n, D))
    o, lse, _ = A.attend(q, K, V, 0.4)
    cuts = np.sort(g.choice(np.arange(1, n), size=int(g.integers(1, 6)), replace=False))
    bounds = [0, *cuts.tolist(), n]
    parts = [A.attend(q, K[a:b], V[a:b], 0.4) for a, b in zip(bounds[:-1], bounds[1:])]
    om, lm = A.merge_partials(np.stack([p[0] for p in parts]), np.array([p[1] for p in parts]))
    np.testing.assert_allclose(om, o, rtol=0, atol=1e-12)
    assert abs(lm - lse) < 1e-12


def test_masked_rows_never_leak_nan():
    g = np.random.default_rng(7)
    Q, K, V = g.standard_normal((3, 4)), g.standard_normal((5, 4)), g.standard_normal((5, 4))
    vis = np.array([[1, 1, 0, 0, 0], [1, 1, 1, 0, 0], [1, 1, 1, 1, 0]], dtype=bool)
    O, lse, _ = A.masked_attention(Q, K, V, vis, 0.5)
    K2, V2 = K.copy(), V.copy()
    K2[4], V2[4] = np.nan, np.nan
    O2, lse2, _ = A.masked_attention(Q, K2, V2, vis, 0.5)
    np.testing.assert_array_equal(O, O2)
    np.testing.assert_array_equal(lse, lse2)


def test_paged_gather_is_page_order_invariant():
    """The same logical rows stored in two page orders give bit-identical
    attention; slot() agrees with the page/offset definition."""
    g = np.random.default_rng(8)
    P, Hkv, D, n_pages, n = 4, 2, 8, 6, 21
    rows = g.standard_normal((n, Hkv, D))
    q = g.standard_normal((2, 2 * Hkv, D))
    outs = []
    for perm in (np.arange(n_pages), g.permutation(n_pages)):
        cache = np.full((n_pages, Hkv, P, D), np.nan)
        C.write_rows(cache, perm, 0, rows)
        np.testing.assert_array_equal(C.gather_rows(cache, perm, n), rows)
        for pos in range(n):
            s = C.slot(perm, pos, P)
            assert s == perm[pos // P] * P + pos % P
            np.testing.assert_array_equal(cache[s // P, :, s % P], rows[pos])
        kv = C.gather_rows(cache, perm, n)
        outs.append(A.verify_attention_seq(q, kv, kv, n - 2, 0.3))
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
    np.testing.assert_array_equal(outs[0][1], outs[1][1])
