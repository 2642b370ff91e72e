"""Pins of the block-causal training attention oracle (Sec. 4.2, "Training with
Block Attention"; Fig. 2), against things other than itself:
* the mask of Fig. 2 (n = 6, b = 2) worked by hand (tests/golden);
* the paper's 1-based boundary n' = floor((j - 2) / b) * b + 1 for every
  target j, restated from the text;
* a scalar pure-Python softmax (math.fsum) for single queries;
* PyTorch's scaled_dot_product_attention with an explicit boolean mask over
  the concatenated [dec; spec] rows (grouped heads);
* special cases: one block covering the sequence is plain causal attention
  over the spec rows (the oracle's verify formulation with no cache), and
  b = 1 gives dec rows [0, p) plus the query's own spec row."""

import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import attention as OAT
from oracle import block_attn as OB

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "block_mask_fig2_n6_b2.txt")


def test_mask_of_fig2_by_hand():
    dec, spec = OB.visibility(6, 2)
    rows = [l for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert len(rows) == 6
    for line in rows:
        p, d, s = [f.strip() for f in line.split(";")]
        p = int(p)
        want_d = [] if d == "-" else [int(x) for x in d.split()]
        want_s = [int(x) for x in s.split()]
        assert np.nonzero(dec[p])[0].tolist() == want_d
        assert np.nonzero(spec[p])[0].tolist() == want_s


@pytest.mark.parametrize("b", [1, 3, 10])
def test_block_start_matches_the_papers_one_based_boundary(b):
    # target token X_j (1-based) is predicted at 0-based position p = j - 2;
    # its context splits at n' = floor((j - 2) / b) * b + 1 (1-based), i.e.
    # the dec rows are the 1-based positions 1 .. n' - 1
    for j in range(2, 60):
        n1 = ((j - 2) // b) * b + 1
        p = j - 2
        assert OB.block_start(p, b) == n1 - 1


def test_single_query_against_scalar_loop():
    g = np.random.default_rng(1)
    n, Hq, Hkv, D, b = 9, 2, 1, 5, 4
    q = g.standard_normal((n, Hq, D))
    kd, vd, ks, vs = (g.standard_normal((n, Hkv, D)) for _ in range(4))
    o, lse = OB.block_causal_attention(q, kd, vd, ks, vs, b, 0.4)
    for p in (0, 3, 4, 6, 8):
        s0 = (p // b) * b
        rows = [(kd[k, 0], vd[k, 0]) for k in range(s0)] + [(ks[k, 0], vs[k, 0]) for k in range(s0, p + 1)]
        for h in range(Hq):
            sc = [0.4 * math.fsum(q[p, h, d] * kk[d] for d in range(D)) for kk, _ in rows]
            m = max(sc)
            w = [math.exp(x - m) for x in sc]
            z = math.fsum(w)
            ref = [math.fsum(w[i] * rows[i][1][d] for i in range(len(rows))) / z for d in range(D)]
            np.testing.assert_allclose(o[p, h], ref, rtol=0, atol=1e-12)
            assert abs(lse[p, h] - (m + math.log(z))) < 1e-12


@pytest.mark.parametrize("n,b,Hq,Hkv", [(23, 5, 8, 2), (16, 16, 4, 4), (40, 7, 4, 1)])
def test_against_torch_sdpa_with_explicit_mask(n, b, Hq, Hkv):
    g = np.random.default_rng(n + b)
    D = 16
    q = g.standard_normal((n, Hq, D))
    kd, vd, ks, vs = (g.standard_normal((n, Hkv, D)) for _ in range(4))
    o, _ = OB.block_causal_attention(q, kd, vd, ks, vs, b, 1 / math.sqrt(D))
    p = torch.arange(n)[:, None]
    k = torch.arange(n)[None, :]
    s = (p // b) * b
    mask = torch.cat([k < s, (k >= s) & (k <= p)], dim=1)          # [n, 2n]
    K = torch.from_numpy(np.concatenate([kd, ks], 0)).permute(1, 0, 2)
    V = torch.from_numpy(np.concatenate([vd, vs], 0)).permute(1, 0, 2)
    Q = torch.from_numpy(q).permute(1, 0, 2)
    ref = F.scaled_dot_product_attention(Q, K, V, attn_mask=mask, enable_gqa=True)
    np.testing.assert_allclose(o, ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)


def test_one_block_is_causal_attention_and_b1_sees_own_row():
    g = np.random.default_rng(3)
    n, Hq, Hkv, D = 12, 4, 2, 8
    q = g.standard_normal((n, Hq, D))
    kd, vd, ks, vs = (g.standard_normal((n, Hkv, D)) for _ in range(4))
    o, lse = OB.block_causal_attention(q, kd, vd, ks, vs, n, 0.3)
    o2, lse2 = OAT.verify_attention_seq(q, ks, vs, 0, 0.3)
    np.testing.assert_allclose(o, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse2, rtol=0, atol=1e-12)
    o1, _ = OB.block_causal_attention(q, kd, vd, ks, vs, 1, 0.3)
    for p in range(n):
        K = np.concatenate([kd[:p], ks[p:p + 1]], 0)
        V = np.concatenate([vd[:p], vs[p:p + 1]], 0)
        for h in range(Hq):
            ref, _, _ = OAT.attend(q[p, h], K[:, h // 2], V[:, h // 2], 0.3)
            np.testing.assert_allclose(o1[p, h], ref, rtol=0, atol=1e-12)
