"""Pins of the dynamic-drafting oracle (Sec. D.1): the sibling-count rule at
and around its boundaries, the top tokens against a scalar brute force and a
library softmax, probabilities that sum with the rest of the vocabulary to 1,
the tie rule, and the stop rule."""

import math

import numpy as np
import pytest
import scipy.special

from oracle import drafting as OD


def test_sibling_count_rule_by_hand():
    p0 = [1.0, 0.96, 0.95, 0.9, 0.8, 0.7, 0.5, 0.2, 0.0]
    assert OD.sibling_count(p0).tolist() == [1, 1, 3, 3, 5, 5, 10, 10, 10]


@pytest.mark.parametrize("seed", range(4))
def test_top_tokens_match_scalar_brute_force(seed):
    g = np.random.default_rng(seed)
    B, V, d = 3, 37, 6
    h = g.standard_normal((B, d))
    W = g.standard_normal((V, d)) * (1 + seed)
    ids, probs, p0, k, stop, lse = OD.draft_head(h, W, 0.7, topk=5)
    for b in range(B):
        z = [math.fsum(h[b, i] * W[v, i] for i in range(d)) for v in range(V)]
        m = max(z)
        zs = math.fsum(math.exp(x - m) for x in z)
        p = [math.exp(x - m) / zs for x in z]
        order = sorted(range(V), key=lambda v: (-z[v], v))[:5]
        assert ids[b].tolist() == order
        np.testing.assert_allclose(probs[b], [p[v] for v in order], rtol=0, atol=1e-14)
        assert abs(lse[b] - (m + math.log(zs))) < 1e-12
        assert k[b] == (1 if p[order[0]] > 0.95 else 3 if p[order[0]] > 0.8
                        else 5 if p[order[0]] > 0.5 else 10)
        assert stop[b] == int(p[order[0]] <= 0.7)


def test_against_library_softmax_and_normalisation():
    g = np.random.default_rng(9)
    B, V, d = 5, 500, 16
    h = g.standard_normal((B, d))
    W = g.standard_normal((V, d))
    ids, probs, p0, k, stop, lse = OD.draft_head(h, W, 0.7)
    p = scipy.special.softmax(h @ W.T, axis=1)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(h @ W.T, axis=1), rtol=0, atol=1e-12)
    for b in range(B):
        np.testing.assert_allclose(probs[b], np.sort(p[b])[::-1][:OD.TOPK], rtol=0, atol=1e-14)
        rest = np.delete(p[b], ids[b]).sum()
        assert abs(probs[b].sum() + rest - 1.0) < 1e-12
        assert (np.diff(probs[b]) <= 0).all()


def test_confident_and_flat_distributions():
    V, d = 50, 4
    W = np.zeros((V, d))
    W[7, 0] = 1.0
    h = np.array([[40.0, 0, 0, 0], [0.0, 0, 0, 0]])
    ids, probs, p0, k, stop, _ = OD.draft_head(h, W, 0.7)
    # a peaked row: one token, no stop
    assert ids[0, 0] == 7 and p0[0] > 0.999 and k[0] == 1 and stop[0] == 0
    # a flat row: all logits equal, ties go to the lowest ids, p0 = 1/V
    assert ids[1].tolist() == list(range(10))
    assert abs(p0[1] - 1.0 / V) < 1e-15 and k[1] == 10 and stop[1] == 1
