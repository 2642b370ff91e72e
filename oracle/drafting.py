"""Confidence-aware dynamic drafting (oracle; test infrastructure).

Sec. D.1 ("Confidence-Aware Dynamic Drafting") lets the decoder keep drafting
while its confidence stays above a threshold tau, and expands the node being
drafted into k sibling candidates chosen by the probability p0 of its top-1
token:

    k = 1 if p0 > 0.95,  3 if 0.8 < p0 <= 0.95,  5 if 0.5 < p0 <= 0.8,  else 10.

Per sequence and draft step this needs the drafter's output distribution: the
LM head over the vocabulary, p = softmax(W_out h), its top tokens and p0.

Readings used here:
* the k candidates are the k most probable tokens, in decreasing probability,
  ties to the lower token id;
* "continue as long as its confidence remains above" tau: drafting goes on
  after a step whose p0 > tau and stops after a step whose p0 <= tau; the
  candidates of that last step are still added to the tree (so that k = 5 and
  k = 10 can occur at all with tau = 0.7);
* logits are W_out h with no bias or temperature (greedy decoding).
"""

from __future__ import annotations

import numpy as np

TOPK = 10


def sibling_count(p0) -> np.ndarray:
    """The piecewise rule of Sec. D.1, elementwise."""
    p0 = np.asarray(p0, dtype=np.float64)
    return np.where(p0 > 0.95, 1, np.where(p0 > 0.8, 3, np.where(p0 > 0.5, 5, 10))).astype(np.int32)


def head_logits(h: np.ndarray, W: np.ndarray) -> np.ndarray:
    """h [B, d], W [V, d] (float64) -> logits [B, V]."""
    return h @ W.T


def draft_head(h: np.ndarray, W: np.ndarray, tau: float, topk: int = TOPK):
    """Returns (ids [B, topk] int32, probs [B, topk], p0 [B], k [B] int32,
    stop [B] int32, lse [B]); lse = log sum_v exp(logit_v) (natural log)."""
    z = head_logits(h, W)
    B, V = z.shape
    m = z.max(axis=1, keepdims=True)
    e = np.exp(z - m)
    s = e.sum(axis=1, keepdims=True)
    p = e / s
    lse = (m + np.log(s))[:, 0]
    ids = np.zeros((B, topk), dtype=np.int32)
    probs = np.zeros((B, topk))
    for b in range(B):
        # decreasing probability, ties to the lower id
        order = np.lexsort((np.arange(V), -z[b]))[:topk]
        ids[b] = order
        probs[b] = p[b, order]
    p0 = probs[:, 0]
    k = sibling_count(p0)
    stop = (p0 <= tau).astype(np.int32)
    return ids, probs, p0, k, stop, lse
