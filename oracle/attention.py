"""Softmax attention over the KV cache, float64 (oracle; test infrastructure).

Sec. 4.1 ("Cheap drafting between verifications") states that the drafter's
cross-attention to the cached deep representations is ordinary self-attention
over the KV cache.  Sec. 3 defines the per-layer cache KV^i_{<t}.  So the
quantity computed at every draft and verify step is textbook softmax attention
of each query head over the rows it may see:

    s_j = scale * <q, K_j>,   p = softmax(s),   o = sum_j p_j V_j,
    lse = log sum_j exp(s_j)

with grouped-query heads: query head h reads KV head h // (Hq / Hkv).

Which rows a query may see follows Alg. 2:
* draft step i (1-based) of a round that starts with L committed rows reads the
  committed rows 0..L-1 of that decoder layer plus the draft rows 0..i-1 (the
  rows of X_draft[0..i-1]; its own row included);
* verify query j (token X_draft[j], j = 0..k) reads rows 0..L+j of the layer
  (causal among the k+1 new rows).
"""

from __future__ import annotations

import numpy as np


def default_scale(head_dim: int) -> float:
    return 1.0 / np.sqrt(head_dim)


def attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, scale: float):
    """One query over n visible rows.

    q [D], K [n, D], V [n, D] (float64, n >= 1).
    Returns (o [D], lse, p [n]); lse is the natural-log sum of exp scores.
    """
    s = scale * (K @ q)
    m = np.max(s)
    e = np.exp(s - m)
    l = np.sum(e)
    p = e / l
    return p @ V, m + np.log(l), p


def masked_attention(Q: np.ndarray, K: np.ndarray, V: np.ndarray, visible: np.ndarray,
                     scale: float):
    """Many queries over shared rows with an explicit visibility mask.

    Q [M, D], K/V [n, D], visible bool [M, n] with at least one True per row.
    Returns (O [M, D], lse [M], P [M, n]).
    """
    S = scale * (Q @ K.T)
    S = np.where(visible, S, -np.inf)
    m = np.max(S, axis=1, keepdims=True)
    E = np.where(visible, np.exp(S - m), 0.0)
    l = np.sum(E, axis=1, keepdims=True)
    P = E / l
    # invisible rows contribute exactly nothing, even if they hold NaN
    O = np.zeros((Q.shape[0], V.shape[1]))
    for r in range(Q.shape[0]):
        cols = np.nonzero(visible[r])[0]
        O[r] = P[r, cols] @ V[cols]
    return O, (m + np.log(l))[:, 0], P


def draft_attention_seq(q: np.ndarray, ctx_k: np.ndarray, ctx_v: np.ndarray,
                        draft_k: np.ndarray, draft_v: np.ndarray, scale: float):
    """Draft attention of one sequence in one decoder layer.

    q [Hq, D]; ctx_k/ctx_v [L, Hkv, D] (committed rows 0..L-1 of the layer's
    cache, KV^dec); draft_k/draft_v [i, Hkv, D] (rows of X_draft[0..i-1]).
    Every query head sees all L + i rows.  Returns (o [Hq, D], lse [Hq]).
    """
    Hq, D = q.shape
    Hkv = ctx_k.shape[1]
    G = Hq // Hkv
    K = np.concatenate([ctx_k, draft_k], axis=0)
    V = np.concatenate([ctx_v, draft_v], axis=0)
    o = np.zeros((Hq, D))
    lse = np.zeros(Hq)
    for g in range(Hkv):
        Qg = q[g * G:(g + 1) * G]
        vis = np.ones((G, K.shape[0]), dtype=bool)
        og, lg, _ = masked_attention(Qg, K[:, g], V[:, g], vis, scale)
        o[g * G:(g + 1) * G] = og
        lse[g * G:(g + 1) * G] = lg
    return o, lse


def verify_attention_seq(q: np.ndarray, k_rows: np.ndarray, v_rows: np.ndarray, L: int,
                         scale: float):
    """Verify attention of one sequence in one layer.

    q [n_q, Hq, D] (queries of X_draft[0..n_q-1]); k_rows/v_rows
    [L + n_q, Hkv, D] (committed rows, then the n_q rows the verify pass just
    appended).  Query j sees rows 0..L+j.  Returns (o [n_q, Hq, D],
    lse [n_q, Hq]).
    """
    n_q, Hq, D = q.shape
    Hkv = k_rows.shape[1]
    G = Hq // Hkv
    n = L + n_q
    o = np.zeros((n_q, Hq, D))
    lse = np.zeros((n_q, Hq))
    for g in range(Hkv):
        Qg = q[:, g * G:(g + 1) * G].reshape(n_q * G, D)       # row = j*G + hh
        vis = np.zeros((n_q * G, n), dtype=bool)
        for j in range(n_q):
            vis[j * G:(j + 1) * G, :L + j + 1] = True
        og, lg, _ = masked_attention(Qg, k_rows[:n, g], v_rows[:n, g], vis, scale)
        o[:, g * G:(g + 1) * G] = og.reshape(n_q, G, D)
        lse[:, g * G:(g + 1) * G] = lg.reshape(n_q, G)
    return o, lse


def merge_partials(o_parts: np.ndarray, lse_parts: np.ndarray):
    """Combine attention over disjoint row sets into attention over their
    union: LSE = log sum_s exp(lse_s), O = sum_s exp(lse_s - LSE) O_s.

    o_parts [S, ..., D], lse_parts [S, ...].  Follows from the definition of
    softmax (each part is normalised by its own sum exp(lse_s)).
    """
    m = np.max(lse_parts, axis=0)
    w = np.exp(lse_parts - m)
    tot = np.sum(w, axis=0)
    LSE = m + np.log(tot)
    O = np.sum((w / tot)[..., None] * o_parts, axis=0)
    return O, LSE
