"""Block-causal training attention of the decoder (oracle; test infrastructure).

Sec. 4.2 ("Training with Block Attention") trains the decoder for drafting by
cutting each sequence into blocks of b tokens.  In the decoder's pass over the
raw embeddings H^0, the query at position p attends
* to the decoder's deep cache KV^dec (from the full forward pass) at every
  position of the preceding blocks, i.e. positions < n'(p), and
* causally to the tokens of its own block through self-attention over the raw
  embeddings: the decoder's own keys and values ("spec" rows here) at
  positions n'(p) .. p,
where n'(p) is the first position of p's block (0-based: (p // b) * b, the
paper's n' = floor((j - 2) / b) * b + 1 for target j = p + 2 in its 1-based
indexing).  Fig. 2 (right) shows the mask for n = 6, b = 2.

The attention itself is the softmax attention of ``attention.attend`` over
the rows the mask lets the query see, with grouped-query heads.
"""

from __future__ import annotations

import numpy as np

from . import attention as _attn


def block_start(p, b: int):
    """First position of the block that holds position p (0-based)."""
    return (np.asarray(p) // b) * b


def visibility(n: int, b: int):
    """(dec [n, n], spec [n, n]) boolean masks: query p sees dec row k iff
    k < block_start(p), spec row k iff block_start(p) <= k <= p."""
    p = np.arange(n)[:, None]
    k = np.arange(n)[None, :]
    s = block_start(p, b)
    return k < s, (k >= s) & (k <= p)


def block_causal_attention(q: np.ndarray, k_dec: np.ndarray, v_dec: np.ndarray,
                           k_spec: np.ndarray, v_spec: np.ndarray, b: int, scale: float):
    """One sequence.  q [n, Hq, D]; k/v_dec and k/v_spec [n, Hkv, D] (float64).
    Returns (o [n, Hq, D], lse [n, Hq]) with natural-log lse."""
    n, Hq, D = q.shape
    Hkv = k_dec.shape[1]
    G = Hq // Hkv
    dec, spec = visibility(n, b)
    o = np.zeros((n, Hq, D))
    lse = np.zeros((n, Hq))
    for p in range(n):
        rows_k = np.concatenate([k_dec[dec[p]], k_spec[spec[p]]], axis=0)
        rows_v = np.concatenate([v_dec[dec[p]], v_spec[spec[p]]], axis=0)
        for h in range(Hq):
            g = h // G
            o[p, h], lse[p, h], _ = _attn.attend(q[p, h], rows_k[:, g], rows_v[:, g], scale)
    return o, lse
