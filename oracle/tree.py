"""Tree-based verification (oracle; test infrastructure).

Sec. D.1 ("Tree-Based Verification") verifies a tree of candidate drafts in one
full-model pass:
* the tree's nodes are linearised into one packed sequence;
* each candidate attends to every verified prefix row and to the candidates on
  its own ancestral path, and to no other branch;
* after the pass, the tree is walked from the root, greedily accepting the
  longest prefix whose verified predictions match the drafted tokens, plus one
  bonus token from the verifier at the first position not accepted;
* the KV cache is then truncated to the accepted path.

Readings used here (the paper gives no layout):
* Node 0 is the root, the last verified token (X_draft[0] of the linear case),
  whose row is not in the cache yet.  Nodes are numbered in a topological
  order: parent[i] < i for i >= 1, parent[0] = -1.
* With L committed rows, the verify pass writes node i's K/V at packed
  position L + i.  Node i sees positions 0..L-1 and L + a for every ancestor
  a of i, itself included.  Its model position (for position embeddings) is
  L + depth(i).
* target[i] is the verifier's argmax at node i: the prediction of the token
  that follows node i.
* The walk: from cur = 0, accept the child c of cur whose token equals
  target[cur]; when several children carry that token, the lowest node index
  is taken.  It stops when no child matches.  The bonus token is
  target[cur].
* Commit: the accepted path's rows move from packed positions L + path[d] to
  L + d (d = 0..n, path[0] = 0), so that the cache again holds one row per
  position of the emitted stream; L becomes L + n + 1.
"""

from __future__ import annotations

import numpy as np

from . import attention as _attn


def depths(parent) -> np.ndarray:
    parent = np.asarray(parent)
    d = np.zeros(len(parent), dtype=np.int64)
    for i in range(1, len(parent)):
        d[i] = d[parent[i]] + 1
    return d


def ancestor_masks(parent) -> np.ndarray:
    """uint32 [n]: bit a of entry i is set when node a is an ancestor of node
    i or node i itself."""
    parent = np.asarray(parent)
    m = np.zeros(len(parent), dtype=np.uint64)
    for i in range(len(parent)):
        a = i
        while a >= 0:
            m[i] |= np.uint64(1) << np.uint64(a)
            a = int(parent[a]) if a > 0 else -1
    return m.astype(np.uint32)


def tree_verify_attention_seq(q: np.ndarray, k_rows: np.ndarray, v_rows: np.ndarray, L: int,
                              parent, scale: float):
    """Verify attention of one sequence's draft tree in one layer.

    q [n, Hq, D] (queries of nodes 0..n-1); k_rows/v_rows [L + n, Hkv, D]
    (committed rows, then the packed rows of the n nodes).  Returns
    (o [n, Hq, D], lse [n, Hq]).
    """
    n, Hq, D = q.shape
    Hkv = k_rows.shape[1]
    G = Hq // Hkv
    anc = ancestor_masks(parent)
    vis_nodes = np.zeros((n, L + n), dtype=bool)
    for j in range(n):
        vis_nodes[j, :L] = True
        for a in range(n):
            if (int(anc[j]) >> a) & 1:
                vis_nodes[j, L + a] = True
    o = np.zeros((n, Hq, D))
    lse = np.zeros((n, Hq))
    for g in range(Hkv):
        Qg = q[:, g * G:(g + 1) * G].reshape(n * G, D)
        vis = np.repeat(vis_nodes, G, axis=0)
        og, lg, _ = _attn.masked_attention(Qg, k_rows[:L + n, g], v_rows[:L + n, g], vis, scale)
        o[:, g * G:(g + 1) * G] = og.reshape(n, G, D)
        lse[:, g * G:(g + 1) * G] = lg.reshape(n, G)
    return o, lse


def tree_accept_commit(tok, parent, n_nodes, target, ctx_lens, page_table, page_size: int):
    """Greedy walk of each sequence's tree.

    tok, parent, target: [B, W] (W >= max n_nodes); tok[b, 0] is the root.
    Returns (accepted [B], tokens [B, W], path [B, W], slots [B, W],
    new_ctx_lens [B]); tokens = the accepted drafts then the bonus; path[d] =
    node at depth d of the accepted path (path[0] = 0); slots = cache slots of
    positions L..L+n after the commit; unused entries are -1.
    """
    tok = np.asarray(tok)
    parent = np.asarray(parent)
    target = np.asarray(target)
    B, W = tok.shape
    accepted = np.zeros(B, dtype=np.int32)
    tokens = np.full((B, W), -1, dtype=np.int32)
    path = np.full((B, W), -1, dtype=np.int32)
    slots = np.full((B, W), -1, dtype=np.int32)
    new_lens = np.array(ctx_lens, dtype=np.int32).copy()
    for b in range(B):
        n_b = int(n_nodes[b])
        cur, walk = 0, [0]
        while True:
            nxt = -1
            for c in range(1, n_b):
                if int(parent[b, c]) == cur and int(tok[b, c]) == int(target[b, cur]):
                    nxt = c
                    break
            if nxt < 0:
                break
            walk.append(nxt)
            cur = nxt
        n = len(walk) - 1
        accepted[b] = n
        for d in range(1, n + 1):
            tokens[b, d - 1] = tok[b, walk[d]]
        tokens[b, n] = target[b, cur]
        path[b, :n + 1] = walk
        L = int(ctx_lens[b])
        for d in range(n + 1):
            pos = L + d
            slots[b, d] = int(page_table[b, pos // page_size]) * page_size + pos % page_size
        new_lens[b] = L + n + 1
    return accepted, tokens, path, slots, new_lens


def compact_path(rows: np.ndarray, L: int, path, n: int) -> np.ndarray:
    """Logical rows of one sequence after the commit: rows [m, ...] indexed by
    position; the accepted path's rows move from L + path[d] to L + d."""
    out = rows.copy()
    for d in range(1, n + 1):
        out[L + d] = rows[L + int(path[d])]
    return out
