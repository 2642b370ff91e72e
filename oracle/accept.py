"""Greedy acceptance and KV commit/rollback (oracle; test infrastructure).

Alg. 2 (inference with fixed draft length), after the verification pass:
* n_accept counts drafts from the front while argmax p_i equals X_draft[i] and
  stops at the first mismatch;
* the bonus token is argmax p_{n_accept+1};
* the sequence gains X_draft[1..n_accept] followed by the bonus token;
* the cache keeps the rows of X_draft[0..n_accept] (positions t..t+n_accept in
  the paper's 1-based count) and drops the rest; t grows by n_accept + 1.

In 0-based terms with L = t - 1 committed rows: the verify pass appended rows
L..L+k_b; rows L..L+n are committed, rows L+n+1..L+k_b are rolled back, and
L becomes L + n + 1.

Array conventions: draft_ids[b, i] is X_draft[i+1] (i < k_b); target_ids[b, i]
is argmax p_{i+1} (i <= k_b).
"""

from __future__ import annotations

import numpy as np


def accept_commit(draft_ids, target_ids, k_b, ctx_lens, page_table, page_size: int):
    """Returns (accepted [B], tokens [B, kmax+1], slots [B, kmax+1],
    new_ctx_lens [B]); unused entries of tokens and slots are -1."""
    draft_ids = np.asarray(draft_ids)
    target_ids = np.asarray(target_ids)
    B = len(k_b)
    width = target_ids.shape[1]
    accepted = np.zeros(B, dtype=np.int32)
    tokens = np.full((B, width), -1, dtype=np.int32)
    slots = np.full((B, width), -1, dtype=np.int32)
    new_lens = np.array(ctx_lens, dtype=np.int32).copy()
    for b in range(B):
        n = 0
        for i in range(int(k_b[b])):
            if int(target_ids[b, i]) == int(draft_ids[b, i]):
                n += 1
            else:
                break
        accepted[b] = n
        for i in range(n):
            tokens[b, i] = draft_ids[b, i]
        tokens[b, n] = target_ids[b, n]
        L = int(ctx_lens[b])
        for i in range(n + 1):
            pos = L + i
            slots[b, i] = int(page_table[b, pos // page_size]) * page_size + pos % page_size
        new_lens[b] = L + n + 1
    return accepted, tokens, slots, new_lens
