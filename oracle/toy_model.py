"""A tiny float64 transformer running SEED's decode loop (oracle; test
infrastructure).

Sec. 4.1 states that the encoder/decoder view is exactly equivalent to
standard autoregressive decoding, and greedy speculative decoding accepts a
draft only where it equals the verifier's argmax; hence greedy SEED (Alg. 2)
must emit exactly the greedy autoregressive token stream whatever the drafts
are.  This module provides both sides of that statement for a small random
model so that the oracle's attention, paged cache, acceptance and
commit/rollback can be checked end to end:

* ``ToyLM.greedy_ar``   -- plain greedy decoding; every step recomputes the
  whole prefix with a dense causal attention matrix (no cache, no oracle
  attention code);
* ``seed_greedy``       -- Alg. 2: d drafts from the last layers (f_dec) fed
  with raw embeddings and attending to the verifier-written deep cache plus
  the draft rows, one (d+1)-query causal verify pass over all layers on a
  paged cache, greedy acceptance, bonus token, rollback (rolled-back rows are
  overwritten with NaN so that any later read shows up).

Model: pre-norm residual blocks (RMS norm without gain), grouped-query
attention, ReLU MLP, learned absolute positions added to the token embedding,
untied output head.
"""

from __future__ import annotations

import numpy as np

from . import accept as _accept
from . import attention as _attn
from . import cache as _cache


class ToyLM:
    def __init__(self, seed: int, n_layers: int = 4, split: int = 2, d_model: int = 32,
                 hq: int = 2, hkv: int = 1, head_dim: int = 16, vocab: int = 50,
                 max_pos: int = 512, d_ff: int = 64):
        g = np.random.default_rng(seed)
        self.n_layers, self.split = n_layers, split
        self.hq, self.hkv, self.hd, self.vocab = hq, hkv, head_dim, vocab
        self.scale = 1.0 / np.sqrt(head_dim)
        self.W_in = g.standard_normal((vocab, d_model))
        self.pos = 0.5 * g.standard_normal((max_pos, d_model))
        self.W_out = g.standard_normal((vocab, d_model)) * 2.0

        def w(a, b):
            return g.standard_normal((a, b)) / np.sqrt(a)

        self.layers = [dict(Wq=w(d_model, hq * head_dim), Wk=w(d_model, hkv * head_dim),
                            Wv=w(d_model, hkv * head_dim), Wo=w(hq * head_dim, d_model),
                            W1=w(d_model, d_ff), W2=w(d_ff, d_model))
                       for _ in range(n_layers)]

    @staticmethod
    def _norm(x):
        return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + 1e-6)

    def embed(self, ids, positions):
        return self.W_in[np.asarray(ids)] + self.pos[np.asarray(positions)]

    def qkv(self, l, h):
        P = self.layers[l]
        x = self._norm(h)
        n = h.shape[0]
        return ((x @ P["Wq"]).reshape(n, self.hq, self.hd),
                (x @ P["Wk"]).reshape(n, self.hkv, self.hd),
                (x @ P["Wv"]).reshape(n, self.hkv, self.hd))

    def post(self, l, h, o):
        P = self.layers[l]
        h = h + o.reshape(h.shape[0], -1) @ P["Wo"]
        return h + np.maximum(self._norm(h) @ P["W1"], 0.0) @ P["W2"]

    def logits(self, h):
        return self._norm(h) @ self.W_out.T

    # ------------------------------------------------------------ dense AR
    def forward_dense(self, ids):
        """Logits at every position plus the per-layer K/V rows; dense causal
        attention, no cache."""
        n = len(ids)
        h = self.embed(ids, np.arange(n))
        G = self.hq // self.hkv
        ks, vs = [], []
        for l in range(self.n_layers):
            q, k, v = self.qkv(l, h)
            ks.append(k)
            vs.append(v)
            o = np.zeros_like(q)
            for hh in range(self.hq):
                S = self.scale * (q[:, hh] @ k[:, hh // G].T)
                S[np.triu_indices(n, 1)] = -np.inf
                S = S - S.max(axis=1, keepdims=True)
                E = np.exp(S)
                o[:, hh] = (E / E.sum(axis=1, keepdims=True)) @ v[:, hh // G]
            h = self.post(l, h, o)
        return self.logits(h), ks, vs

    def greedy_ar(self, prompt, n_new):
        """Returns (tokens, smallest top-1/top-2 logit gap seen)."""
        ids = list(prompt)
        gap = np.inf
        for _ in range(n_new):
            lg = self.forward_dense(ids)[0][-1]
            top2 = np.sort(lg)[-2:]
            gap = min(gap, top2[1] - top2[0])
            ids.append(int(np.argmax(lg)))
        return ids[len(prompt):], gap


def seed_greedy(model: ToyLM, prompt, n_new: int, d: int, drafter: str = "model",
                reference=None, page_size: int = 4, page_seed: int = 0):
    """Alg. 2 with draft length d on a paged cache in a random page order.

    drafter: 'model' (argmax of f_dec on raw embeddings), 'perfect' (the
    reference stream's next token) or 'adversarial' (always a wrong token).
    Returns (tokens, accepted count per round).
    """
    L = len(prompt) - 1                     # committed rows (t - 1)
    pending = int(prompt[-1])               # X_t, not yet in the cache
    cap = len(prompt) + n_new + d + 2
    n_pages = -(-cap // page_size)
    pt = np.random.default_rng(page_seed).permutation(n_pages).astype(np.int32)
    shape = (n_pages, model.hkv, page_size, model.hd)
    kc = [np.full(shape, np.nan) for _ in range(model.n_layers)]
    vc = [np.full(shape, np.nan) for _ in range(model.n_layers)]
    if L > 0:
        _, ks, vs = model.forward_dense(list(prompt[:L]))
        for l in range(model.n_layers):
            _cache.write_rows(kc[l], pt, 0, ks[l])
            _cache.write_rows(vc[l], pt, 0, vs[l])

    dec = range(model.split, model.n_layers)
    out, rounds = [], []
    while len(out) < n_new:
        # drafting phase: d tokens from f_dec on raw embeddings
        drafts = [pending]
        dk = {l: [] for l in dec}
        dv = {l: [] for l in dec}
        for i in range(1, d + 1):
            h = model.embed([drafts[i - 1]], [L + i - 1])
            for l in dec:
                q, k, v = model.qkv(l, h)
                dk[l].append(k[0])
                dv[l].append(v[0])
                o, _ = _attn.draft_attention_seq(
                    q[0], _cache.gather_rows(kc[l], pt, L), _cache.gather_rows(vc[l], pt, L),
                    np.stack(dk[l]), np.stack(dv[l]), model.scale)
                h = model.post(l, h, o[None])
            x = int(np.argmax(model.logits(h)[0]))
            ref_i = len(out) + i - 1
            if drafter == "perfect" and ref_i < len(reference):
                x = int(reference[ref_i])
            elif drafter == "adversarial" and ref_i < len(reference):
                x = (int(reference[ref_i]) + 1) % model.vocab
            drafts.append(x)

        # verification phase: all layers, d+1 queries, causal among them
        H = model.embed(drafts, L + np.arange(d + 1))
        for l in range(model.n_layers):
            q, k, v = model.qkv(l, H)
            _cache.write_rows(kc[l], pt, L, k)
            _cache.write_rows(vc[l], pt, L, v)
            o, _ = _attn.verify_attention_seq(
                q, _cache.gather_rows(kc[l], pt, L + d + 1), _cache.gather_rows(vc[l], pt, L + d + 1),
                L, model.scale)
            H = model.post(l, H, o)
        target = np.argmax(model.logits(H), axis=1)

        draft_ids = np.array([drafts[1:] + [0]], dtype=np.int64)[:, :max(d, 1)]
        acc, tokens, _, new_L = _accept.accept_commit(
            draft_ids, target[None, :], [d], [L], pt[None, :], page_size)
        n = int(acc[0])
        for l in range(model.n_layers):
            _cache.poison_from(kc[l], pt, int(new_L[0]), n_pages * page_size)
            _cache.poison_from(vc[l], pt, int(new_L[0]), n_pages * page_size)
        out.extend(int(t) for t in tokens[0, :n + 1])
        pending = int(tokens[0, n])
        L = int(new_L[0])
        rounds.append(n)
    return out[:n_new], rounds


def seed_tree_greedy(model: ToyLM, prompt, n_new: int, depth: int, width: int,
                     drafter: str = "model", reference=None, page_size: int = 4,
                     page_seed: int = 0, mistake: str | None = None, tau: float | None = None,
                     max_nodes: int = 32):
    """SEED with a draft tree and tree-based verification (Sec. D.1).

    Each round drafts a main branch of `depth` tokens with f_dec (as in Alg. 2);
    at every step the node being extended gets `width` children, the drafter's
    top-`width` distinct tokens, and the top-1 child continues the branch.
    drafter 'perfect' / 'adversarial' force the top-1 child to the reference
    token / a wrong token (its siblings stay the drafter's next choices).  All
    nodes are verified in one pass with the tree mask; the tree is walked
    greedily; the accepted path's rows are compacted into place.

    mistake (planted, for the tests): 'causal' lets every node see all earlier
    packed rows (siblings included); 'nocompact' skips moving the accepted
    rows.

    tau (dynamic drafting, Sec. D.1): when given, `width` is ignored; each
    step adds k children by the sibling-count rule on the drafter's top-1
    probability p0, drafting stops after a step with p0 <= tau or at `depth`
    steps, and the tree holds at most `max_nodes` nodes.  Returns (tokens,
    accepted count per round).
    """
    from . import drafting as _drafting
    from . import tree as _tree

    L = len(prompt) - 1
    pending = int(prompt[-1])
    n_nodes = 1 + depth * width if tau is None else max_nodes
    cap = len(prompt) + n_new + n_nodes + 2
    n_pages = -(-cap // page_size)
    pt = np.random.default_rng(page_seed).permutation(n_pages).astype(np.int32)
    shape = (n_pages, model.hkv, page_size, model.hd)
    kc = [np.full(shape, np.nan) for _ in range(model.n_layers)]
    vc = [np.full(shape, np.nan) for _ in range(model.n_layers)]
    if L > 0:
        _, ks, vs = model.forward_dense(list(prompt[:L]))
        for l in range(model.n_layers):
            _cache.write_rows(kc[l], pt, 0, ks[l])
            _cache.write_rows(vc[l], pt, 0, vs[l])

    dec = range(model.split, model.n_layers)
    out, rounds = [], []
    while len(out) < n_new:
        # ---- drafting: the main branch, with `width` children per step
        tok, parent = [pending], [-1]
        main = 0
        dk = {l: [] for l in dec}
        dv = {l: [] for l in dec}
        for i in range(1, depth + 1):
            h = model.embed([tok[main]], [L + i - 1])
            for l in dec:
                q, k, v = model.qkv(l, h)
                dk[l].append(k[0])
                dv[l].append(v[0])
                o, _ = _attn.draft_attention_seq(
                    q[0], _cache.gather_rows(kc[l], pt, L), _cache.gather_rows(vc[l], pt, L),
                    np.stack(dk[l]), np.stack(dv[l]), model.scale)
                h = model.post(l, h, o[None])
            lg = model.logits(h)[0]
            order = [int(t) for t in np.argsort(-lg, kind="stable")]
            if tau is not None:
                e = np.exp(lg - lg.max())
                p0 = float(e.max() / e.sum())
                width = min(int(_drafting.sibling_count([p0])[0]), max_nodes - len(tok))
            ref_i = len(out) + i - 1
            first = None
            if drafter == "perfect" and reference is not None and ref_i < len(reference):
                first = int(reference[ref_i])
            elif drafter == "adversarial" and reference is not None and ref_i < len(reference):
                first = (int(reference[ref_i]) + 1) % model.vocab
            kids = ([first] if first is not None else []) + [t for t in order if t != first]
            kids = kids[:width]
            base = len(tok)
            for t in kids:
                tok.append(t)
                parent.append(main)
            main = base
            if tau is not None and (p0 <= tau or len(tok) >= max_nodes):
                break
        n = len(tok)

        # ---- verification: all nodes in one pass with the tree mask
        dep = _tree.depths(parent)
        H = model.embed(tok, L + dep)
        pmask = list(range(-1, n - 1)) if mistake == "causal" else parent
        for l in range(model.n_layers):
            q, k, v = model.qkv(l, H)
            _cache.write_rows(kc[l], pt, L, k)
            _cache.write_rows(vc[l], pt, L, v)
            o, _ = _tree.tree_verify_attention_seq(
                q, _cache.gather_rows(kc[l], pt, L + n), _cache.gather_rows(vc[l], pt, L + n),
                L, pmask, model.scale)
            H = model.post(l, H, o)
        target = np.argmax(model.logits(H), axis=1)

        # ---- greedy walk, commit of the accepted path
        acc, tokens, path, _, new_L = _tree.tree_accept_commit(
            np.array([tok]), np.array([parent]), [n], target[None, :], [L], pt[None, :],
            page_size)
        m = int(acc[0])
        for l in range(model.n_layers):
            if mistake != "nocompact":
                for c in (kc[l], vc[l]):
                    rows = _cache.gather_rows(c, pt, L + n)
                    rows = _tree.compact_path(rows, L, path[0], m)
                    _cache.write_rows(c, pt, L, rows[L:L + m + 1])
            _cache.poison_from(kc[l], pt, int(new_L[0]), n_pages * page_size)
            _cache.poison_from(vc[l], pt, int(new_L[0]), n_pages * page_size)
        out.extend(int(t) for t in tokens[0, :m + 1])
        pending = int(tokens[0, m])
        L = int(new_L[0])
        rounds.append(m)
    return out[:n_new], rounds
