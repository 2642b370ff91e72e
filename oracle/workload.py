"""The oracle run over a synthetic workload (oracle; test infrastructure).

Keeps its own model of every sequence's committed cache and reproduces, from
the seeded generators alone, what each call of a decode round must return:
draft attention (Sec. 4.1; Alg. 2 drafting phase), verify attention (Alg. 2
verification phase) and accept/commit (Alg. 2, acceptance and truncation).
It never reads device memory.

Cache model: the initial context rows of (layer, b, KV head) come from
``gen.ctx_block``; a position committed in round r as the j-th verify row holds
row j of that round's ``gen.verify_kv_new``.  Provenance (round, j) per
committed position is the same for every layer, so one list per sequence
describes all layers.
"""

from __future__ import annotations

import numpy as np

from workloads import gen
from workloads.configs import PAGE_SIZE, Workload

from . import accept as _accept
from . import attention as _attn


class OracleRun:
    def __init__(self, wl: Workload, rounds: int | None = None):
        self.wl = wl
        self.scale = _attn.default_scale(wl.head_dim)
        self.lens0 = gen.ctx_lens(wl)
        self.lens = self.lens0.astype(np.int64).copy()
        self.max_pages = gen.max_pages(wl, wl.rounds if rounds is None else rounds)
        self.page_table = gen.page_table(wl, self.max_pages)
        self.prov = [[] for _ in range(wl.batch)]       # committed (round, j) past lens0
        self._ctx_cache = {}
        self._new_cache = {}

    # ---------------------------------------------------------------- rows
    def _ctx_rows(self, layer: int, b: int, kind: int) -> np.ndarray:
        """float64 [lens0[b], Hkv, D] initial context rows."""
        key = (layer, b, kind)
        if key not in self._ctx_cache:
            L = int(self.lens0[b])
            blocks = [gen.bf16_bits_to_f64(gen.ctx_block(self.wl, layer, b, h, kind, L))
                      for h in range(self.wl.hkv)]
            self._ctx_cache[key] = np.stack(blocks, axis=1) if L else \
                np.zeros((0, self.wl.hkv, self.wl.head_dim))
        return self._ctx_cache[key]

    def _verify_new(self, rnd: int, layer: int, kind: int) -> np.ndarray:
        key = (rnd, layer, kind)
        if key not in self._new_cache:
            self._new_cache[key] = gen.bf16_bits_to_f64(gen.verify_kv_new(self.wl, rnd, layer, kind))
        return self._new_cache[key]

    def committed_rows(self, layer: int, b: int, kind: int) -> np.ndarray:
        """[lens[b], Hkv, D]: the committed cache rows of (layer, b)."""
        base = self._ctx_rows(layer, b, kind)
        if not self.prov[b]:
            return base
        newk = gen.K_VERIFY if kind == gen.K_CTX else gen.V_VERIFY
        extra = np.stack([self._verify_new(r, layer, newk)[b, j] for r, j in self.prov[b]])
        return np.concatenate([base, extra], axis=0)

    # ---------------------------------------------------------------- calls
    def draft(self, rnd: int, step: int, layer: int, bs=None):
        """Draft attention of draft step `step` (1-based) in decoder layer
        `layer` for sequences bs (default: those drafting at this step).
        Returns {b: (o [Hq, D], lse [Hq])}."""
        wl = self.wl
        k_b = gen.round_plan(wl, rnd)[0]
        q = gen.bf16_bits_to_f64(gen.draft_q(wl, rnd, step, layer))
        dk = [gen.bf16_bits_to_f64(gen.draft_kv_new(wl, rnd, i, layer, gen.K_DRAFT))
              for i in range(1, step + 1)]
        dv = [gen.bf16_bits_to_f64(gen.draft_kv_new(wl, rnd, i, layer, gen.V_DRAFT))
              for i in range(1, step + 1)]
        res = {}
        for b in (range(wl.batch) if bs is None else bs):
            if step > k_b[b]:
                continue
            res[b] = _attn.draft_attention_seq(
                q[b], self.committed_rows(layer, b, gen.K_CTX),
                self.committed_rows(layer, b, gen.V_CTX),
                np.stack([x[b] for x in dk]), np.stack([x[b] for x in dv]), self.scale)
        return res

    def verify(self, rnd: int, layer: int, bs=None):
        """Verify attention of `layer` in round rnd: {b: (o [n_q, Hq, D],
        lse [n_q, Hq])} with n_q = k_b + 1."""
        wl = self.wl
        k_b = gen.round_plan(wl, rnd)[0]
        q = gen.bf16_bits_to_f64(gen.verify_q(wl, rnd, layer))
        nk = self._verify_new(rnd, layer, gen.K_VERIFY)
        nv = self._verify_new(rnd, layer, gen.V_VERIFY)
        res = {}
        for b in (range(wl.batch) if bs is None else bs):
            n = int(k_b[b]) + 1
            L = int(self.lens[b])
            K = np.concatenate([self.committed_rows(layer, b, gen.K_CTX), nk[b, :n]], axis=0)
            V = np.concatenate([self.committed_rows(layer, b, gen.V_CTX), nv[b, :n]], axis=0)
            res[b] = _attn.verify_attention_seq(q[b, :n], K, V, L, self.scale)
        return res

    def accept(self, rnd: int):
        """Accept/commit of round rnd; advances the cache model.  Returns
        (accepted, tokens, slots, new_lens)."""
        k_b, _, draft_ids, target_ids = gen.round_plan(self.wl, rnd)
        acc, tok, slots, new_lens = _accept.accept_commit(
            draft_ids, target_ids, k_b, self.lens.astype(np.int32), self.page_table, PAGE_SIZE)
        for b in range(self.wl.batch):
            self.prov[b].extend((rnd, j) for j in range(int(acc[b]) + 1))
        self.lens = new_lens.astype(np.int64)
        return acc, tok, slots, new_lens
