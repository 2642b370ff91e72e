"""Device-side materialisation of the synthetic workloads and the decode-round
driver used by the GPU tests and bench.py.

Plumbing only: the pool of bf16 values goes to the GPU once, every input block
is a view (window) of it, the paged caches are filled with torch copies, and a
round is the sequence of C-ABI calls of Alg. 2 (draft appends and draft
attention per draft step and decoder layer, cache appends and verify attention
per layer, accept/commit).  No attention or acceptance arithmetic happens
here.
"""

from __future__ import annotations

import math

import numpy as np
import torch

import paper_2609_36590_gb300 as seed

from . import gen
from .configs import PAGE_SIZE, Workload


def bf16_tensor(bits: np.ndarray, device) -> torch.Tensor:
    return torch.from_numpy(np.array(bits, copy=True).view(np.int16)).to(device).view(torch.bfloat16)


class DeviceWorkload:
    """Caches, inputs and state of one workload on one GPU.

    layers: which layers' caches exist (default: all); the verify pass runs
    over these, the draft over the workload's decoder layers (which must be
    among them).  rounds: how many rounds the page table must hold.
    """

    def __init__(self, wl: Workload, device="cuda", layers=None, rounds=None):
        self.wl = wl
        self.device = device
        B, D = wl.batch, wl.head_dim
        self.rounds = wl.rounds if rounds is None else rounds
        self.layers = list(range(wl.n_layers)) if layers is None else sorted(layers)
        for l in wl.dec_layers:
            assert l in self.layers, "decoder layers must be materialised"
        self.cfg = seed.SeedConfig(hq=wl.hq, hkv=wl.hkv, head_dim=D, kmax=wl.kmax,
                                   page_size=PAGE_SIZE)
        self.lens0 = gen.ctx_lens(wl)
        self.max_pages = gen.max_pages(wl, self.rounds)
        self.pt_np = gen.page_table(wl, self.max_pages)
        self.num_pages = B * self.max_pages
        self.pool = bf16_tensor(gen.value_pool(wl.index), device)
        self.page_table = torch.from_numpy(self.pt_np).to(device)
        self.ctx_lens = torch.from_numpy(self.lens0.copy()).to(device)
        self.kv = {l: self._build_cache(l) for l in self.layers}
        shp = (B, wl.hkv, wl.kmax, D)
        self.draft_k = {l: torch.zeros(shp, dtype=torch.bfloat16, device=device) for l in wl.dec_layers}
        self.draft_v = {l: torch.zeros(shp, dtype=torch.bfloat16, device=device) for l in wl.dec_layers}
        self.ws = seed.new_workspace(self.cfg, B, device)
        self.err = torch.zeros(1, dtype=torch.int32, device=device)
        self.out_d = torch.zeros(B, wl.hq, D, dtype=torch.float32, device=device)
        self.lse_d = torch.zeros(B, wl.hq, dtype=torch.float32, device=device)
        self.out_v = torch.zeros(B, wl.kmax + 1, wl.hq, D, dtype=torch.float32, device=device)
        self.lse_v = torch.zeros(B, wl.kmax + 1, wl.hq, dtype=torch.float32, device=device)
        W = wl.kmax + 1
        self.accepted = torch.zeros(B, dtype=torch.int32, device=device)
        self.tokens = torch.zeros(B, W, dtype=torch.int32, device=device)
        self.slots = torch.zeros(B, W, dtype=torch.int32, device=device)
        self._inputs = {}

    # ------------------------------------------------------------ inputs
    def window(self, kind: int, coords, n: int) -> torch.Tensor:
        off = gen.window_offset(self.wl, kind, *coords)
        return self.pool[off:off + n]

    def _build_cache(self, layer: int) -> seed.PagedKV:
        wl = self.wl
        D, Hkv = wl.head_dim, wl.hkv
        shape = (self.num_pages, Hkv, PAGE_SIZE, D)
        k = torch.full(shape, float("nan"), dtype=torch.bfloat16, device=self.device)
        v = torch.full(shape, float("nan"), dtype=torch.bfloat16, device=self.device)
        for b in range(wl.batch):
            L = int(self.lens0[b])
            npg = -(-L // PAGE_SIZE)
            if npg == 0:
                continue
            pids = self.page_table[b, :npg].long()
            for kind, dst in ((gen.K_CTX, k), (gen.V_CTX, v)):
                blk = torch.stack([self.window(kind, (layer, b, h), L * D).view(L, D)
                                   for h in range(Hkv)])
                if kind == gen.K_CTX and wl.key_stress > 0:
                    blk = blk.clone()
                    for h in range(Hkv):
                        rows = np.nonzero(gen.stress_rows(wl, layer, b, h, L))[0]
                        if len(rows):
                            r = torch.from_numpy(rows).to(self.device)
                            blk[h, r] = blk[h, r] * 8
                pad = torch.full((Hkv, npg * PAGE_SIZE, D), float("nan"), dtype=torch.bfloat16,
                                 device=self.device)
                pad[:, :L] = blk
                dst[pids] = pad.view(Hkv, npg, PAGE_SIZE, D).transpose(0, 1)
        return seed.PagedKV(k, v, self.page_table)

    def round_inputs(self, rnd: int) -> dict:
        if rnd in self._inputs:
            return self._inputs[rnd]
        wl = self.wl
        B, Hq, Hkv, D, K = wl.batch, wl.hq, wl.hkv, wl.head_dim, wl.kmax
        k_b, n_plan, draft_ids, target_ids = gen.round_plan(wl, rnd)
        dev = self.device
        ins = dict(k_b_np=k_b, n_plan=n_plan,
                   k_b=torch.from_numpy(k_b).to(dev),
                   n_q=torch.from_numpy(k_b + 1).to(dev),
                   draft_ids=torch.from_numpy(draft_ids).to(dev),
                   target_ids=torch.from_numpy(target_ids).to(dev),
                   steps=int(k_b.max()))
        ins["draft_lens"] = [torch.from_numpy(np.where(k_b >= i, i, 0).astype(np.int32)).to(dev)
                             for i in range(1, ins["steps"] + 1)]
        ins["draft"] = {}
        for i in range(1, ins["steps"] + 1):
            for l in wl.dec_layers:
                ins["draft"][(i, l)] = (
                    self.window(gen.Q_DRAFT, (rnd, i, l), B * Hq * D).view(B, Hq, D),
                    self.window(gen.K_DRAFT, (rnd, i, l), B * Hkv * D).view(B, Hkv, D),
                    self.window(gen.V_DRAFT, (rnd, i, l), B * Hkv * D).view(B, Hkv, D))
        ins["verify"] = {}
        for l in self.layers:
            ins["verify"][l] = (
                self.window(gen.Q_VERIFY, (rnd, l), B * (K + 1) * Hq * D).view(B, K + 1, Hq, D),
                self.window(gen.K_VERIFY, (rnd, l), B * (K + 1) * Hkv * D).view(B, K + 1, Hkv, D),
                self.window(gen.V_VERIFY, (rnd, l), B * (K + 1) * Hkv * D).view(B, K + 1, Hkv, D))
        self._inputs[rnd] = ins
        return ins

    # ------------------------------------------------------------ one round
    def draft_step(self, ins: dict, i: int, on_draft=None, marks=None) -> None:
        """marks: optional (before, after) callables run around each attention
        call, given ("draft", (i, layer)); bench.py records timing events there."""
        for l in self.wl.dec_layers:
            q, kn, vn = ins["draft"][(i, l)]
            dl = ins["draft_lens"][i - 1]
            seed.seed_draft_kv_append(self.cfg, kn, vn, dl, self.draft_k[l], self.draft_v[l], self.err)
            self.draft_attn(ins, i, l, marks)
            if on_draft is not None:
                on_draft(i, l, self.out_d, self.lse_d)

    def draft_attn(self, ins: dict, i: int, l: int, marks=None) -> None:
        q = ins["draft"][(i, l)][0]
        if marks:
            marks[0]("draft", (i, l))
        seed.seed_draft_attn(self.cfg, q, self.kv[l], self.draft_k[l], self.draft_v[l],
                             self.ctx_lens, ins["draft_lens"][i - 1], self.out_d, self.lse_d,
                             self.ws, self.err)
        if marks:
            marks[1]("draft", (i, l))

    def verify_layer(self, ins: dict, l: int, on_verify=None, marks=None) -> None:
        q, kn, vn = ins["verify"][l]
        seed.seed_kv_append(self.cfg, self.kv[l], kn, vn, ins["n_q"], self.ctx_lens, self.err)
        self.verify_attn(ins, l, marks)
        if on_verify is not None:
            on_verify(l, self.out_v, self.lse_v)

    def verify_attn(self, ins: dict, l: int, marks=None) -> None:
        if marks:
            marks[0]("verify", l)
        seed.seed_verify_attn(self.cfg, ins["verify"][l][0], ins["n_q"], self.kv[l],
                              self.ctx_lens, self.out_v, self.lse_v, self.ws, self.err)
        if marks:
            marks[1]("verify", l)

    def accept(self, ins: dict) -> None:
        seed.seed_accept_commit(self.wl.kmax, ins["draft_ids"], ins["target_ids"], ins["k_b"],
                                self.page_table, PAGE_SIZE, self.ctx_lens, self.accepted,
                                self.tokens, self.slots, self.err)

    def run_round(self, rnd: int, on_draft=None, on_verify=None) -> None:
        """Alg. 2, one round: k_b draft steps (2 decoder layers each), the
        verify pass over the materialised layers, then accept/commit."""
        ins = self.round_inputs(rnd)
        for i in range(1, ins["steps"] + 1):
            self.draft_step(ins, i, on_draft)
        for l in self.layers:
            self.verify_layer(ins, l, on_verify)
        self.accept(ins)

    # ------------------------------------------------------------ accounting
    def round_bytes(self, lens: np.ndarray, k_b: np.ndarray) -> dict:
        """Algorithmic HBM bytes of one round: every visible K/V row once per
        call, plus queries, new rows and outputs."""
        wl = self.wl
        R = wl.row_bytes
        qd = wl.hq * wl.head_dim
        act = [(int(lens[b]), int(k_b[b])) for b in range(wl.batch)]
        draft = 0
        for i in range(1, int(k_b.max()) + 1):
            for L, kb in act:
                if i <= kb:
                    # ctx + draft rows, q in, o (+lse) out, one new row appended
                    draft += len(wl.dec_layers) * ((L + i) * R + qd * 2 + qd * 4 + wl.hq * 4 + 2 * R)
        verify = 0
        for L, kb in act:
            n = kb + 1
            verify += len(self.layers) * ((L + n) * R + n * (qd * 2 + qd * 4 + wl.hq * 4) + n * R * 2)
        return dict(draft=draft, verify=verify)
