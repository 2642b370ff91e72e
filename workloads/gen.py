"""Seeded synthetic inputs, shared by the oracle and the CUDA path.

This module draws numbers and lays them out; it holds none of the method's
arithmetic (no attention, no acceptance rule).  Both sides consume the same
bytes: bf16 values are produced here as uint16 bit patterns.

Recipe
------
* One value pool per workload: ``POOL_ELEMS`` draws of N(0, 1) (float32,
  PCG64) rounded to bf16 with round-to-nearest-even.
* Every tensor block (the initial context keys of one (layer, sequence, KV
  head), the queries of one (round, draft step, layer), the new K/V rows of a
  verify pass, ...) is a window of that pool whose offset comes from its own
  ``SeedSequence`` stream keyed by the block's coordinates.  A block can
  therefore be regenerated on its own, which lets the oracle check sampled
  outputs of full-size runs without materialising the whole cache on the host.
* Key-stress rows (the batch-4, 32k-prefix long-context workload): each key
  row (layer, b, h, pos) of the initial context is scaled by 8 with
  probability ``key_stress``, drawn per block.
  Multiplying a bf16 value by 8 is exact.
* Context lengths, draft lengths, acceptance patterns, token ids and page
  orders each come from their own keyed stream.
"""

from __future__ import annotations

import functools
import math

import numpy as np

from .configs import PAGE_SIZE, Workload

BASE_SEED = 20260
POOL_ELEMS = 1 << 24
MAX_BLOCK = 1 << 23          # largest window handed out (elements)
WINDOW_ALIGN = 64            # window offsets are multiples of this (elements)
BF16_NAN = 0x7FC0            # quiet NaN used to poison stale cache rows

# stream tags
_T_POOL, _T_OFF, _T_LEN, _T_ROUND, _T_STRESS, _T_PAGES = range(6)
# block kinds
K_CTX, V_CTX, Q_DRAFT, K_DRAFT, V_DRAFT, Q_VERIFY, K_VERIFY, V_VERIFY = range(8)


def rng(*key: int) -> np.random.Generator:
    ss = np.random.SeedSequence(entropy=BASE_SEED, spawn_key=tuple(int(k) for k in key))
    return np.random.Generator(np.random.PCG64(ss))


# ---------------------------------------------------------------- bf16 bits
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(b).astype(np.float64)


# ---------------------------------------------------------------- the pool
@functools.lru_cache(maxsize=8)
def value_pool(wl_index: int) -> np.ndarray:
    """uint16 [POOL_ELEMS]: N(0,1) draws rounded to bf16."""
    x = rng(wl_index, _T_POOL).standard_normal(POOL_ELEMS, dtype=np.float32)
    out = f32_to_bf16_bits(x)
    out.setflags(write=False)
    return out


def window_offset(wl: Workload, kind: int, *coords: int) -> int:
    """Pool offset (elements) of the block (kind, *coords)."""
    g = rng(wl.index, _T_OFF, kind, *coords)
    slots = (POOL_ELEMS - MAX_BLOCK) // WINDOW_ALIGN
    return int(g.integers(0, slots)) * WINDOW_ALIGN


def window(wl: Workload, n: int, kind: int, *coords: int) -> np.ndarray:
    if n > MAX_BLOCK:
        raise ValueError(f"block of {n} elements exceeds MAX_BLOCK")
    off = window_offset(wl, kind, *coords)
    return value_pool(wl.index)[off:off + n]


# ---------------------------------------------------------------- lengths
def ctx_lens(wl: Workload) -> np.ndarray:
    """Initial committed context length L_b (rows already in the cache)."""
    g = rng(wl.index, _T_LEN)
    B = wl.batch
    if wl.ctx == "fixed":
        out = np.full(B, wl.ctx_lo, dtype=np.int64)
    elif wl.ctx == "uniform":
        out = g.integers(wl.ctx_lo, wl.ctx_hi + 1, size=B)
    elif wl.ctx == "loguniform":
        out = np.floor(np.exp(g.uniform(math.log(wl.ctx_lo), math.log(wl.ctx_hi), size=B)))
    else:
        raise ValueError(wl.ctx)
    return out.astype(np.int32)


def max_pages(wl: Workload, rounds: int | None = None) -> int:
    """Pages per sequence: room for the initial context plus `rounds` rounds of
    k_max+1 appended rows."""
    r = wl.rounds if rounds is None else rounds
    cap = int(ctx_lens(wl).max()) + r * (wl.kmax + 1) + 1
    return -(-cap // PAGE_SIZE)


def page_table(wl: Workload, n_pages_per_seq: int) -> np.ndarray:
    """int32 [B, n_pages_per_seq] physical page ids into a pool of
    B * n_pages_per_seq pages: identity order, or a seeded permutation."""
    B = wl.batch
    total = B * n_pages_per_seq
    if wl.paged_random:
        perm = rng(wl.index, _T_PAGES).permutation(total)
    else:
        perm = np.arange(total)
    return perm.reshape(B, n_pages_per_seq).astype(np.int32)


# ---------------------------------------------------------------- KV blocks
def stress_rows(wl: Workload, layer: int, b: int, h: int, n_rows: int) -> np.ndarray:
    """bool [n_rows]: key rows of the initial context scaled by 8."""
    if wl.key_stress <= 0.0:
        return np.zeros(n_rows, dtype=bool)
    return rng(wl.index, _T_STRESS, layer, b, h).random(n_rows) < wl.key_stress


def scale_bf16_by_8(bits: np.ndarray) -> np.ndarray:
    return f32_to_bf16_bits(bf16_bits_to_f32(bits) * np.float32(8.0))


def ctx_block(wl: Workload, layer: int, b: int, h: int, kind: int, n_rows: int) -> np.ndarray:
    """uint16 [n_rows, D]: rows 0..n_rows-1 of the initial context of
    (layer, b, KV head h); kind is K_CTX or V_CTX."""
    D = wl.head_dim
    blk = window(wl, n_rows * D, kind, layer, b, h).reshape(n_rows, D)
    if kind == K_CTX and wl.key_stress > 0.0:
        rows = stress_rows(wl, layer, b, h, n_rows)
        if rows.any():
            blk = blk.copy()
            blk[rows] = scale_bf16_by_8(blk[rows])
    return blk


def draft_q(wl: Workload, rnd: int, step: int, layer: int) -> np.ndarray:
    """uint16 [B, Hq, D]: draft query of draft step `step` (1-based)."""
    n = wl.batch * wl.hq * wl.head_dim
    return window(wl, n, Q_DRAFT, rnd, step, layer).reshape(wl.batch, wl.hq, wl.head_dim)


def draft_kv_new(wl: Workload, rnd: int, step: int, layer: int, kind: int) -> np.ndarray:
    """uint16 [B, Hkv, D]: the K (kind K_DRAFT) or V (V_DRAFT) row the drafter
    produces for X_draft[step-1] in `layer`."""
    n = wl.batch * wl.hkv * wl.head_dim
    return window(wl, n, kind, rnd, step, layer).reshape(wl.batch, wl.hkv, wl.head_dim)


def verify_q(wl: Workload, rnd: int, layer: int) -> np.ndarray:
    """uint16 [B, kmax+1, Hq, D]: verify queries for X_draft[0..kmax]."""
    n = wl.batch * (wl.kmax + 1) * wl.hq * wl.head_dim
    return window(wl, n, Q_VERIFY, rnd, layer).reshape(wl.batch, wl.kmax + 1, wl.hq, wl.head_dim)


def verify_kv_new(wl: Workload, rnd: int, layer: int, kind: int) -> np.ndarray:
    """uint16 [B, kmax+1, Hkv, D]: K (K_VERIFY) or V (V_VERIFY) rows the
    verifier produces for X_draft[0..kmax] in `layer`."""
    n = wl.batch * (wl.kmax + 1) * wl.hkv * wl.head_dim
    return window(wl, n, kind, rnd, layer).reshape(wl.batch, wl.kmax + 1, wl.hkv, wl.head_dim)


# ---------------------------------------------------------------- acceptance
def round_plan(wl: Workload, rnd: int):
    """Draft lengths and token ids of one round.

    Returns (k_b int32[B], n_planned int32[B], draft_ids int32[B, kmax],
    target_ids int32[B, kmax+1]).  draft_ids[b, i] stands for X_draft[i+1];
    target_ids[b, i] for argmax p_{i+1}.  The ids are built so that the first
    mismatch falls at n_planned[b] (no mismatch when n_planned[b] == k_b[b]).
    Positions i >= k_b[b] repeat the target id, so reading past k_b would
    accept more than planned.
    """
    g = rng(wl.index, _T_ROUND, rnd)
    B, K, V = wl.batch, wl.kmax, wl.vocab
    if wl.ragged_k:
        k_b = g.integers(1, K + 1, size=B)
    else:
        k_b = np.full(B, K, dtype=np.int64)
    if wl.accept == "forced" or wl.accept == "uniform":
        n = np.array([g.integers(0, kb + 1) for kb in k_b], dtype=np.int64)
    elif wl.accept == "geom":
        n = np.minimum(g.geometric(wl.geom_p, size=B) - 1, k_b)
    else:
        raise ValueError(wl.accept)
    target = g.integers(0, V, size=(B, K + 1))
    draft = g.integers(0, V, size=(B, K))
    shift = g.integers(1, V, size=B)            # 1..V-1: never a match
    for b in range(B):
        nb, kb = int(n[b]), int(k_b[b])
        draft[b, :nb] = target[b, :nb]
        if nb < kb:
            draft[b, nb] = (target[b, nb] + shift[b]) % V
        draft[b, kb:] = target[b, kb:K]
    return (k_b.astype(np.int32), n.astype(np.int32),
            draft.astype(np.int32), target.astype(np.int32))


# ---------------------------------------------------------------- small cases
def small_case(seed: int, B: int, hq: int, hkv: int, D: int, kmax: int, max_ctx: int,
               paged_random: bool = True, key_scale: float = 1.0) -> dict:
    """A random problem small enough for the oracle to check every output.

    Lengths cover the edges (0, 1, a page minus/plus one, multiples of the
    page) when B is large enough.  Returns uint16 bf16 bits for all tensors:
      rows_k/rows_v [B, max_ctx+kmax+1, hkv, D]  logical cache rows by position
      q_draft [B, hq, D], q_verify [B, kmax+1, hq, D]
      draft_k/draft_v [B, hkv, kmax, D]
    and int32 lens [B], draft_lens [B] (0..kmax), n_q [B] (0..kmax+1),
    page_table [B, max_pages], max_pages.
    """
    g = rng(9000, seed)
    edges = [0, 1, PAGE_SIZE - 1, PAGE_SIZE, PAGE_SIZE + 1, 2 * PAGE_SIZE, max_ctx]
    lens = g.integers(0, max_ctx + 1, size=B)
    for i in range(min(B, len(edges))):
        lens[i] = min(edges[i], max_ctx)
    n_q = g.integers(1, kmax + 2, size=B)
    draft_lens = g.integers(1, kmax + 1, size=B)
    if B >= 3:
        n_q[B - 1] = 0                      # a sequence that skips the verify call
        draft_lens[B - 2] = 0               # ... and one that skips the draft call
    n_rows = max_ctx + kmax + 1
    max_pages = -(-n_rows // PAGE_SIZE) + 1
    perm = g.permutation(B * max_pages) if paged_random else np.arange(B * max_pages)
    pt = perm.reshape(B, max_pages)

    def bits(shape, s=1.0):
        return f32_to_bf16_bits(g.standard_normal(shape, dtype=np.float32) * np.float32(s))

    return dict(
        lens=lens.astype(np.int32), n_q=n_q.astype(np.int32),
        draft_lens=draft_lens.astype(np.int32), page_table=pt.astype(np.int32),
        max_pages=max_pages,
        rows_k=bits((B, n_rows, hkv, D), key_scale), rows_v=bits((B, n_rows, hkv, D)),
        q_draft=bits((B, hq, D)), q_verify=bits((B, kmax + 1, hq, D)),
        draft_k=bits((B, hkv, kmax, D)), draft_v=bits((B, hkv, kmax, D)))


def accept_case(seed: int, B: int, kmax: int, vocab: int = 50, max_ctx: int = 300) -> dict:
    """Random acceptance inputs: k_b in 0..kmax, token ids with a planned first
    mismatch (sometimes none), positions past k_b equal to the target (so a
    reader that ignores k_b over-accepts), lengths and a page permutation."""
    g = rng(9100, seed)
    k_b = g.integers(0, kmax + 1, size=B)
    target = g.integers(0, vocab, size=(B, kmax + 1))
    draft = g.integers(0, vocab, size=(B, kmax))
    for b in range(B):
        n = int(g.integers(0, k_b[b] + 1))
        draft[b, :n] = target[b, :n]
        if n < k_b[b]:
            draft[b, n] = (target[b, n] + 1 + g.integers(0, vocab - 1)) % vocab
        draft[b, k_b[b]:] = target[b, k_b[b]:kmax]
    lens = g.integers(0, max_ctx + 1, size=B)
    max_pages = -(-(max_ctx + kmax + 1) // PAGE_SIZE)
    pt = g.permutation(B * max_pages).reshape(B, max_pages)
    return dict(k_b=k_b.astype(np.int32), draft_ids=draft.astype(np.int32),
                target_ids=target.astype(np.int32), lens=lens.astype(np.int32),
                page_table=pt.astype(np.int32), max_pages=max_pages)
