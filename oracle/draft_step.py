"""One draft step of SEED's decoder (oracle; test infrastructure).

Sec. 4.1 ("cheap drafting"): between verifications the decoder f_dec -- the
model's last l - l' = 2 transformer layers -- takes the raw embedding W_in x
of the latest token, attends to the deep KV cache of the verified prefix plus
the rows of the earlier drafts, and the LM head gives the next token's
distribution.  The computational-cost appendix fixes the work per draft token:
per decoder layer W_Q, W_K, W_V, W_O and three MLP matrices, plus the head
(tied to the input embedding).  The paper's models are Qwen3 base models, so
the layer is written in that family's pre-norm form:

    a   = RMSNorm(x; g_attn)
    q, k, v = a Wq^T, a Wk^T, a Wv^T                  (heads of D)
    q, k = RoPE(RMSNorm_head(q; g_q)), RoPE(RMSNorm_head(k; g_k))   at the token's position
    (k, v) become this step's draft row; o = attention(q; cache rows [0, L) + draft rows)
    x  += o Wo^T
    m   = RMSNorm(x; g_mlp)
    x  += (silu(m Wg^T) * (m Wu^T)) Wd^T
and after the last decoder layer h = RMSNorm(x; g_final) goes to the head.

Precision reading: weights and embeddings are bf16; the residual stream x is
kept at full precision; the operands of every matrix product and of the
attention (a, q, k, v, o, m and the MLP activation) are rounded to bf16
(round to nearest even, through float32), as a bf16 inference stack stores
them.  Everything else here is float64.

Positions: with L committed rows, draft step i (1-based) feeds the token at
position L + i - 1 (the last verified token at L for i = 1) and writes draft
row i - 1 (Alg. 2; the step's own row is visible to its query).
"""

from __future__ import annotations

import numpy as np

from . import attention as _attn
from . import drafting as _drafting

EPS = 1e-6
ROPE_THETA = 1.0e6


def bf16_round(x) -> np.ndarray:
    """Round to bf16 (nearest, ties to even) through float32; returns float64."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    nan = np.isnan(f)
    r = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    out = r.astype(np.uint32).view(np.float32).astype(np.float64)
    return np.where(nan, np.nan, out)


def rms_norm(x: np.ndarray, g: np.ndarray | None, eps: float = EPS) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    y = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return y if g is None else y * g


def rope(x: np.ndarray, pos, theta: float = ROPE_THETA) -> np.ndarray:
    """Rotary position embedding, rotate-half pairing (i, i + D/2), angle
    pos * theta^(-2i/D).  x [..., D]; pos broadcasts against x[..., 0]."""
    D = x.shape[-1]
    half = D // 2
    inv = theta ** (-(2.0 * np.arange(half)) / D)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * inv
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def decoder_layer(x: np.ndarray, P: dict, pos, ctx_k, ctx_v, draft_k, draft_v, hq: int,
                  hkv: int, D: int, scale: float | None = None):
    """One decoder layer for one draft step of a batch.

    x [B, dm] residual stream; P holds (float64 arrays of bf16 values)
    g_attn [dm], Wqkv [(hq + 2 hkv) D, dm] (rows: q heads, k heads, v heads),
    g_q [D], g_k [D], Wo [dm, hq D], g_mlp [dm], Wg [F, dm], Wu [F, dm],
    Wd [dm, F].  pos [B]; ctx_k/ctx_v: per sequence [L_b, hkv, D] committed
    rows of this layer's cache; draft_k/draft_v: per sequence [i - 1, hkv, D]
    draft rows written by the earlier steps.
    Returns (x_new [B, dm], k_row [B, hkv, D], v_row [B, hkv, D], t) where t
    holds the bf16-rounded intermediates a, q, k, v, o, m, act and x_mid."""
    B = x.shape[0]
    scale = _attn.default_scale(D) if scale is None else scale
    a = bf16_round(rms_norm(x, P["g_attn"]))
    qkv = a @ P["Wqkv"].T
    q = qkv[:, :hq * D].reshape(B, hq, D)
    k = qkv[:, hq * D:(hq + hkv) * D].reshape(B, hkv, D)
    v = qkv[:, (hq + hkv) * D:].reshape(B, hkv, D)
    pos = np.asarray(pos)
    q = bf16_round(rope(rms_norm(q, P["g_q"]), pos[:, None]))
    k = bf16_round(rope(rms_norm(k, P["g_k"]), pos[:, None]))
    v = bf16_round(v)
    o = np.zeros((B, hq, D))
    for b in range(B):
        dk = np.concatenate([draft_k[b], k[b][None]], axis=0)
        dv = np.concatenate([draft_v[b], v[b][None]], axis=0)
        o[b], _ = _attn.draft_attention_seq(q[b], ctx_k[b], ctx_v[b], dk, dv, scale)
    ob = bf16_round(o.reshape(B, hq * D))
    x_mid = x + ob @ P["Wo"].T
    m = bf16_round(rms_norm(x_mid, P["g_mlp"]))
    act = bf16_round(silu(m @ P["Wg"].T) * (m @ P["Wu"].T))
    x_new = x_mid + act @ P["Wd"].T
    t = dict(a=a, q=q, k=k, v=v, o=ob, x_mid=x_mid, m=m, act=act)
    return x_new, k, v, t


def draft_step(tokens, W_emb: np.ndarray, layers: list, g_final: np.ndarray, pos, ctx, drafts,
               hq: int, hkv: int, D: int, tau: float):
    """A whole draft step: embedding, the decoder layers, final norm, and the
    dynamic-drafting head (Sec. D.1) with the tied embedding as W_out.

    tokens [B]; W_emb [V, dm]; layers: list of P dicts; ctx: per layer a pair
    (ctx_k, ctx_v) of per-sequence lists; drafts: per layer a pair
    (draft_k, draft_v) of per-sequence lists.  Returns (head outputs of
    drafting.draft_head, h [B, dm], per-layer (k_row, v_row), per-layer
    intermediates)."""
    x = W_emb[np.asarray(tokens)].astype(np.float64)
    rows, inter = [], []
    for l, P in enumerate(layers):
        x, k, v, t = decoder_layer(x, P, pos, ctx[l][0], ctx[l][1], drafts[l][0], drafts[l][1],
                                   hq, hkv, D)
        rows.append((k, v))
        t["x_out"] = x
        inter.append(t)
    h = bf16_round(rms_norm(x, g_final))
    return _drafting.draft_head(h, W_emb, tau), h, rows, inter
