"""Pins of the draft-step oracle (Sec. 4.1 drafting with the model's last
layers; the layer in the Qwen3 form the paper's models use), against things
other than itself:
* bf16 rounding, RMS norm and SiLU against PyTorch's own routines;
* RoPE against a complex-number formulation, plus its closed forms (position
  0 is the identity, pairs keep their norm, rotations compose);
* the whole decoder layer against an independent float64 PyTorch
  formulation (F.rms_norm, complex RoPE, scaled_dot_product_attention with
  grouped heads, F.silu), with the same bf16 rounding points;
* special cases: a single visible row returns its V; zero output and MLP
  projections leave the residual stream unchanged;
* the draft step equals its parts (embedding, layers, final norm, head)."""

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import draft_step as DS
from oracle import drafting as OD


def test_bf16_round_matches_torch():
    g = np.random.default_rng(0)
    x = np.concatenate([g.standard_normal(5000) * 10.0 ** g.integers(-30, 30, 5000),
                        [0.0, -0.0, 1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 3.0e38, -3.4e38,
                         np.inf, -np.inf, 1e-40]])
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    got = DS.bf16_round(x)
    np.testing.assert_array_equal(got, want)
    assert np.isnan(DS.bf16_round(np.array([np.nan]))[0])


def test_rms_norm_and_silu_match_torch():
    g = np.random.default_rng(1)
    x = g.standard_normal((7, 64)) * 3.0
    w = g.standard_normal(64)
    want = F.rms_norm(torch.from_numpy(x), (64,), torch.from_numpy(w), eps=DS.EPS).numpy()
    np.testing.assert_allclose(DS.rms_norm(x, w), want, rtol=1e-13, atol=0)
    np.testing.assert_allclose(DS.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-13, atol=1e-15)


def rope_complex(x, pos, theta):
    D = x.shape[-1]
    half = D // 2
    z = x[..., :half] + 1j * x[..., half:]
    inv = 1.0 / theta ** (np.arange(0, D, 2) / D)
    z = z * np.exp(1j * np.asarray(pos, dtype=np.float64)[..., None] * inv)
    return np.concatenate([z.real, z.imag], axis=-1)


def test_rope_complex_form_and_closed_forms():
    g = np.random.default_rng(2)
    x = g.standard_normal((5, 3, 128))
    pos = np.array([0, 1, 7, 4095, 123456])
    r = DS.rope(x, pos[:, None])
    np.testing.assert_allclose(r, rope_complex(x, pos[:, None], DS.ROPE_THETA), rtol=0, atol=1e-9)
    np.testing.assert_allclose(r[0], x[0], rtol=0, atol=0)                 # position 0
    pair = lambda y: y[..., :64] ** 2 + y[..., 64:] ** 2
    np.testing.assert_allclose(pair(r), pair(x), rtol=1e-12)               # rotation keeps norms
    np.testing.assert_allclose(DS.rope(DS.rope(x, 11), 31), DS.rope(x, 42), rtol=0, atol=1e-11)


def make_layer(g, dm, hq, hkv, D, F_):
    b = lambda shape, s: DS.bf16_round(g.standard_normal(shape) * s)
    return dict(g_attn=b(dm, 1.0) + 1.0, Wqkv=b(((hq + 2 * hkv) * D, dm), dm ** -0.5),
                g_q=b(D, 0.2) + 1.0, g_k=b(D, 0.2) + 1.0, Wo=b((dm, hq * D), (hq * D) ** -0.5),
                g_mlp=b(dm, 0.2) + 1.0, Wg=b((F_, dm), dm ** -0.5), Wu=b((F_, dm), dm ** -0.5),
                Wd=b((dm, F_), F_ ** -0.5))


def torch_layer(x, P, pos, ctx_k, ctx_v, draft_k, draft_v, hq, hkv, D):
    """The same layer written with PyTorch routines (float64)."""
    T = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    r16 = lambda t: t.to(torch.float32).to(torch.bfloat16).to(torch.float64)
    B, dm = x.shape
    x = T(x)
    a = r16(F.rms_norm(x, (dm,), T(P["g_attn"]), eps=DS.EPS))
    qkv = a @ T(P["Wqkv"]).T
    q = qkv[:, :hq * D].reshape(B, hq, D)
    k = qkv[:, hq * D:(hq + hkv) * D].reshape(B, hkv, D)
    v = qkv[:, (hq + hkv) * D:].reshape(B, hkv, D)

    def rope_t(t):
        z = torch.complex(t[..., :D // 2], t[..., D // 2:])
        inv = 1.0 / DS.ROPE_THETA ** (torch.arange(0, D, 2, dtype=torch.float64) / D)
        ang = T(pos)[:, None, None] * inv
        z = z * torch.polar(torch.ones_like(ang), ang)
        return torch.cat([z.real, z.imag], dim=-1)

    q = r16(rope_t(F.rms_norm(q, (D,), T(P["g_q"]), eps=DS.EPS)))
    k = r16(rope_t(F.rms_norm(k, (D,), T(P["g_k"]), eps=DS.EPS)))
    v = r16(v)
    o = torch.zeros(B, hq, D, dtype=torch.float64)
    for b in range(B):
        K = torch.cat([T(ctx_k[b]), T(draft_k[b]), k[b][None]], 0).permute(1, 0, 2)
        V = torch.cat([T(ctx_v[b]), T(draft_v[b]), v[b][None]], 0).permute(1, 0, 2)
        o[b] = F.scaled_dot_product_attention(q[b][:, None], K, V, enable_gqa=True)[:, 0]
    x = x + r16(o.reshape(B, hq * D)) @ T(P["Wo"]).T
    m = r16(F.rms_norm(x, (dm,), T(P["g_mlp"]), eps=DS.EPS))
    act = r16(F.silu(m @ T(P["Wg"]).T) * (m @ T(P["Wu"]).T))
    return (x + act @ T(P["Wd"]).T).numpy(), k.numpy(), v.numpy()


def layer_inputs(g, B, hkv, D, lens, i):
    ctx_k = [g.standard_normal((L, hkv, D)) for L in lens]
    ctx_v = [g.standard_normal((L, hkv, D)) for L in lens]
    dk = [g.standard_normal((i - 1, hkv, D)) for _ in lens]
    dv = [g.standard_normal((i - 1, hkv, D)) for _ in lens]
    return ctx_k, ctx_v, dk, dv


@pytest.mark.parametrize("seed,i", [(0, 1), (1, 3), (2, 5)])
def test_layer_matches_torch_formulation(seed, i):
    g = np.random.default_rng(10 + seed)
    B, dm, hq, hkv, D, F_ = 3, 48, 4, 2, 16, 40
    P = make_layer(g, dm, hq, hkv, D, F_)
    x = g.standard_normal((B, dm))
    lens = [0, 5, 17][:B]
    ctx_k, ctx_v, dk, dv = layer_inputs(g, B, hkv, D, lens, i)
    pos = np.array(lens) + i - 1
    got, k, v, _ = DS.decoder_layer(x, P, pos, ctx_k, ctx_v, dk, dv, hq, hkv, D)
    want, wk, wv = torch_layer(x, P, pos, ctx_k, ctx_v, dk, dv, hq, hkv, D)
    np.testing.assert_allclose(k, wk, rtol=0, atol=1e-12)
    np.testing.assert_allclose(v, wv, rtol=0, atol=0)
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-10)


def test_single_row_returns_v_and_zero_projections_keep_x():
    g = np.random.default_rng(3)
    B, dm, hq, hkv, D, F_ = 2, 32, 4, 2, 16, 24
    P = make_layer(g, dm, hq, hkv, D, F_)
    x = g.standard_normal((B, dm))
    empty = [np.zeros((0, hkv, D))] * B
    _, k, v, t = DS.decoder_layer(x, P, [0, 0], empty, empty, empty, empty, hq, hkv, D)
    # one visible row (its own): each query head returns its KV head's v
    o = t["o"].reshape(B, hq, D)
    for h in range(hq):
        np.testing.assert_array_equal(o[:, h], v[:, h // (hq // hkv)])
    Z = dict(P, Wo=np.zeros_like(P["Wo"]), Wd=np.zeros_like(P["Wd"]))
    x2, _, _, t2 = DS.decoder_layer(x, Z, [3, 9], empty, empty, empty, empty, hq, hkv, D)
    np.testing.assert_array_equal(x2, x)
    Z = dict(P, Wd=np.zeros_like(P["Wd"]))
    x3, _, _, t3 = DS.decoder_layer(x, Z, [3, 9], empty, empty, empty, empty, hq, hkv, D)
    np.testing.assert_array_equal(x3, t3["x_mid"])


def test_draft_step_is_its_parts():
    g = np.random.default_rng(4)
    B, dm, hq, hkv, D, F_, V = 2, 32, 4, 2, 16, 24, 300
    layers = [make_layer(g, dm, hq, hkv, D, F_) for _ in range(2)]
    W = DS.bf16_round(g.standard_normal((V, dm)))
    g_final = DS.bf16_round(g.standard_normal(dm) * 0.2 + 1.0)
    tokens = np.array([7, 123])
    lens = [4, 9]
    ctx, drafts = [], []
    for _ in range(2):
        ck, cv, dk, dv = layer_inputs(g, B, hkv, D, lens, 2)
        ctx.append((ck, cv))
        drafts.append((dk, dv))
    pos = np.array(lens) + 1
    (ids, probs, p0, k, stop, lse), h, rows, inter = DS.draft_step(
        tokens, W, layers, g_final, pos, ctx, drafts, hq, hkv, D, 0.7)
    x = W[tokens]
    for l in range(2):
        x, kr, vr, _ = DS.decoder_layer(x, layers[l], pos, *ctx[l], *drafts[l], hq, hkv, D)
        np.testing.assert_array_equal(kr, rows[l][0])
    hh = DS.bf16_round(DS.rms_norm(x, g_final))
    np.testing.assert_array_equal(hh, h)
    want = OD.draft_head(hh, W, 0.7)
    np.testing.assert_array_equal(ids, want[0])
    np.testing.assert_array_equal(lse, want[5])
