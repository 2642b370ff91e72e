"""GPU parity of the dynamic-drafting head (Sec. D.1) through the C ABI
against the oracle: log-sum-exp and top-10 probabilities within the parity
tolerance, top-10 ids exact wherever the oracle's logits are separated by more
than the float32 noise (and otherwise within that noise of the oracle's value
at the same rank), and the sibling count and stop flag exactly as the rule
gives them on the kernel's own p0 (and as the oracle's wherever p0 is not at
a threshold)."""

import numpy as np
import pytest
import torch

from oracle import drafting as OD
from workloads import gen

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


@pytest.fixture(scope="module")
def S():
    assert torch.cuda.is_available(), "GPU test run without a GPU"
    from paper_2609_36590_gb300 import build
    build.build()
    import paper_2609_36590_gb300 as s
    return s


def bf16(g, shape, scale=1.0):
    return gen.f32_to_bf16_bits((g.standard_normal(shape) * scale).astype(np.float32))


def dev16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def run(S, hb, wb, tau):
    B, V = hb.shape[0], wb.shape[0]
    ids = torch.full((B, 10), -9, dtype=torch.int32, device="cuda")
    probs = torch.full((B, 10), -9.0, device="cuda")
    n_sib = torch.full((B,), -9, dtype=torch.int32, device="cuda")
    stop = torch.full((B,), -9, dtype=torch.int32, device="cuda")
    lse = torch.full((B,), -9.0, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    S.seed_draft_head_topk(dev16(hb), dev16(wb), tau, ids, probs, n_sib, stop, lse,
                           S.new_draft_head_workspace(B), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return (ids.cpu().numpy(), probs.cpu().numpy(), n_sib.cpu().numpy(), stop.cpu().numpy(),
            lse.cpu().numpy())


def rule(p0, tau):
    return (np.where(p0 > 0.95, 1, np.where(p0 > 0.8, 3, np.where(p0 > 0.5, 5, 10))),
            (p0 <= tau).astype(np.int32))


def check(hb, wb, tau, got, rows=None):
    ids, probs, n_sib, stop, lse = got
    h = gen.bf16_bits_to_f64(hb)
    W = gen.bf16_bits_to_f64(wb)
    rows = range(h.shape[0]) if rows is None else rows
    sub = np.array(list(rows))
    o_ids, o_probs, o_p0, o_k, o_stop, o_lse = OD.draft_head(h[sub], W, tau)
    z = h[sub] @ W.T
    k_rule, s_rule = rule(probs[sub, 0].astype(np.float64), tau)
    assert (n_sib[sub] == k_rule).all() and (stop[sub] == s_rule).all()
    for r, b in enumerate(sub):
        assert abs(lse[b] - o_lse[r]) <= ATOL, f"lse b={b}: {lse[b]} vs {o_lse[r]}"
        eps = 1e-4 * max(1.0, np.abs(z[r]).max())
        zs = np.sort(z[r])[::-1]
        assert len(set(ids[b].tolist())) == 10
        for k in range(10):
            zg = z[r, ids[b, k]]
            assert abs(zg - zs[k]) <= eps, f"b={b} rank {k}: logit {zg} vs {zs[k]}"
            separated = (k == 0 or zs[k - 1] - zs[k] > eps) and (k == 9 or zs[k] - zs[k + 1] > eps)
            if separated:
                assert ids[b, k] == o_ids[r, k], f"b={b} rank {k}"
        p_or = np.exp(z[r, ids[b]] - o_lse[r])
        diff = np.abs(probs[b] - p_or)
        assert diff.max() <= ATOL, f"probs b={b}: {diff.max()}"
        big = p_or > 1e-2
        if big.any():
            assert (diff[big] / p_or[big]).max() <= RTOL
        p0 = o_p0[r]
        if min(abs(p0 - t) for t in (0.5, 0.8, 0.95, tau)) > 1e-4:
            assert n_sib[b] == o_k[r] and stop[b] == o_stop[r]


CASES = [
    # B, d, V, tau
    (1, 64, 1000, 0.7),
    (5, 512, 40000, 0.7),
    (37, 256, 9000, 0.5),
    (128, 128, 5000, 0.7),
    (33, 192, 3000, 0.7),       # a second chunk of 32 sequences holding one
    (65, 128, 20000, 0.3),      # four chunks, the last two partly or wholly empty
    (96, 320, 7001, 0.9),
    (16, 64, 128 * 152 * 2 + 37, 0.7),   # two to three tiles per CTA, ragged last tile
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}_d{}_V{}".format(*c[:3]))
def test_head_matches_oracle(S, case):
    B, d, V, tau = case
    g = np.random.default_rng(B * 7 + d)
    # per-sequence logit scales from flat to peaked distributions
    scales = np.geomspace(0.05, 12.0, B) if B > 1 else np.array([3.0])
    hb = gen.f32_to_bf16_bits((g.standard_normal((B, d)) * scales[:, None]).astype(np.float32))
    wb = bf16(g, (V, d), 1.0 / np.sqrt(d))
    got = run(S, hb, wb, tau)
    check(hb, wb, tau, got)
    k = got[2]
    assert len(set(k.tolist())) >= (3 if B >= 32 else 1)   # several branches of the rule seen


def test_head_at_4b_scale_sampled(S):
    """Qwen3-4B-sized head (d_model 2560, vocab 151936), batch 64; eight
    sequences checked against the oracle."""
    B, d, V, tau = 64, 2560, 151936, 0.7
    g = np.random.default_rng(77)
    scales = np.geomspace(0.05, 12.0, B)
    hb = gen.f32_to_bf16_bits((g.standard_normal((B, d)) * scales[:, None]).astype(np.float32))
    wb = bf16(g, (V, d), 1.0 / np.sqrt(d))
    got = run(S, hb, wb, tau)
    check(hb, wb, tau, got, rows=[0, 9, 20, 31, 40, 50, 58, 63])


def test_head_is_deterministic(S):
    B, d, V = 16, 256, 20000
    g = np.random.default_rng(5)
    hb = bf16(g, (B, d), 2.0)
    wb = bf16(g, (V, d), 1.0 / np.sqrt(d))
    a = run(S, hb, wb, 0.7)
    b = run(S, hb, wb, 0.7)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_head_equal_logits_keep_the_lower_id(S):
    """Rows of W that are bit-identical give bit-identical logits on any CTA
    and row quarter; the top list orders them by id (the oracle's rule)."""
    B, d, V = 3, 128, 50000
    g = np.random.default_rng(11)
    hb = bf16(g, (B, d), 1.0)
    wb = bf16(g, (V, d), 1.0 / np.sqrt(d))
    h = gen.bf16_bits_to_f32(hb).astype(np.float64)
    dup = [40001, 77, 23456, 129, 49999, 12800]        # spread over tiles, CTAs and quarters
    for b in range(B):
        # a row aligned with h[b] is the clear maximum for sequence b
        row = gen.f32_to_bf16_bits((h[b] / np.linalg.norm(h[b]) * 4.0).astype(np.float32))
        for r in dup[2 * b:2 * b + 2]:
            wb[r] = row
    got = run(S, hb, wb, 0.7)
    ids = got[0]
    for b in range(B):
        pair = sorted(dup[2 * b:2 * b + 2])
        assert ids[b, :2].tolist() == pair
    check(hb, wb, 0.7, got)
