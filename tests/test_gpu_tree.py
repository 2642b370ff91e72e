"""GPU parity of tree-based verification (Sec. D.1) through the C ABI against
the oracle: tree verify attention (max abs <= 2e-3, max rel <= 1e-2 on
|o| > 1e-2), a chain tree equal bit for bit to the linear verify, the greedy
walk and commit (bit-exact), the compaction of the accepted path's cache rows
(bit-exact) and the device error flags."""

import numpy as np
import pytest
import torch

from oracle import attention as OAT
from oracle import tree as OT
from workloads import gen

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2
SENTINEL = 12345.0


@pytest.fixture(scope="module")
def S():
    assert torch.cuda.is_available(), "GPU test run without a GPU"
    from paper_2609_36590_gb300 import build
    build.build()
    import paper_2609_36590_gb300 as s
    return s


def dev16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def f64(bits):
    return gen.bf16_bits_to_f64(bits)


def paged(rows, nrows, pt, num_pages):
    B, _, hkv, D = rows.shape
    cache = np.full((num_pages, hkv, 16, D), gen.BF16_NAN, dtype=np.uint16)
    for b in range(B):
        pos = np.arange(int(nrows[b]))
        cache[pt[b, pos // 16], :, pos % 16] = rows[b, pos]
    return cache


def assert_close(got, ref, what):
    got = np.asarray(got, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    diff = np.abs(got - ref)
    assert diff.max() <= ATOL, f"{what}: max abs err {diff.max():.3g}"
    big = np.abs(ref) > 1e-2
    if big.any():
        rel = (diff[big] / np.abs(ref[big])).max()
        assert rel <= RTOL, f"{what}: max rel err {rel:.3g}"


def random_trees(g, B, W, allow_empty=True):
    """parent [B, W] (-1 past n), n_nodes [B]; some sequences get no tree."""
    parent = np.full((B, W), -1, dtype=np.int32)
    n_nodes = g.integers(1, W + 1, size=B).astype(np.int32)
    n_nodes[0] = W
    if allow_empty and B >= 3:
        n_nodes[B - 1] = 0
    for b in range(B):
        for i in range(1, int(n_nodes[b])):
            # mostly bushy near the root, sometimes a long chain
            parent[b, i] = i - 1 if g.random() < 0.3 else int(g.integers(0, i))
    return parent, n_nodes


def anc_of(parent, n_nodes):
    B, W = parent.shape
    anc = np.zeros((B, W), dtype=np.uint32)
    for b in range(B):
        n = int(n_nodes[b])
        if n:
            anc[b, :n] = OT.ancestor_masks(parent[b, :n])
    return anc


TREE_CASES = [
    # B, hq, hkv, D, kmax, max_ctx, paged_random
    (6, 32, 8, 128, 7, 300, True),
    (4, 32, 8, 128, 31, 1100, False),
    (5, 16, 16, 128, 12, 2000, True),
    (3, 64, 8, 128, 15, 500, True),
    (9, 8, 1, 128, 7, 3000, True),     # few pairs, long contexts: pairs split over many CTAs
    (6, 8, 4, 64, 7, 500, True),       # head_dim 64, 16 rows: the keys-as-rows kernel
]


@pytest.mark.parametrize("case", TREE_CASES, ids=lambda c: "B{}_hq{}_hkv{}_k{}_L{}".format(
    c[0], c[1], c[2], c[4], c[5]))
def test_tree_verify_matches_oracle(S, case):
    B, hq, hkv, D, kmax, max_ctx, rnd = case
    c = gen.small_case(21, B, hq, hkv, D, kmax, max_ctx, rnd, 1.0)
    g = np.random.default_rng(5)
    W = kmax + 1
    parent, n_nodes = random_trees(g, B, W)
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    num_pages = B * c["max_pages"]
    lens = c["lens"]
    kv = S.PagedKV(dev16(paged(c["rows_k"], lens + n_nodes, c["page_table"], num_pages)),
                   dev16(paged(c["rows_v"], lens + n_nodes, c["page_table"], num_pages)),
                   torch.from_numpy(c["page_table"]).cuda())
    out = torch.full((B, W, hq, D), SENTINEL, device="cuda")
    lse = torch.full((B, W, hq), SENTINEL, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    anc = torch.from_numpy(anc_of(parent, n_nodes).view(np.int32)).cuda()
    S.seed_tree_verify_attn(cfg, dev16(c["q_verify"]), torch.from_numpy(n_nodes).cuda(), anc, kv,
                            torch.from_numpy(lens).cuda(), out, lse, S.new_workspace(cfg, B), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    out, lse = out.cpu().numpy(), lse.cpu().numpy()
    scale = OAT.default_scale(D)
    for b in range(B):
        n, L = int(n_nodes[b]), int(lens[b])
        assert (out[b, n:] == SENTINEL).all() and (lse[b, n:] == SENTINEL).all()
        if n == 0:
            continue
        o, l = OT.tree_verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                            f64(c["rows_v"][b, :L + n]), L, parent[b, :n], scale)
        assert_close(out[b, :n], o, f"tree o b={b} L={L} n={n}")
        assert_close(lse[b, :n], l, f"tree lse b={b}")


def test_chain_tree_is_bitwise_the_linear_verify(S):
    B, hq, hkv, D, kmax = 5, 32, 8, 128, 8
    c = gen.small_case(22, B, hq, hkv, D, kmax, 900, True, 8.0)
    W = kmax + 1
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    num_pages = B * c["max_pages"]
    n_q = c["n_q"]
    kv = S.PagedKV(dev16(paged(c["rows_k"], c["lens"] + n_q, c["page_table"], num_pages)),
                   dev16(paged(c["rows_v"], c["lens"] + n_q, c["page_table"], num_pages)),
                   torch.from_numpy(c["page_table"]).cuda())
    chain = np.tile(np.arange(-1, W - 1, dtype=np.int32), (B, 1))
    anc = torch.from_numpy(anc_of(chain, np.full(B, W)).view(np.int32)).cuda()
    q, nq, lens = dev16(c["q_verify"]), torch.from_numpy(n_q).cuda(), torch.from_numpy(c["lens"]).cuda()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = S.new_workspace(cfg, B)
    o1 = torch.full((B, W, hq, D), SENTINEL, device="cuda")
    l1 = torch.full((B, W, hq), SENTINEL, device="cuda")
    o2, l2 = o1.clone(), l1.clone()
    S.seed_verify_attn(cfg, q, nq, kv, lens, o1, l1, ws, err)
    S.seed_tree_verify_attn(cfg, q, nq, anc, kv, lens, o2, l2, ws, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def tree_inputs(g, B, W, vocab):
    parent, n_nodes = random_trees(g, B, W, allow_empty=False)
    tok = np.full((B, W), -1, dtype=np.int32)
    for b in range(B):
        for i in range(int(n_nodes[b])):
            tok[b, i] = int(g.integers(0, vocab))
    target = g.integers(0, vocab, size=(B, W)).astype(np.int32)
    return parent, n_nodes, tok, target


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("kmax", [3, 12, 31])
def test_tree_accept_is_bit_exact(S, seed, kmax):
    g = np.random.default_rng(300 + seed)
    B, W, ps = 40, kmax + 1, 16
    parent, n_nodes, tok, target = tree_inputs(g, B, W, vocab=3)
    max_pages = 8
    pt = g.permutation(B * max_pages).reshape(B, max_pages).astype(np.int32)
    lens = g.integers(0, max_pages * ps - W, size=B).astype(np.int32)
    acc_o, tok_o, path_o, slot_o, lens_o = OT.tree_accept_commit(tok, parent, n_nodes, target,
                                                                 lens, pt, ps)
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    ctx = d(lens)
    accepted = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    tokens, path, slots = (torch.full((B, W), -7, dtype=torch.int32, device="cuda")
                           for _ in range(3))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    S.seed_tree_accept_commit(kmax, d(tok), d(parent), d(n_nodes), d(target), d(pt), ps, ctx,
                              accepted, tokens, path, slots, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    np.testing.assert_array_equal(accepted.cpu().numpy(), acc_o)
    np.testing.assert_array_equal(tokens.cpu().numpy(), tok_o)
    np.testing.assert_array_equal(path.cpu().numpy(), path_o)
    np.testing.assert_array_equal(slots.cpu().numpy(), slot_o)
    np.testing.assert_array_equal(ctx.cpu().numpy(), lens_o)
    assert (acc_o > 0).any()


def test_tree_accept_flags_bad_trees(S):
    B, kmax = 3, 4
    W = kmax + 1
    tok = np.zeros((B, W), dtype=np.int32)
    target = np.zeros((B, W), dtype=np.int32)
    parent = np.tile(np.arange(-1, W - 1, dtype=np.int32), (B, 1))
    parent[1, 3] = 3                      # a node that is its own parent
    n_nodes = np.array([W, W, W + 1], dtype=np.int32)   # too many nodes in sequence 2
    pt = np.arange(B * 4, dtype=np.int32).reshape(B, 4)
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    ctx = d(np.array([5, 6, 7], dtype=np.int32))
    accepted = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    tokens, path, slots = (torch.full((B, W), -7, dtype=torch.int32, device="cuda")
                           for _ in range(3))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    S.seed_tree_accept_commit(kmax, d(tok), d(parent), d(n_nodes), d(target), d(pt), 16, ctx,
                              accepted, tokens, path, slots, err)
    torch.cuda.synchronize()
    e = int(err.item())
    assert e & 128 and e & 4
    assert ctx.cpu().numpy().tolist() == [5 + W, 6, 7]   # bad sequences left unchanged
    assert accepted.cpu().numpy().tolist()[1:] == [-7, -7]


@pytest.mark.parametrize("seed", range(3))
def test_tree_compaction_is_bit_exact(S, seed):
    g = np.random.default_rng(400 + seed)
    B, hq, hkv, D, kmax, ps = 12, 16, 8, 128, 15, 16
    W = kmax + 1
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    parent, n_nodes, tok, target = tree_inputs(g, B, W, vocab=2)
    max_pages = 12
    pt = g.permutation(B * max_pages).reshape(B, max_pages).astype(np.int32)
    lens = g.integers(0, max_pages * ps - W, size=B).astype(np.int32)
    n_rows = max_pages * ps
    rows_k = gen.f32_to_bf16_bits(g.standard_normal((B, n_rows, hkv, D)).astype(np.float32))
    rows_v = gen.f32_to_bf16_bits(g.standard_normal((B, n_rows, hkv, D)).astype(np.float32))
    full = np.full(B, n_rows)
    kc = dev16(paged(rows_k, full, pt, B * max_pages))
    vc = dev16(paged(rows_v, full, pt, B * max_pages))
    kv = S.PagedKV(kc, vc, torch.from_numpy(pt).cuda())
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    ctx = d(lens)
    accepted = torch.zeros(B, dtype=torch.int32, device="cuda")
    tokens, path, slots = (torch.zeros((B, W), dtype=torch.int32, device="cuda") for _ in range(3))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    S.seed_tree_accept_commit(kmax, d(tok), d(parent), d(n_nodes), d(target), kv.page_table, ps,
                              ctx, accepted, tokens, path, slots, err)
    S.seed_tree_kv_compact(cfg, kv, path, accepted, ctx, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    acc_o, _, path_o, _, _ = OT.tree_accept_commit(tok, parent, n_nodes, target, lens, pt, ps)
    kbits = kc.view(torch.int16).cpu().numpy().view(np.uint16)
    vbits = vc.view(torch.int16).cpu().numpy().view(np.uint16)
    moved = 0
    for b in range(B):
        L, n = int(lens[b]), int(acc_o[b])
        for rows, bits in ((rows_k, kbits), (rows_v, vbits)):
            want = OT.compact_path(rows[b], L, path_o[b], n)
            pos = np.arange(L + n + 1)
            got = bits[pt[b, pos // ps], :, pos % ps]
            np.testing.assert_array_equal(got, want[:L + n + 1])
        moved += int((path_o[b, 1:n + 1] != np.arange(1, n + 1)).sum())
    assert moved > 0
