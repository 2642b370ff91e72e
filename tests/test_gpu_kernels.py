"""GPU parity of every C-ABI entry point against the oracle on small seeded
problems that span several tiles, split units and ragged tails: draft and
verify attention (max abs <= 2e-3, max rel <= 1e-2 on |o| > 1e-2), cache
appends and accept/commit (bit-exact), untouched outputs of skipped
sequences, determinism, page-order invariance and device-side error flags."""

import numpy as np
import pytest
import torch

from oracle import accept as OA
from oracle import attention as OAT
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
    """bf16 bits [num_pages, hkv, 16, D] holding rows[b, :nrows[b]]; NaN elsewhere."""
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


CASES = [
    # B, hq, hkv, D, kmax, max_ctx, paged_random, key_scale
    (9, 8, 2, 64, 4, 70, True, 1.0),
    (7, 32, 8, 128, 4, 300, True, 1.0),
    (5, 32, 8, 128, 8, 1100, False, 1.0),
    (4, 16, 16, 128, 16, 200, True, 1.0),
    (4, 16, 8, 64, 2, 500, True, 8.0),
    (3, 64, 8, 128, 4, 100, True, 1.0),
    # few (sequence, KV head) pairs with long contexts: each pair split over
    # many CTAs, G = 8 query heads per KV head
    (9, 8, 1, 128, 4, 3000, True, 1.0),
    (16, 8, 1, 128, 8, 1100, True, 1.0),
    # more than 16 draft rows: the draft rows span two pages (one of them
    # may open the next 128-row tile)
    (6, 32, 8, 128, 24, 300, True, 1.0),
    (4, 8, 8, 128, 31, 150, True, 1.0),
    (6, 16, 8, 64, 20, 200, True, 1.0),
    # head_dim 64 with 72 query rows per KV head: the CUDA-core verify route
    (4, 64, 8, 64, 8, 300, True, 1.0),
    # few pairs, short page tables, <= 32 query rows: the cluster kernel
    # (clusters of 16, 12 or 8 CTAs for up to 7, 8 and 15 pairs on a
    # GB300), with 8, 16, 24 and 32 query rows, two draft pages and x8 keys
    (8, 4, 1, 128, 7, 2000, True, 1.0),
    (2, 16, 2, 128, 3, 900, True, 8.0),
    (3, 8, 4, 128, 7, 1500, False, 1.0),
    (2, 4, 4, 128, 24, 400, True, 1.0),
    (5, 8, 2, 128, 4, 2300, True, 1.0),
]


@pytest.mark.parametrize("case", [c for c in CASES if c[3] == 128])
def test_attention_route(S, case):
    """The cases with few (sequence, KV head) pairs, short page tables and at
    most 32 query rows run on the cluster kernel; the others on the query-rows
    tensor-core kernel (G * W1 <= 128 for every head_dim 128 case here)."""
    B, hq, hkv, D, kmax, max_ctx = case[:6]
    max_pages = -(-(max_ctx + kmax + 1) // 16) + 1       # as gen.small_case
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    for draft in (True, False):
        rows = (hq // hkv) * (1 if draft else kmax + 1)
        route = S.seed_attn_route(cfg, B, draft, max_pages)
        few = B * hkv <= 7 or (B * hkv <= 8 and max_pages + 2 <= 12 * 19) or \
            (B * hkv <= 15 and max_pages + 2 <= 8 * 19)
        if rows <= 32 and few:
            assert route in (8, 12, 16), (case, draft, route)
        else:
            assert route == S.ROUTE_TC_ROWS, (case, draft, route)


def make(S, seed, case):
    B, hq, hkv, D, kmax, max_ctx, rnd_pages, ks = case
    c = gen.small_case(seed, B, hq, hkv, D, kmax, max_ctx, rnd_pages, ks)
    cfg = S.SeedConfig(hq=hq, hkv=hkv, head_dim=D, kmax=kmax)
    c["cfg"] = cfg
    c["num_pages"] = B * c["max_pages"]
    c["pt_dev"] = torch.from_numpy(c["page_table"]).cuda()
    c["ws"] = S.new_workspace(cfg, B)
    c["err"] = torch.zeros(1, dtype=torch.int32, device="cuda")
    c["scale"] = OAT.default_scale(D)
    return c


def kv_for(S, c, nrows):
    k = dev16(paged(c["rows_k"], nrows, c["page_table"], c["num_pages"]))
    v = dev16(paged(c["rows_v"], nrows, c["page_table"], c["num_pages"]))
    return S.PagedKV(k, v, c["pt_dev"])


def run_draft(S, c, kv):
    B, hq, D = c["q_draft"].shape
    out = torch.full((B, hq, D), SENTINEL, device="cuda")
    lse = torch.full((B, hq), SENTINEL, device="cuda")
    S.seed_draft_attn(c["cfg"], dev16(c["q_draft"]), kv, dev16(c["draft_k"]), dev16(c["draft_v"]),
                      torch.from_numpy(c["lens"]).cuda(), torch.from_numpy(c["draft_lens"]).cuda(),
                      out, lse, c["ws"], c["err"])
    torch.cuda.synchronize()
    return out.cpu().numpy(), lse.cpu().numpy()


def run_verify(S, c, kv):
    B, W, hq, D = c["q_verify"].shape
    out = torch.full((B, W, hq, D), SENTINEL, device="cuda")
    lse = torch.full((B, W, hq), SENTINEL, device="cuda")
    S.seed_verify_attn(c["cfg"], dev16(c["q_verify"]), torch.from_numpy(c["n_q"]).cuda(), kv,
                       torch.from_numpy(c["lens"]).cuda(), out, lse, c["ws"], c["err"])
    torch.cuda.synchronize()
    return out.cpu().numpy(), lse.cpu().numpy()


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}_hq{}_hkv{}_D{}_k{}_L{}".format(*c[:6]))
def test_draft_attention_matches_oracle(S, case):
    c = make(S, 1, case)
    out, lse = run_draft(S, c, kv_for(S, c, c["lens"]))
    assert int(c["err"].item()) == 0
    for b in range(case[0]):
        dl, L = int(c["draft_lens"][b]), int(c["lens"][b])
        if dl == 0:
            assert (out[b] == SENTINEL).all() and (lse[b] == SENTINEL).all()
            continue
        o, l = OAT.draft_attention_seq(
            f64(c["q_draft"][b]), f64(c["rows_k"][b, :L]), f64(c["rows_v"][b, :L]),
            f64(c["draft_k"][b, :, :dl].transpose(1, 0, 2)),
            f64(c["draft_v"][b, :, :dl].transpose(1, 0, 2)), c["scale"])
        assert_close(out[b], o, f"draft o b={b} L={L} dl={dl}")
        assert_close(lse[b], l, f"draft lse b={b}")


@pytest.mark.parametrize("case", [(8, 32, 8, 128, 24, 260, True, 1.0),
                                  (8, 16, 8, 64, 20, 260, True, 1.0)],
                         ids=["D128_G4", "D64_G2"])
def test_draft_rows_span_pages_and_tiles(S, case):
    """More than 16 draft rows fill two pages after the cache pages; with 7 or
    15 cache pages the second draft page opens the next 128-row tile."""
    c = make(S, 3, case)
    kmax = case[4]
    c["lens"] = np.array([97, 112, 111, 240, 225, 0, 16, 255], dtype=np.int32)
    c["draft_lens"] = np.minimum(np.array([17, 24, 16, 20, 24, 18, 23, 1]), kmax).astype(np.int32)
    out, lse = run_draft(S, c, kv_for(S, c, c["lens"]))
    assert int(c["err"].item()) == 0
    for b in range(case[0]):
        dl, L = int(c["draft_lens"][b]), int(c["lens"][b])
        o, l = OAT.draft_attention_seq(
            f64(c["q_draft"][b]), f64(c["rows_k"][b, :L]), f64(c["rows_v"][b, :L]),
            f64(c["draft_k"][b, :, :dl].transpose(1, 0, 2)),
            f64(c["draft_v"][b, :, :dl].transpose(1, 0, 2)), c["scale"])
        assert_close(out[b], o, f"draft o b={b} L={L} dl={dl}")
        assert_close(lse[b], l, f"draft lse b={b}")


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}_hq{}_hkv{}_D{}_k{}_L{}".format(*c[:6]))
def test_verify_attention_matches_oracle(S, case):
    c = make(S, 2, case)
    out, lse = run_verify(S, c, kv_for(S, c, c["lens"] + c["n_q"]))
    assert int(c["err"].item()) == 0
    for b in range(case[0]):
        n, L = int(c["n_q"][b]), int(c["lens"][b])
        assert (out[b, n:] == SENTINEL).all() and (lse[b, n:] == SENTINEL).all()
        if n == 0:
            continue
        o, l = OAT.verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                        f64(c["rows_v"][b, :L + n]), L, c["scale"])
        assert_close(out[b, :n], o, f"verify o b={b} L={L} n={n}")
        assert_close(lse[b, :n], l, f"verify lse b={b}")


@pytest.mark.parametrize("nq,dl", [((5, 3, 2), (4, 1, 2)), ((1, 5, 4), (2, 4, 3))])
def test_few_pairs_at_the_page_limit(S, nq, dl):
    """Three sequences x four KV heads (12 pairs, G = 4, k = 4): the cluster
    kernel with clusters of 8 CTAs, one sequence of 149 cache pages (the
    CTAs of its pairs at their 19-page limit), one near 2048 tokens."""
    case = (3, 16, 4, 128, 4, 2370, True, 1.0)
    c = make(S, 4, case)
    assert c["max_pages"] + 2 <= 8 * 19
    c["lens"] = np.array([2370, 2047, 100], dtype=np.int32)
    c["n_q"] = np.array(nq, dtype=np.int32)
    c["draft_lens"] = np.array(dl, dtype=np.int32)
    out, lse = run_verify(S, c, kv_for(S, c, c["lens"] + c["n_q"]))
    assert int(c["err"].item()) == 0
    for b in range(3):
        n, L = int(c["n_q"][b]), int(c["lens"][b])
        assert (out[b, n:] == SENTINEL).all()
        o, l = OAT.verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                        f64(c["rows_v"][b, :L + n]), L, c["scale"])
        assert_close(out[b, :n], o, f"verify o b={b} L={L} n={n}")
        assert_close(lse[b, :n], l, f"verify lse b={b}")
    out, lse = run_draft(S, c, kv_for(S, c, c["lens"]))
    assert int(c["err"].item()) == 0
    for b in range(3):
        d, L = int(c["draft_lens"][b]), int(c["lens"][b])
        o, l = OAT.draft_attention_seq(
            f64(c["q_draft"][b]), f64(c["rows_k"][b, :L]), f64(c["rows_v"][b, :L]),
            f64(c["draft_k"][b, :, :d].transpose(1, 0, 2)),
            f64(c["draft_v"][b, :, :d].transpose(1, 0, 2)), c["scale"])
        assert_close(out[b], o, f"draft o b={b} L={L} dl={d}")
        assert_close(lse[b], l, f"draft lse b={b}")


def spike_rows(c, which, step, log2_gap):
    """Key rows that score log2_gap (in log2 units of the softmax) above a
    typical score for query head G g of KV head g: every step-th visible row
    from position 130 on (past the first 128-key tile), plus, for the draft
    call, the first draft row.  Each is a multiple of that query row."""
    B, hkv, D = c["rows_k"].shape[0], c["rows_k"].shape[2], c["rows_k"].shape[3]
    hq = c["q_draft"].shape[1]
    G = hq // hkv
    lg2e = 1.0 / np.log(2.0)
    for b in range(B):
        L = int(c["lens"][b])
        for g in range(hkv):
            q = f64(c["q_draft"][b, g * G] if which == "draft" else c["q_verify"][b, 0, g * G])
            alpha = log2_gap / (c["scale"] * lg2e * float(q @ q))
            row = gen.f32_to_bf16_bits((alpha * q).astype(np.float32))
            for pos in range(130, L, step):
                c["rows_k"][b, pos, g] = row
            if which == "draft":
                c["draft_k"][b, g, 0] = row


@pytest.mark.parametrize("case", [(10, 32, 8, 128, 4, 1100, True, 1.0),
                                  (10, 16, 8, 64, 2, 900, True, 1.0),
                                  (8, 4, 1, 128, 4, 1100, True, 1.0)],
                         ids=["D128_G4", "D64_G2", "D128_G4_few_pairs"])
@pytest.mark.parametrize("gap", [40.0, 300.0], ids=["gap40", "gap300"])
def test_late_score_spikes_match_oracle(S, case, gap):
    """Scores far above the first tile's maximum, in later tiles and in the
    draft rows: a gap below 64 (log2) stays on the fast path with weights up
    to 2^gap; a gap of 300 takes the exact recomputation of the piece."""
    c = make(S, 3, case)
    spike_rows(c, "draft", 97, gap)
    out, lse = run_draft(S, c, kv_for(S, c, c["lens"]))
    assert int(c["err"].item()) == 0
    for b in range(case[0]):
        dl, L = int(c["draft_lens"][b]), int(c["lens"][b])
        if dl == 0:
            continue
        o, l = OAT.draft_attention_seq(
            f64(c["q_draft"][b]), f64(c["rows_k"][b, :L]), f64(c["rows_v"][b, :L]),
            f64(c["draft_k"][b, :, :dl].transpose(1, 0, 2)),
            f64(c["draft_v"][b, :, :dl].transpose(1, 0, 2)), c["scale"])
        assert_close(out[b], o, f"draft o b={b} L={L} dl={dl}")
        assert_close(lse[b], l, f"draft lse b={b}")
    c = make(S, 4, case)
    spike_rows(c, "verify", 113, gap)
    out, lse = run_verify(S, c, kv_for(S, c, c["lens"] + c["n_q"]))
    assert int(c["err"].item()) == 0
    for b in range(case[0]):
        n, L = int(c["n_q"][b]), int(c["lens"][b])
        if n == 0:
            continue
        o, l = OAT.verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                        f64(c["rows_v"][b, :L + n]), L, c["scale"])
        assert_close(out[b, :n], o, f"verify o b={b} L={L} n={n}")
        assert_close(lse[b, :n], l, f"verify lse b={b}")


def test_deterministic_and_page_order_invariant(S):
    case = (5, 32, 8, 128, 8, 1100, True, 1.0)
    c = make(S, 3, case)
    kv = kv_for(S, c, c["lens"] + c["n_q"])
    o1, l1 = run_verify(S, c, kv)
    for _ in range(3):
        o2, l2 = run_verify(S, c, kv)
        np.testing.assert_array_equal(o1, o2)
        np.testing.assert_array_equal(l1, l2)
    d1 = run_draft(S, c, kv_for(S, c, c["lens"]))
    # same logical rows, identity page order
    c2 = make(S, 3, case[:6] + (False, 1.0))
    for key in ("rows_k", "rows_v", "q_verify", "q_draft", "draft_k", "draft_v", "lens", "n_q",
                "draft_lens"):
        c2[key] = c[key]
    o3, l3 = run_verify(S, c2, kv_for(S, c2, c2["lens"] + c2["n_q"]))
    np.testing.assert_array_equal(o1, o3)
    np.testing.assert_array_equal(l1, l3)
    d3 = run_draft(S, c2, kv_for(S, c2, c2["lens"]))
    np.testing.assert_array_equal(d1[0], d3[0])


def test_kv_append_is_bit_exact(S):
    case = (7, 32, 8, 128, 4, 300, True, 1.0)
    c = make(S, 4, case)
    B, kmax = case[0], case[4]
    kv = kv_for(S, c, c["lens"])
    W = kmax + 1
    k_new = np.stack([c["rows_k"][b, c["lens"][b]:c["lens"][b] + W] for b in range(B)])
    v_new = np.stack([c["rows_v"][b, c["lens"][b]:c["lens"][b] + W] for b in range(B)])
    S.seed_kv_append(c["cfg"], kv, dev16(k_new), dev16(v_new), torch.from_numpy(c["n_q"]).cuda(),
                     torch.from_numpy(c["lens"]).cuda(), c["err"])
    torch.cuda.synchronize()
    assert int(c["err"].item()) == 0
    want = paged(c["rows_k"], c["lens"] + c["n_q"], c["page_table"], c["num_pages"])
    got = kv.k.view(torch.int16).cpu().numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)
    want = paged(c["rows_v"], c["lens"] + c["n_q"], c["page_table"], c["num_pages"])
    np.testing.assert_array_equal(kv.v.view(torch.int16).cpu().numpy().view(np.uint16), want)


def test_draft_append_is_bit_exact(S):
    case = (6, 32, 8, 128, 8, 64, True, 1.0)
    c = make(S, 5, case)
    B, hkv, kmax, D = case[0], case[2], case[4], case[3]
    dk = torch.zeros(B, hkv, kmax, D, dtype=torch.bfloat16, device="cuda")
    dv = torch.zeros_like(dk)
    for i in range(1, kmax + 1):
        dl = np.where(c["draft_lens"] >= i, i, 0).astype(np.int32)
        S.seed_draft_kv_append(c["cfg"], dev16(np.ascontiguousarray(c["draft_k"][:, :, i - 1])),
                               dev16(np.ascontiguousarray(c["draft_v"][:, :, i - 1])),
                               torch.from_numpy(dl).cuda(), dk, dv, c["err"])
    torch.cuda.synchronize()
    assert int(c["err"].item()) == 0
    got_k = dk.view(torch.int16).cpu().numpy().view(np.uint16)
    got_v = dv.view(torch.int16).cpu().numpy().view(np.uint16)
    for b in range(B):
        n = int(c["draft_lens"][b])
        np.testing.assert_array_equal(got_k[b, :, :n], c["draft_k"][b, :, :n])
        np.testing.assert_array_equal(got_v[b, :, :n], c["draft_v"][b, :, :n])
        assert (got_k[b, :, n:] == 0).all()


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("kmax", [1, 4, 8, 16])
def test_accept_commit_is_bit_exact(S, seed, kmax):
    B = 37
    a = gen.accept_case(seed, B, kmax)
    acc, tok, slots, new_lens = OA.accept_commit(a["draft_ids"], a["target_ids"], a["k_b"],
                                                 a["lens"], a["page_table"], 16)
    t = {k: torch.from_numpy(v).cuda() for k, v in a.items() if isinstance(v, np.ndarray)}
    lens = t["lens"].clone()
    g_acc = torch.zeros(B, dtype=torch.int32, device="cuda")
    g_tok = torch.zeros(B, kmax + 1, dtype=torch.int32, device="cuda")
    g_slot = torch.zeros_like(g_tok)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    S.seed_accept_commit(kmax, t["draft_ids"], t["target_ids"], t["k_b"], t["page_table"], 16,
                         lens, g_acc, g_tok, g_slot, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    np.testing.assert_array_equal(g_acc.cpu().numpy(), acc)
    np.testing.assert_array_equal(g_tok.cpu().numpy(), tok)
    np.testing.assert_array_equal(g_slot.cpu().numpy(), slots)
    np.testing.assert_array_equal(lens.cpu().numpy(), new_lens)


@pytest.mark.parametrize("case", [(4, 32, 8, 128, 4, 100, True, 1.0),
                                  (4, 16, 4, 64, 4, 100, True, 1.0),
                                  (3, 16, 4, 128, 4, 100, True, 1.0)],
                         ids=["query_rows_D128", "keys_as_rows_D64", "cluster_D128"])
def test_device_errors_are_flagged_not_fatal(S, case):
    c = make(S, 6, case)
    if case[0] == 3:   # 12 pairs and a short page table: the cluster kernel
        assert S.seed_attn_route(c["cfg"], case[0], False, c["max_pages"]) in (8, 12, 16)
    kv = kv_for(S, c, c["lens"] + c["n_q"])
    B = case[0]
    # negative length / length past capacity
    bad = c["lens"].copy()
    bad[1] = -3
    bad[2] = c["max_pages"] * 16 + 5
    c2 = dict(c, lens=bad)
    run_draft(S, c2, kv)
    assert int(c["err"].item()) & 1
    # page id out of range
    c["err"].zero_()
    pt = c["page_table"].copy()
    pt[0, 0] = c["num_pages"] + 7
    kv2 = S.PagedKV(kv.k, kv.v, torch.from_numpy(pt).cuda())
    c3 = dict(c, pt_dev=kv2.page_table)
    lens = np.full(B, 20, dtype=np.int32)
    run_verify(S, dict(c3, lens=lens), kv2)
    assert int(c["err"].item()) & 8
    # draft length past kmax, n_q past kmax+1
    c["err"].zero_()
    run_draft(S, dict(c, draft_lens=np.full(B, 9, dtype=np.int32)), kv)
    assert int(c["err"].item()) & 2
    c["err"].zero_()
    run_verify(S, dict(c, n_q=np.full(B, 7, dtype=np.int32)), kv)
    assert int(c["err"].item()) & 4
    # k_b past kmax in accept
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    kb = torch.full((B,), 9, dtype=torch.int32, device="cuda")
    ids = torch.zeros(B, 4, dtype=torch.int32, device="cuda")
    tg = torch.zeros(B, 5, dtype=torch.int32, device="cuda")
    lens_t = torch.zeros(B, dtype=torch.int32, device="cuda")
    out = [torch.zeros(B, dtype=torch.int32, device="cuda"),
           torch.zeros(B, 5, dtype=torch.int32, device="cuda"),
           torch.zeros(B, 5, dtype=torch.int32, device="cuda")]
    S.seed_accept_commit(4, ids, tg, kb, c["pt_dev"], 16, lens_t, *out, err)
    torch.cuda.synchronize()
    assert int(err.item()) & 16
    assert (lens_t.cpu().numpy() == 0).all()
    # the context stays usable: a valid call still matches
    c["err"].zero_()
    out_ok, _ = run_verify(S, c, kv)
    assert int(c["err"].item()) == 0 and np.isfinite(out_ok[0, :c["n_q"][0]]).all()


def test_many_short_pieces_repeated(S):
    """Many 1-3 tile sequences: every CTA's range holds several pieces, each
    with its own epilogue, so the hand-offs between the kernel's roles run
    hundreds of times per launch.  Repeated draft and verify launches raise no
    device error and keep matching the oracle."""
    case = (96, 32, 8, 128, 8, 300, True, 1.0)
    c = make(S, 7, case)
    kv_d = kv_for(S, c, c["lens"])
    kv_v = kv_for(S, c, c["lens"] + c["n_q"])
    outs = []
    for rep in range(12):
        outs.append(run_draft(S, c, kv_d) if rep % 2 == 0 else run_verify(S, c, kv_v))
        assert int(c["err"].item()) == 0, f"launch {rep}: device error {int(c['err'].item())}"
    for rep in range(2, 12):
        assert np.array_equal(outs[rep][0], outs[rep - 2][0]), f"launch {rep} differs"
    od, ld = outs[0]
    ov, lv = outs[1]
    for b in range(0, case[0], 5):
        dl, L, n = int(c["draft_lens"][b]), int(c["lens"][b]), int(c["n_q"][b])
        if dl:
            o, l = OAT.draft_attention_seq(
                f64(c["q_draft"][b]), f64(c["rows_k"][b, :L]), f64(c["rows_v"][b, :L]),
                f64(c["draft_k"][b, :, :dl].transpose(1, 0, 2)),
                f64(c["draft_v"][b, :, :dl].transpose(1, 0, 2)), c["scale"])
            assert_close(od[b], o, f"draft o b={b}")
            assert_close(ld[b], l, f"draft lse b={b}")
        if n:
            o, l = OAT.verify_attention_seq(f64(c["q_verify"][b, :n]), f64(c["rows_k"][b, :L + n]),
                                            f64(c["rows_v"][b, :L + n]), L, c["scale"])
            assert_close(ov[b, :n], o, f"verify o b={b}")
            assert_close(lv[b, :n], l, f"verify lse b={b}")
