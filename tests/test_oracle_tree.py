"""Pins of the tree-verification oracle (Sec. D.1), against things other than
itself:
* a chain tree is the linear verify pass (attention and acceptance);
* each node's output equals the linear verify of its own ancestral path, built
  independently from the parent array (the paper's claim that the tree mask
  reproduces each branch's own autoregressive evaluation);
* a scalar pure-Python loop for one node;
* the greedy walk equals a brute-force search over all root paths;
* hand-worked walks, including the tie rule;
* end to end: SEED with draft trees and tree verification emits exactly the
  greedy AR stream of a toy model, and two planted mistakes (siblings that see
  each other; no compaction of the accepted path) break that equality."""

import itertools
import math

import numpy as np
import pytest

from oracle import accept as OA
from oracle import attention as OAT
from oracle import tree as OT
from oracle.toy_model import ToyLM, seed_tree_greedy


def random_tree(g, n):
    parent = [-1] + [int(g.integers(0, i)) for i in range(1, n)]
    return np.array(parent)


def path_of(parent, j):
    p = []
    while j >= 0:
        p.append(j)
        j = int(parent[j]) if j > 0 else -1
    return p[::-1]


def test_masks_and_depths_by_hand():
    #      0
    #    / | \
    #   1  2  3
    #  / \     \
    # 4   5     6
    parent = [-1, 0, 0, 0, 1, 1, 3]
    assert OT.depths(parent).tolist() == [0, 1, 1, 1, 2, 2, 2]
    anc = OT.ancestor_masks(parent).tolist()
    assert anc == [0b1, 0b11, 0b101, 0b1001, 0b10011, 0b100011, 0b1001001]


@pytest.mark.parametrize("seed", range(3))
def test_chain_tree_is_linear_verify(seed):
    g = np.random.default_rng(seed)
    n, L, Hq, Hkv, D = 5, 7, 4, 2, 8
    q = g.standard_normal((n, Hq, D))
    K = g.standard_normal((L + n, Hkv, D))
    V = g.standard_normal((L + n, Hkv, D))
    o1, l1 = OT.tree_verify_attention_seq(q, K, V, L, np.arange(-1, n - 1), 0.3)
    o2, l2 = OAT.verify_attention_seq(q, K, V, L, 0.3)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_node_equals_linear_verify_of_its_path(seed):
    g = np.random.default_rng(10 + seed)
    n, L, Hq, Hkv, D = 9, 6, 4, 2, 8
    parent = random_tree(g, n)
    q = g.standard_normal((n, Hq, D))
    K = g.standard_normal((L + n, Hkv, D))
    V = g.standard_normal((L + n, Hkv, D))
    o, lse = OT.tree_verify_attention_seq(q, K, V, L, parent, 0.25)
    for j in range(n):
        p = path_of(parent, j)
        rows = [*range(L)] + [L + a for a in p]
        oc, lc = OAT.verify_attention_seq(q[p], K[rows], V[rows], L, 0.25)
        np.testing.assert_allclose(o[j], oc[-1], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[j], lc[-1], rtol=0, atol=1e-12)


def test_scalar_brute_force_one_node():
    g = np.random.default_rng(3)
    n, L, D = 6, 4, 5
    parent = np.array([-1, 0, 0, 1, 2, 3])
    q = g.standard_normal((n, 1, D))
    K = g.standard_normal((L + n, 1, D))
    V = g.standard_normal((L + n, 1, D))
    o, lse = OT.tree_verify_attention_seq(q, K, V, L, parent, 0.5)
    j = 5                                     # path 0 -> 1 -> 3 -> 5
    rows = list(range(L)) + [L + 0, L + 1, L + 3, L + 5]
    s = [0.5 * math.fsum(q[j, 0, d] * K[r, 0, d] for d in range(D)) for r in rows]
    m = max(s)
    w = [math.exp(x - m) for x in s]
    z = math.fsum(w)
    ref = [math.fsum(w[i] * V[rows[i], 0, d] for i in range(len(rows))) / z for d in range(D)]
    np.testing.assert_allclose(o[j, 0], ref, rtol=0, atol=1e-12)
    assert abs(lse[j, 0] - (m + math.log(z))) < 1e-12


def test_chain_accept_is_linear_accept():
    g = np.random.default_rng(4)
    B, k = 6, 5
    pt = np.arange(B * 8, dtype=np.int32).reshape(B, 8)
    lens = g.integers(0, 20, size=B)
    target = g.integers(0, 3, size=(B, k + 1))
    drafts = g.integers(0, 3, size=(B, k))
    tok = np.concatenate([np.full((B, 1), 9), drafts], axis=1)
    parent = np.tile(np.arange(-1, k), (B, 1))
    a1, t1, path, s1, L1 = OT.tree_accept_commit(tok, parent, [k + 1] * B, target, lens, pt, 4)
    a2, t2, s2, L2 = OA.accept_commit(drafts, target, [k] * B, lens, pt, 4)
    np.testing.assert_array_equal(a1, a2)
    np.testing.assert_array_equal(t1, t2)
    np.testing.assert_array_equal(s1, s2)
    np.testing.assert_array_equal(L1, L2)
    for b in range(B):
        assert path[b, :a1[b] + 1].tolist() == list(range(a1[b] + 1))


def brute_force_walk(tok, parent, target, n):
    """All nodes whose every edge p -> c has tok[c] == target[p]; with
    distinct sibling tokens they form one chain from the root."""
    ok = []
    for c in range(n):
        p = path_of(parent, c)
        if all(tok[p[i + 1]] == target[p[i]] for i in range(len(p) - 1)):
            ok.append(p)
    return max(ok, key=len)


@pytest.mark.parametrize("seed", range(30))
def test_walk_matches_brute_force(seed):
    g = np.random.default_rng(100 + seed)
    n, V = int(g.integers(1, 16)), 4
    parent = random_tree(g, n)
    tok = np.zeros(n, dtype=np.int64)
    for c in range(1, n):
        used = {int(tok[s]) for s in range(1, c) if parent[s] == parent[c]}
        free = [t for t in range(V + n) if t not in used]
        tok[c] = free[int(g.integers(0, min(len(free), V)))]
    target = g.integers(0, V, size=n)
    acc, tokens, path, _, _ = OT.tree_accept_commit(
        tok[None], parent[None], [n], target[None], [0], np.arange(8)[None], 16)
    want = brute_force_walk(tok, parent, target, n)
    m = int(acc[0])
    assert path[0, :m + 1].tolist() == want
    assert tokens[0, :m].tolist() == [int(tok[c]) for c in want[1:]]
    assert tokens[0, m] == target[want[-1]]


def test_walk_by_hand_and_tie_rule():
    # root 0 -> {1: tok 5, 2: tok 7}; 1 -> {3: tok 2}; 2 -> {4: tok 2}
    parent = np.array([[-1, 0, 0, 1, 2]])
    tok = np.array([[9, 5, 7, 2, 2]])
    pt = np.arange(4)[None]
    # target at root 7 -> node 2; target at 2 is 2 -> node 4; bonus target[4] = 8
    target = np.array([[7, 0, 2, 1, 8]])
    acc, tokens, path, slots, L = OT.tree_accept_commit(tok, parent, [5], target, [10], pt, 4)
    assert acc[0] == 2 and tokens[0].tolist() == [7, 2, 8, -1, -1]
    assert path[0].tolist() == [0, 2, 4, -1, -1] and L[0] == 13
    assert slots[0, :3].tolist() == [10, 11, 12]
    # two children of the root carry the same token: the lower index wins
    tok2 = np.array([[9, 7, 7, 2, 2]])
    acc, tokens, path, _, _ = OT.tree_accept_commit(tok2, parent, [5], target, [10], pt, 4)
    assert path[0, :acc[0] + 1].tolist() == [0, 1]       # node 1's child has tok 2 but target[1] = 0
    assert tokens[0, :2].tolist() == [7, 0]
    # nothing matches: only the bonus
    acc, tokens, path, _, L = OT.tree_accept_commit(tok, parent, [5], np.array([[1, 0, 0, 0, 0]]),
                                                    [10], pt, 4)
    assert acc[0] == 0 and tokens[0, 0] == 1 and L[0] == 11


def test_compact_path_by_hand():
    rows = np.arange(12.0)[:, None]
    out = OT.compact_path(rows, 5, [0, 2, 4], 2)
    assert out[5:8, 0].tolist() == [5.0, 7.0, 9.0]
    np.testing.assert_array_equal(out[:5], rows[:5])


# ---------------------------------------------------------------- end to end
N_NEW = 20
PROMPT = [3, 17, 8, 41, 5, 22, 9]


@pytest.fixture(scope="module")
def model_and_ref():
    for seed in range(20):
        m = ToyLM(seed)
        ref, gap = m.greedy_ar(PROMPT, N_NEW)
        if gap > 1e-9 and len(set(ref)) > 3:
            return m, ref
    raise AssertionError("no toy model with a clear argmax margin")


@pytest.mark.parametrize("depth,width", [(1, 1), (3, 2), (4, 3)])
@pytest.mark.parametrize("drafter", ["model", "perfect", "adversarial"])
def test_tree_seed_equals_greedy_ar(model_and_ref, depth, width, drafter):
    m, ref = model_and_ref
    out, rounds = seed_tree_greedy(m, PROMPT, N_NEW, depth, width, drafter=drafter,
                                   reference=ref, page_seed=depth * 10 + width)
    assert out == ref
    assert all(0 <= n <= depth for n in rounds)
    if drafter == "perfect":
        assert all(n == depth for n in rounds[:-1])


def test_siblings_rescue_a_wrong_main_branch(model_and_ref):
    """With the main child always wrong, width >= 2 still accepts tokens
    through the siblings in some rounds (width 1 never can)."""
    m, ref = model_and_ref
    _, r1 = seed_tree_greedy(m, PROMPT, N_NEW, 3, 1, drafter="adversarial", reference=ref)
    _, r3 = seed_tree_greedy(m, PROMPT, N_NEW, 3, 3, drafter="adversarial", reference=ref)
    assert all(n == 0 for n in r1)
    assert any(n > 0 for n in r3)


@pytest.mark.parametrize("mistake", ["causal", "nocompact"])
def test_planted_tree_mistakes_are_noticed(model_and_ref, mistake):
    m, ref = model_and_ref
    outs = [seed_tree_greedy(m, PROMPT, N_NEW, depth, 3, drafter=dr, reference=ref,
                             mistake=mistake)[0]
            for depth in (2, 4) for dr in ("model", "adversarial")]
    assert any(o != ref for o in outs)


@pytest.mark.parametrize("tau", [0.0, 0.5, 0.7, 1.01])
def test_dynamic_drafting_trees_keep_greedy_ar(model_and_ref, tau):
    """Trees built by the dynamic-drafting rule (k siblings from the drafter's
    p0, stop after a step with p0 <= tau) and checked by tree verification
    still emit exactly the greedy AR stream."""
    m, ref = model_and_ref
    out, rounds = seed_tree_greedy(m, PROMPT, N_NEW, 6, 1, tau=tau, max_nodes=24)
    assert out == ref
    assert all(0 <= n <= 6 for n in rounds)
    if tau > 1.0:
        assert all(n <= 1 for n in rounds)   # every step stops after its first level
