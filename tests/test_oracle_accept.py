"""Pins for oracle.accept: hand-worked cases of Alg. 2 (tests/golden), and an
exhaustive sweep of match patterns against the first-mismatch index computed
a second way."""

import os

import numpy as np
import pytest

from oracle.accept import accept_commit

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "accept_alg2.txt")


def _golden_cases():
    cases = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        f = [list(map(int, x.split())) for x in line.split(";")]
        cases.append(dict(k=f[0][0], draft=f[1], target=f[2], L=f[3][0], P=f[4][0], pt=f[5],
                          n=f[6][0], tokens=f[7], slots=f[8], new_L=f[9][0]))
    return cases


@pytest.mark.parametrize("case", _golden_cases(), ids=lambda c: f"k{c['k']}_L{c['L']}")
def test_golden_alg2_cases(case):
    width = len(case["target"])
    draft = np.zeros((1, max(width - 1, 1)), dtype=np.int32)
    draft[0, :len(case["draft"])] = case["draft"][:draft.shape[1]]
    acc, tok, slots, new_L = accept_commit(draft, np.array([case["target"]]), [case["k"]],
                                           [case["L"]], np.array([case["pt"]]), case["P"])
    n = case["n"]
    assert acc[0] == n
    assert tok[0, :n + 1].tolist() == case["tokens"]
    assert (tok[0, n + 1:] == -1).all()
    assert slots[0, :n + 1].tolist() == case["slots"]
    assert (slots[0, n + 1:] == -1).all()
    assert new_L[0] == case["new_L"]


@pytest.mark.parametrize("k", range(0, 9))
def test_exhaustive_match_patterns(k):
    """Every match/mismatch pattern over k_b in 0..k: n is the index of the
    first mismatch within the first k_b positions (else k_b); committed slots
    are the page-table images of L..L+n; L advances by n+1."""
    g = np.random.default_rng(k)
    P, n_pages = 4, 8
    pt = g.permutation(n_pages)[None, :].astype(np.int32)
    width = k + 1
    for k_b in range(0, k + 1):
        for bits in range(1 << k):
            match = [(bits >> i) & 1 == 1 for i in range(k)]
            target = g.integers(0, 100, size=width)
            draft = np.where(match, target[:k], (target[:k] + 1) % 100) if k else np.zeros(1, int)
            L = int(g.integers(0, n_pages * P - width))
            acc, tok, slots, new_L = accept_commit(draft[None], target[None], [k_b], [L], pt, P)
            mism = [i for i in range(k_b) if not match[i]]
            n = mism[0] if mism else k_b
            assert acc[0] == n
            assert tok[0, :n].tolist() == draft[:n].tolist()
            assert tok[0, n] == target[n]
            for i in range(n + 1):
                page, off = divmod(L + i, P)
                assert slots[0, i] == pt[0, page] * P + off
            assert new_L[0] == L + n + 1


def test_batch_rows_are_independent():
    g = np.random.default_rng(11)
    B, K, P = 5, 6, 16
    target = g.integers(0, 9, size=(B, K + 1))
    draft = g.integers(0, 9, size=(B, K))
    k_b = g.integers(0, K + 1, size=B)
    L = g.integers(0, 40, size=B)
    pt = np.stack([g.permutation(8) for _ in range(B)]).astype(np.int32)
    acc, tok, slots, new_L = accept_commit(draft, target, k_b, L, pt, P)
    for b in range(B):
        a1, t1, s1, n1 = accept_commit(draft[b:b + 1], target[b:b + 1], k_b[b:b + 1], L[b:b + 1],
                                       pt[b:b + 1], P)
        assert acc[b] == a1[0] and new_L[b] == n1[0]
        assert (tok[b] == t1[0]).all() and (slots[b] == s1[0]).all()
