"""End-to-end pin of the oracle's attention, paged cache, acceptance and
rollback: greedy SEED (Alg. 2) on a tiny float64 transformer must emit exactly
the greedy autoregressive stream (Sec. 4.1: the encoder/decoder view is
exactly standard decoding; drafts are only accepted where they equal the
verifier's argmax).  The AR side recomputes every prefix with a dense causal
attention matrix and shares no attention code with the oracle."""

import numpy as np
import pytest

from oracle.toy_model import ToyLM, seed_greedy

N_NEW = 24
PROMPT = [3, 17, 8, 41, 5, 22, 9]


@pytest.fixture(scope="module")
def model_and_ref():
    for seed in range(20):
        m = ToyLM(seed)
        ref, gap = m.greedy_ar(PROMPT, N_NEW)
        if gap > 1e-9 and len(set(ref)) > 3:
            return m, ref
    raise AssertionError("no toy model with a clear argmax margin")


@pytest.mark.parametrize("d", [0, 1, 4, 8])
@pytest.mark.parametrize("drafter", ["model", "perfect", "adversarial"])
def test_seed_equals_greedy_ar(model_and_ref, d, drafter):
    m, ref = model_and_ref
    out, rounds = seed_greedy(m, PROMPT, N_NEW, d, drafter=drafter, reference=ref,
                              page_seed=d + 7)
    assert out == ref
    assert all(0 <= n <= d for n in rounds)
    if d == 0:
        assert all(n == 0 for n in rounds) and len(rounds) == N_NEW
    if drafter == "perfect" and d > 0:
        # every round but possibly the last one accepts all d drafts
        assert all(n == d for n in rounds[:-1])
    if drafter == "adversarial":
        assert all(n == 0 for n in rounds)


def test_planted_commit_mistake_is_noticed(model_and_ref):
    """Planted mistake in the oracle: a commit that keeps one row too few
    (forgets the row of X_draft[0]) must break the equality with greedy AR."""
    import oracle.accept as acc_mod

    m, ref = model_and_ref
    real = acc_mod.accept_commit

    def short(draft_ids, target_ids, k_b, ctx_lens, page_table, page_size):
        a, t, s, L = real(draft_ids, target_ids, k_b, ctx_lens, page_table, page_size)
        return a, t, s, L - 1

    acc_mod.accept_commit = short
    try:
        out, _ = seed_greedy(m, PROMPT, N_NEW, 4, drafter="model", reference=ref)
    finally:
        acc_mod.accept_commit = real
    assert out != ref


def test_planted_mask_mistake_is_noticed(model_and_ref):
    """Planted mistake: verify queries that also see the later new rows (no
    causal mask among the k+1 rows) must break the equality."""
    import oracle.attention as att_mod

    m, ref = model_and_ref
    real = att_mod.verify_attention_seq

    def no_mask(q, k_rows, v_rows, L, scale):
        n_q = q.shape[0]
        G = q.shape[1] // k_rows.shape[1]
        out = np.zeros_like(q)
        for j in range(n_q):
            for h in range(q.shape[1]):
                out[j, h] = att_mod.attend(q[j, h], k_rows[:L + n_q, h // G],
                                           v_rows[:L + n_q, h // G], scale)[0]
        return out, np.zeros(q.shape[:2])

    att_mod.verify_attention_seq = no_mask
    try:
        out, _ = seed_greedy(m, PROMPT, N_NEW, 4, drafter="perfect", reference=ref)
    finally:
        att_mod.verify_attention_seq = real
    assert out != ref
