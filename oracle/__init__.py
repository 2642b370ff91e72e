"""Oracle for the SEED draft/verify attention path -- TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 CPU statement of what the path computes, written from
the paper (SEED: Self-Speculative Decoding via Implicit Encoder-Decoder):

* ``attention``  -- softmax attention over the KV cache (Sec. 4.1, "Cheap
  drafting between verifications": the drafter's cross-attention is ordinary
  self-attention over the cache), for the draft query and for the k+1 causal
  verify queries (Alg. 2, drafting and verification phases).
* ``cache``      -- the paged KV cache: slot of a logical position, gathering a
  sequence's rows, appending rows (Alg. 2; cache updates left implicit in
  Sec. 3).
* ``accept``     -- greedy longest-prefix acceptance, bonus token and the
  commit/rollback of cache rows (Alg. 2, acceptance and truncation steps).
* ``tree``       -- tree-based verification (Sec. D.1): the tree mask (each
  candidate sees the verified prefix and its own ancestral path), the greedy
  walk from the root with its bonus token, and the compaction of the accepted
  path's cache rows.
* ``drafting``   -- confidence-aware dynamic drafting (Sec. D.1): the
  drafter's distribution over the vocabulary, its top tokens, the
  sibling-count rule on the top-1 probability and the stop threshold.
* ``draft_step`` -- one whole draft step (Sec. 4.1 drafting; the work the
  computational-cost appendix counts): raw embedding, the decoder layers in
  the pre-norm form of the paper's Qwen3 models (RMS norms, q/k norms, RoPE,
  grouped attention over the deep cache plus the draft rows, SwiGLU MLP),
  final norm and the dynamic-drafting head.
* ``block_attn`` -- the decoder's block-causal training attention (Sec. 4.2,
  "Training with Block Attention"; Fig. 2): deep-cache rows of the preceding
  blocks plus causal self-attention within the query's own block.
* ``toy_model``  -- a tiny float64 transformer running Alg. 2 end to end (with
  a linear draft or a draft tree) and plain greedy decoding, for the
  exactness property of Sec. 4.1.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  It shares
no code with the CUDA path and never imports it.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(brute force, closed forms, library cross-checks, invariants, exactness of the
end-to-end loop).  Nothing is "parity unpinned".
"""
