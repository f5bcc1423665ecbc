"""CPU oracle of the unified AI query: plain, slow, float64, obviously correct.

TEST INFRASTRUCTURE ONLY.  The tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The product path (the
CUDA library and its Python binding) never imports this package, and this
package never imports the product.  Inputs come from the ``synth`` generator.

Parity status per function:
  relational.*            pinned (brute force, invariants, hand-worked cases;
                          masked_sum: hand cases, exact integers, fsum vs sorted sums)
  transformer.rmsnorm     pinned (closed form on constant rows, torch rms_norm)
  transformer.rope        pinned (rotation closed form, relative invariance)
  transformer.causal_attention  pinned (torch SDPA, identical-key prefix mean)
  transformer.label_logits      pinned (zero-weight bias closed form,
                          identity-layer closed form, causality, GQA duplication)
  transformer.vocab_logits  pinned (label rows equal the pinned label head,
                          row t equals the logits of the first t+1 tokens)
  transformer.greedy_generate  pinned (zero-weight bias closed form, the
                          permutation-head closed form y_t = pi^(t+1)(x), eos/pad)
  relational.like_contains     pinned (delimited-string containment, edge cases)
  relational.self_join_pairs   pinned (hand-worked fixture, grouped 2-combinations,
                          sum of C(n_g, 2) closed form)
  query.run_pair_select   pinned (pair prompt layout, zero-weight bias closed form,
                          logits equal the concatenated prompt's label logits)
  whole-model numerics at random weights: parity unpinned beyond the
                          component pins (the paper prints no model outputs).
"""
