"""Pins of the oracle's generation half (AI_TRANSFORM greedy decoding and the
LIKE '%pattern%' filter) against closed forms, the already pinned label head,
causality and an independent formulation of substring containment (CPU only)."""
from dataclasses import replace

import numpy as np
import pytest

import synth
from oracle import query as oq
from oracle import relational as rel
from oracle import transformer as tf

SMALL = synth.ModelShape(n_layers=2, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16,
                         d_ffn=96, vocab=300)


def _bf16(a):
    return synth.f32_to_bf16_bits(np.asarray(a, np.float32))


def test_vocab_logits_label_rows_equal_label_head():
    m = tf.Model(SMALL, synth.make_weights(SMALL, 21))
    seq = np.random.default_rng(1).integers(0, SMALL.vocab, 9)
    labels = [100, 101, 7, 299]
    z = tf.vocab_logits(m, [seq])
    assert z.shape == (9, SMALL.vocab)
    assert np.allclose(z[-1, labels], tf.label_logits(m, [seq], labels)[0], rtol=1e-12, atol=1e-12)


def test_vocab_logits_row_t_is_the_prefix_next_token_distribution():
    m = tf.Model(SMALL, synth.make_weights(SMALL, 22))
    seq = np.random.default_rng(2).integers(0, SMALL.vocab, 10)
    full = tf.vocab_logits(m, [seq])
    for t in (0, 4, 9):
        assert np.allclose(full[t], tf.vocab_logits(m, [seq[:t + 1]])[-1], rtol=1e-12, atol=1e-12)


def test_first_argmax_takes_lowest_index_on_ties():
    assert tf.first_argmax(np.array([1.0, 3.0, 3.0, 2.0])) == 1
    assert tf.first_argmax(np.array([-1.0])) == 0
    assert tf.first_argmax(np.array([0.0, 0.0])) == 0


def test_greedy_zero_weights_repeats_bias_argmax_and_eos_masks():
    s = SMALL
    w = synth.make_weights(s, 0, zero=True)
    b = np.random.default_rng(3).standard_normal(s.vocab)
    w["lm_bias"] = _bf16(b)
    m = tf.Model(s, w)
    top = int(np.argmax(tf.bf16_to_f64(w["lm_bias"])))
    toks, n = tf.greedy_generate(m, np.array([5, 6, 7]), 4)
    assert toks.tolist() == [top] * 4 and n == 4
    toks, n = tf.greedy_generate(m, np.array([5]), 4, eos=top, pad=9)
    assert toks.tolist() == [top, 9, 9, 9] and n == 0


def _permutation_model(perm):
    """Identity embedding, zero blocks, unit gains, LM head = permutation:
    the residual stays e_x, the final norm scales it by ~sqrt(d), and the
    logits are largest exactly at pi(x)."""
    v = len(perm)
    s = replace(SMALL, d_model=v, vocab=v, n_heads=2, n_kv_heads=1, head_dim=8, d_ffn=32)
    w = synth.make_weights(s, 0, zero=True)
    w["embed"] = _bf16(np.eye(v))
    head = np.zeros((v, v))
    head[perm, np.arange(v)] = 1.0       # row pi(i) reads input feature i
    w["lm_head"] = _bf16(head)
    for l in range(s.n_layers):
        w[f"l{l}.attn_norm"] = _bf16(np.ones(v))
        w[f"l{l}.mlp_norm"] = _bf16(np.ones(v))
    w["final_norm"] = _bf16(np.ones(v))
    return tf.Model(s, w)


def test_greedy_permutation_head_closed_form():
    rng = np.random.default_rng(4)
    perm = rng.permutation(16)
    while np.array_equal(perm[perm], np.arange(16)):   # not an involution: pi and pi^-1 differ
        perm = rng.permutation(16)
    m = _permutation_model(perm)
    prompt = np.array([3, 11, 2])
    toks, n = tf.greedy_generate(m, prompt, 6)
    want, x = [], 2
    for _ in range(6):
        x = int(perm[x])
        want.append(x)
    assert toks.tolist() == want and n == 6
    # eos at the second step: the first token, then the eos, then pad
    toks, n = tf.greedy_generate(m, prompt, 6, eos=want[1], pad=15)
    assert toks.tolist() == [want[0], want[1], 15, 15, 15, 15] and n == 1


def _delimited(seq):
    return "," + ",".join(str(int(x)) for x in seq) + ","


@pytest.mark.parametrize("seed", range(6))
def test_like_contains_matches_delimited_string_search(seed):
    rng = np.random.default_rng(seed)
    for _ in range(200):
        t = rng.integers(0, 4, rng.integers(0, 12))
        p = rng.integers(0, 4, rng.integers(1, 4))
        want = _delimited(p) in _delimited(t) if len(t) else False
        assert rel.like_contains(t, p) == want


def test_like_contains_edge_cases():
    assert rel.like_contains([], [])
    assert rel.like_contains([1, 2], [])
    assert not rel.like_contains([], [1])
    assert rel.like_contains([1, 2, 3], [1, 2, 3])
    assert not rel.like_contains([1, 2], [1, 2, 3])
    assert rel.like_contains([4, 1, 2], [1, 2])                  # at the end
    assert not rel.like_contains([12, 3], [2, 3])                # tokens, not digits
    assert rel.like_contains([7, 7, 8], [7, 8])                  # overlapping start


def test_like_aggregate_counts_and_ids():
    a = oq.like_aggregate(np.array([True, False, True]), np.array([4, 9, 12]))
    assert a["count"] == 2 and a["row_ids"].tolist() == [4, 12]


def test_run_transform_tiny_permutation_table():
    perm = np.roll(np.arange(16), -1)            # pi(x) = x + 1 mod 16
    m = _permutation_model(perm)
    tab = synth.Table(4, {"r": np.array([1, 5, 3, 4], np.int32)},
                      np.array([0, 2, 3, 3, 5], np.int64), np.array([9, 1, 6, 0, 14], np.int32))
    prefix = np.array([2], np.int32)
    res = oq.run_transform(tab, prefix, [("r", rel.GE, 3)], m, 3, like=[8, 9])
    assert res.cand_rows.tolist() == [1, 2, 3]
    # last prompt tokens: row 1 -> 6, row 2 (empty text) -> prefix 2, row 3 -> 14
    assert res.tokens.tolist() == [[7, 8, 9], [3, 4, 5], [15, 0, 1]]
    assert res.match.tolist() == [True, False, False]
    assert res.agg == {"count": 1, "row_ids": res.agg["row_ids"]} and res.agg["row_ids"].tolist() == [1]
