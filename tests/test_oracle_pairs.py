"""Pins of the oracle's Table 2 Q4 half: the key self-join over the selected
rows, the pair prompt and the per-pair aggregate (CPU only)."""
import itertools
import os

import numpy as np
import pytest

import synth
from oracle import query as oq
from oracle import relational as rel
from oracle import transformer as tf

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read(name):
    rows = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            k, *v = line.split()
            rows.setdefault(k, []).append([int(x) for x in v])
    return rows


def test_self_join_hand_worked():
    g = _read("self_join_small.txt")
    movie = np.array(g["movie"][0], np.int64)
    score = np.array(g["score"][0], np.int32)
    rows = rel.compact(rel.predicate_mask({"score": score}, [("score", rel.LT, 40)], len(movie)))
    assert rel.self_join_pairs(movie, rows) == [tuple(p) for p in g["pair"]]


def _grouped_pairs(keys, rows):
    """Independent formulation: group the rows by key, all 2-combinations of
    each group, sorted."""
    groups = {}
    for r in sorted(rows):
        groups.setdefault(int(keys[r]), []).append(int(r))
    return sorted(p for g in groups.values() for p in itertools.combinations(g, 2))


@pytest.mark.parametrize("seed", range(6))
def test_self_join_equals_grouped_combinations_and_closed_form(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(0, 60))
    keys = rng.integers(-3, 5, n).astype(np.int64) * (2 ** 40)   # wide keys, few distinct
    rows = np.flatnonzero(rng.random(n) < 0.7)
    pairs = rel.self_join_pairs(keys, rows)
    assert pairs == _grouped_pairs(keys, rows)
    _, counts = np.unique(keys[rows], return_counts=True)
    assert len(pairs) == int(sum(c * (c - 1) // 2 for c in counts))       # sum of C(n_g, 2)
    assert all(a < b and keys[a] == keys[b] for a, b in pairs)


def test_pair_prompt_layout():
    off = np.array([0, 2, 2, 5], np.int64)
    tok = np.array([1, 2, 3, 4, 5], np.int32)
    p = oq.pair_prompts(np.array([9], np.int32), off, tok, [(0, 2), (1, 2)])
    assert [x.tolist() for x in p] == [[9, 1, 2, 3, 4, 5], [9, 3, 4, 5]]


def test_pair_select_zero_weights_bias_decides_every_pair():
    s = synth.TINY
    w = synth.make_weights(s, 0, zero=True)
    b = np.zeros(s.vocab, np.float32)
    b[100], b[101] = 0.5, -0.25
    w["lm_bias"] = synth.f32_to_bf16_bits(b)
    m = tf.Model(s, w)
    tab = synth.Table(6, {"k": np.array([1, 2, 1, 1, 2, 3], np.int64), "v": np.array([0, 1, 2, 3, 4, 5], np.int32)},
                      np.arange(7, dtype=np.int64) * 2, np.arange(12, dtype=np.int32))
    r = oq.run_pair_select(tab, "k", [("v", rel.LE, 4)], np.array([7, 8], np.int32), [100, 101], m)
    assert r.pairs.tolist() == [[0, 2], [0, 3], [1, 4], [2, 3]]
    assert np.allclose(r.logits, [[0.5, -0.25]] * 4)
    assert r.agg["count"] == 4 and r.agg["yes_pairs"].tolist() == r.pairs.tolist()


def test_pair_logits_are_the_concatenated_prompt_label_logits():
    s = synth.TINY
    W = synth.make_weights(s, 31)
    m = tf.Model(s, W)
    rng = np.random.default_rng(4)
    lens = rng.integers(0, 6, 5)
    off = np.zeros(6, np.int64)
    np.cumsum(lens, out=off[1:])
    tab = synth.Table(5, {"k": np.array([4, 4, 4, 2, 2], np.int64)}, off,
                      rng.integers(0, s.vocab, int(off[-1])).astype(np.int32))
    prefix = np.array([3, 1], np.int32)
    r = oq.run_pair_select(tab, "k", [], prefix, [100, 101], m, sample=np.array([1, 3]))
    want = [r.pairs[1], r.pairs[3]]
    seqs = [np.concatenate([prefix, tab.tokens[off[a]:off[a + 1]], tab.tokens[off[b]:off[b + 1]]]) for a, b in want]
    assert np.allclose(r.logits, tf.label_logits(m, seqs, [100, 101]), rtol=1e-12, atol=1e-12)
    assert r.agg is None
