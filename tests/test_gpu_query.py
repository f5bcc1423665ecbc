"""Query-level parity through the C-ABI: relational results bit-exact against
the oracle, label logits within the margin tolerance, decisions on every
clear row, and aggregates equal to the oracle's aggregation of the GPU's own
decision vector (Table 2 Q1/Q2 shapes, the reviews-movies join of Section 4,
the multi-label GROUP BY)."""
from dataclasses import replace

import numpy as np
import pytest

import synth
from helpers import compare_logits, gpu_ctx, oracle_preds, weights_list
from oracle import query as oq
from oracle import relational as rel
from oracle import transformer as tf
from paper_2608_10139_gb300 import aiq

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = gpu_ctx()
    yield c
    c.close()


def _load(ctx, t: synth.Table):
    text = (t.offsets, t.tokens) if t.offsets is not None else None
    return ctx.load_table(t.cols, text, n_rows=t.n_rows)


# ------------------------------------------------------------ relational ---

def _random_table(n, seed):
    rng = np.random.default_rng(seed)
    return synth.Table(n, {"a": rng.integers(0, 10, n).astype(np.int32),
                           "b": rng.integers(-2**40, 2**40, n).astype(np.int64),
                           "c": rng.standard_normal(n).astype(np.float32)})


PRED_SETS = [
    [],
    [("a", rel.GE, 5)],
    [("a", rel.LT, 3), ("b", rel.GT, 0)],
    [("a", rel.NE, 4), ("c", rel.LE, 0.25), ("b", rel.LE, 2**39)],
    [("a", rel.EQ, 7)],
    [("a", rel.GT, 100)],          # nothing survives
    [("a", rel.GE, -2**40)],       # constant outside the int32 range: everything survives
]


@pytest.mark.parametrize("n", [0, 1, 31, 2047, 2048, 2049, 100_003, (1 << 22) + 777, 1 << 24])
def test_filter_compaction_bit_exact(ctx, n):
    t = _random_table(n, n)
    ref_t = ctx.load_table(t.cols, n_rows=n)
    try:
        for preds in PRED_SETS:
            r = ctx.run_select(ref_t, 0, preds, [], [0, 1], flags=aiq.FLAG_RELATIONAL_ONLY)
            want = rel.compact(rel.predicate_mask(t.cols, preds, n))
            assert r.n_candidates == len(want)
            assert np.array_equal(r.cand_row_ids, want), preds
    finally:
        ctx.free_table(ref_t)


def test_join_small_with_orphans_and_repeats(ctx):
    rng = np.random.default_rng(3)
    m, n = 300, 5000
    keys = synth.distinct_int63(rng, m)
    keys[:3] = [-7, 0, 2**62]                      # negative / zero keys hash too
    build = synth.Table(m, {"k": keys, "year": rng.integers(1950, 2025, m).astype(np.int32)})
    fk = np.where(rng.random(n) < 0.8, keys[rng.integers(0, m, n)], rng.integers(0, 2**62, n))
    probe = synth.Table(n, {"k": fk.astype(np.int64), "a": rng.integers(0, 10, n).astype(np.int32)})
    tb, tp = ctx.load_table(build.cols, n_rows=m), ctx.load_table(probe.cols, n_rows=n)
    for bpreds, ppreds in [([], []), ([("year", rel.GE, 2010)], []), ([("year", rel.LT, 1990)], [("a", rel.GE, 5)])]:
        r = ctx.run_join_select(tb, "k", bpreds, tp, "k", 0, ppreds, [], [0, 1], agg=aiq.AGG_COUNT,
                                flags=aiq.FLAG_RELATIONAL_ONLY)
        cand, cand_b = oq.join_candidates(probe, build, "k", "k", ppreds, bpreds,
                                          brute_force=(bpreds == [] and ppreds == []))
        assert np.array_equal(r.cand_row_ids, cand)
        assert np.array_equal(r.cand_build_rows, cand_b)
    ctx.free_table(tb)
    ctx.free_table(tp)


def test_join_rejects_duplicate_and_sentinel_build_keys(ctx):
    for keys in ([5, 9, 5], [1, -2**63, 3]):
        build = ctx.load_table({"k": np.array(keys, np.int64)})
        probe = ctx.load_table({"k": np.array([5, 1], np.int64)})
        with pytest.raises(aiq.AiqError) as e:
            ctx.run_join_select(build, "k", [], probe, "k", 0, [], [], [0, 1], agg=aiq.AGG_COUNT,
                                flags=aiq.FLAG_RELATIONAL_ONLY)
        assert e.value.status == aiq.ERR_INVALID_ARG
        ctx.free_table(build)
        ctx.free_table(probe)
    # the context stays usable afterwards
    t = ctx.load_table({"a": np.arange(10, dtype=np.int32)})
    r = ctx.run_select(t, 0, [("a", rel.GE, 5)], [], [0, 1], flags=aiq.FLAG_RELATIONAL_ONLY)
    assert r.cand_row_ids.tolist() == [5, 6, 7, 8, 9]


# ------------------------------------------------------------ full query ---

def _model(ctx, shape, seed):
    W = synth.make_weights(shape, seed)
    return ctx.load_model(shape, weights_list(shape, W)), W


def _select_parity(ctx, w, budget=None):
    q = synth.make_inputs(w)
    mh, W = _model(ctx, w.model, w.weight_seed)
    t = _load(ctx, q.table)
    if budget:
        ctx.set_option("token_budget", budget)
    try:
        r = ctx.run_select(t, mh, oracle_preds(w.preds), q.prefix, w.label_ids, agg=w.agg, flags=aiq.FLAG_LOGITS)
    finally:
        ctx.set_option("token_budget", 131072)
    o = oq.run_select(q.table, q.prefix, oracle_preds(w.preds), w.label_ids, w.agg, tf.Model(w.model, W, True))
    assert np.array_equal(r.cand_row_ids, o.cand_rows)
    compare_logits(r.label_logits, o.logits, w.name)
    agg = oq.aggregate(w.agg, r.decisions, o.cand_rows, len(w.label_ids))
    if len(w.label_ids) == 2:
        assert r.count == agg["count"]
        assert np.array_equal(r.decisions, rel.decide(r.label_logits.astype(np.float64)))
    if w.agg == synth.AGG_ROW_IDS:
        assert np.array_equal(r.row_ids, agg["row_ids"])
    if w.agg == synth.AGG_GROUP_LABEL:
        assert np.array_equal(r.label_counts, agg["label_counts"])
    n_tok = sum(len(q.prefix) + len(q.table.text(i)) for i in o.cand_rows)
    assert r.n_tokens == n_tok
    if len(o.cand_rows):   # the shared prefix runs once; each row runs only its own tokens
        assert r.n_prefill_tokens == n_tok - len(q.prefix) * (len(o.cand_rows) - 1)
    ctx.free_table(t)
    ctx.free_model(mh)
    return r


def test_c1_tiny_select_full_parity(ctx):
    _select_parity(ctx, synth.C1_TINY)


def test_c1_chunking_is_invisible(ctx):
    w = synth.C1_TINY
    a = _select_parity(ctx, w)
    b = _select_parity(ctx, w, budget=130)   # every chunk holds a couple of rows
    assert b.n_chunks > 10
    assert np.array_equal(a.label_logits, b.label_logits)   # rows never interact: bit-identical


def test_two_term_mlp_activations(ctx):
    """mlp_split forced on for a small model (by default only models of 32
    layers and d 4096 load with it): the query still matches the oracle, on a
    tighter bound than the one-term path reaches, and its AI_TRANSFORM path
    (the decode loop's MLP GEMMs) runs too."""
    w = synth.C1_TINY
    gqa = replace(w.model, d_model=256, n_heads=8, n_kv_heads=2, head_dim=64, d_ffn=512)
    ctx.set_option("mlp_split", 1)
    try:
        for shape in (w.model, gqa):
            r = _select_parity(ctx, replace(w, model=shape))
            assert r.n_candidates > 0
        q = synth.make_inputs(w)
        mh, W = _model(ctx, gqa, w.weight_seed)
        t = _load(ctx, q.table)
        g = ctx.run_transform(t, mh, oracle_preds(w.preds), q.prefix, 3)
        assert g.n_candidates > 0 and g.gen_tokens.shape[1] == 3
        ctx.free_table(t)
        ctx.free_model(mh)
    finally:
        ctx.set_option("mlp_split", -1)


def test_tiny_row_ids_query(ctx):
    w = replace(synth.C2_SELECT, name="c2_tiny", n_rows=3000, model=synth.TINY,
                text=synth.TextRecipe("lognormal", 16, 200, median=60.0), prefix_len=32)
    _select_parity(ctx, w)


def test_tiny_multilabel_group_by(ctx):
    w = replace(synth.C4_MULTILABEL, name="c4_tiny", n_rows=2000, model=synth.TINY,
                text=synth.TextRecipe("lognormal", 32, 300, median=80.0), prefix_len=24)
    _select_parity(ctx, w)


def test_tiny_join_group_by_build_key(ctx):
    w = replace(synth.C3_JOIN, name="c3_tiny", n_rows=4000, join_build_rows=500, model=synth.TINY,
                text=synth.TextRecipe("lognormal", 16, 120, median=40.0), prefix_len=16)
    q = synth.make_inputs(w)
    mh, W = _model(ctx, w.model, w.weight_seed)
    tb, tp = _load(ctx, q.build), _load(ctx, q.table)
    bp = oracle_preds(w.join_build_preds)
    r = ctx.run_join_select(tb, "movie_id", bp, tp, "movie_id", mh, [], q.prefix, w.label_ids,
                            agg=synth.AGG_GROUP_BUILD_KEY, flags=aiq.FLAG_LOGITS)
    o = oq.run_join_select(q.table, q.build, "movie_id", "movie_id", [], bp, q.prefix, w.label_ids,
                           w.agg, tf.Model(w.model, W, True))
    assert np.array_equal(r.cand_row_ids, o.cand_rows)
    assert np.array_equal(r.cand_build_rows, o.cand_build_rows)
    compare_logits(r.label_logits, o.logits, w.name)
    agg = oq.aggregate(w.agg, r.decisions, o.cand_rows, 2, o.cand_build_rows, q.build.cols["movie_id"])
    assert np.array_equal(r.group_build_rows, agg["group_build_rows"])
    assert np.array_equal(r.group_keys, agg["group_keys"])
    assert np.array_equal(r.group_counts, agg["group_counts"])
    assert int(r.group_counts.sum()) == r.count


def test_rows_with_empty_text(ctx):
    """A row whose text is empty is decided on the prefix alone; with no prefix
    such a row's prompt would be empty, which is refused."""
    w = synth.C1_TINY
    q = synth.make_inputs(w)
    lens = np.diff(q.table.offsets)
    lens[::7] = 0                                   # every 7th row loses its text
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tokens = np.concatenate([q.table.text(i)[:lens[i]] for i in range(q.table.n_rows)]).astype(np.int32)
    table = synth.Table(q.table.n_rows, q.table.cols, offsets, tokens)
    mh, W = _model(ctx, w.model, w.weight_seed)
    t = _load(ctx, table)
    preds = oracle_preds(w.preds)
    r = ctx.run_select(t, mh, preds, q.prefix, w.label_ids, agg=w.agg, flags=aiq.FLAG_LOGITS)
    o = oq.run_select(table, q.prefix, preds, w.label_ids, w.agg, tf.Model(w.model, W, True))
    assert np.array_equal(r.cand_row_ids, o.cand_rows)
    compare_logits(r.label_logits, o.logits, "empty-text rows")
    empty = np.diff(offsets)[o.cand_rows] == 0
    assert empty.sum() > 5 and np.all(r.label_logits[empty] == r.label_logits[empty][0])
    with pytest.raises(aiq.AiqError) as e:
        ctx.run_select(t, mh, preds, np.zeros(0, np.int32), w.label_ids)
    assert e.value.status == aiq.ERR_INVALID_ARG
    ctx.free_table(t)
    ctx.free_model(mh)


def test_degenerate_queries(ctx):
    w = synth.C1_TINY
    q = synth.make_inputs(w)
    mh, W = _model(ctx, w.model, w.weight_seed)
    t = _load(ctx, q.table)
    # no row survives: empty results, count 0
    r = ctx.run_select(t, mh, [("rating", rel.GT, 5)], q.prefix, w.label_ids, agg=synth.AGG_ROW_IDS)
    assert r.n_candidates == 0 and r.count == 0 and r.row_ids.size == 0
    # empty prefix and a single row
    r = ctx.run_select(t, mh, [("rating", rel.EQ, 3)], np.zeros(0, np.int32), w.label_ids,
                       agg=synth.AGG_COUNT, flags=aiq.FLAG_LOGITS)
    o = oq.run_select(q.table, np.zeros(0, np.int32), [("rating", rel.EQ, 3)], w.label_ids, w.agg,
                      tf.Model(w.model, W, True))
    compare_logits(r.label_logits, o.logits, "no prefix")
    # invalid inputs are rejected with a status, not a fault
    for kw in [dict(labels=[100, 5000]), dict(prefix=[4096])]:
        with pytest.raises(aiq.AiqError) as e:
            ctx.run_select(t, mh, [], kw.get("prefix", q.prefix), kw.get("labels", w.label_ids))
        assert e.value.status == aiq.ERR_INVALID_ARG
    with pytest.raises(aiq.AiqError) as e:
        ctx.run_select(t, 12345, [], q.prefix, w.label_ids)
    assert e.value.status == aiq.ERR_NOT_FOUND
    ctx.free_table(t)
    ctx.free_model(mh)


def test_sum_aggregate_matches_oracle_on_gpu_decisions(ctx):
    """Fig. 2's SELECT SUM(values) ... WHERE AI_IF(...) = 1: integer sums exact,
    the float sum within fp64 rounding of the correctly rounded sum."""
    w = synth.C1_TINY
    q = synth.make_inputs(w)
    W = synth.make_weights(w.model, w.weight_seed)
    rng = np.random.default_rng(17)
    n = q.table.n_rows
    cols = dict(q.table.cols)
    cols["v32"] = rng.integers(-2 ** 31, 2 ** 31 - 1, n).astype(np.int32)
    cols["v64"] = rng.integers(-2 ** 50, 2 ** 50, n).astype(np.int64)
    cols["vf"] = (rng.standard_normal(n) * 1e3).astype(np.float32)
    m = ctx.load_model(w.model, weights_list(w.model, W))
    t = ctx.load_table(cols, (q.table.offsets, q.table.tokens))
    preds = oracle_preds(w.preds)
    for name in ("v32", "v64", "vf"):
        r = ctx.run_select(t, m, preds, q.prefix, w.label_ids, agg=aiq.AGG_SUM, flags=aiq.FLAG_LOGITS,
                           sum_column=name)
        want = rel.masked_sum(r.decisions, r.cand_row_ids, cols[name])
        assert r.count == rel.count_yes(r.decisions)
        if name == "vf":
            bound = 1e-12 * float(np.abs(cols[name]).astype(np.float64).sum())
            assert abs(r.sum - want) <= bound, (r.sum, want)
        else:
            assert r.sum == want
    e = ctx.run_select(t, m, [("rating", rel.GT, 100)], q.prefix, w.label_ids, agg=aiq.AGG_SUM, sum_column="v64")
    assert e.count == 0 and e.sum == 0
    with pytest.raises(aiq.AiqError):
        ctx.run_select(t, m, preds, q.prefix, w.label_ids, agg=aiq.AGG_SUM, sum_column="text")
    ctx.free_table(t)
    ctx.free_model(m)
