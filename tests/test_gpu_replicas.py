"""Multi-GPU replicas, checked on one GPU: the path shards by rows (each
replica runs the whole query on a contiguous row range of the fact table,
with the model and any join build side replicated), and the only exchange is
the merge of the small results.  Running the shards one after another on one
GPU and merging them on the host must give the unsharded answer bit-exactly:
rows never interact inside the query."""
from dataclasses import replace

import numpy as np
import pytest

import synth
from helpers import gpu_ctx, oracle_preds, weights_list
from paper_2608_10139_gb300 import aiq, shard

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = gpu_ctx()
    yield c
    c.close()


def _rows(t: synth.Table, lo: int, hi: int) -> synth.Table:
    """Rows [lo, hi) of a table, text offsets rebased to the slice."""
    off = t.offsets[lo:hi + 1] - t.offsets[lo]
    return synth.Table(hi - lo, {k: v[lo:hi].copy() for k, v in t.cols.items()}, off.astype(np.int64),
                       t.tokens[t.offsets[lo]:t.offsets[hi]].copy())


def _load(ctx, t: synth.Table):
    return ctx.load_table(t.cols, (t.offsets, t.tokens), n_rows=t.n_rows)


def _check_merge(full, parts):
    merged = shard.merge(parts)
    for k, v in full.items():
        assert np.array_equal(np.asarray(merged[k]), np.asarray(v)), k


SELECT_CASES = {
    "row_ids": replace(synth.C2_SELECT, name="c2_tiny_replicas", n_rows=3000, model=synth.TINY,
                       text=synth.TextRecipe("lognormal", 16, 200, median=60.0), prefix_len=32),
    "group_by_label": replace(synth.C4_MULTILABEL, name="c4_tiny_replicas", n_rows=2000, model=synth.TINY,
                              text=synth.TextRecipe("lognormal", 32, 300, median=80.0), prefix_len=24),
}


@pytest.mark.parametrize("name", list(SELECT_CASES))
@pytest.mark.parametrize("world", [2, 3])
def test_select_shards_merge_to_the_unsharded_result(ctx, name, world):
    w = SELECT_CASES[name]
    q = synth.make_inputs(w)
    m = ctx.load_model(w.model, weights_list(w.model, synth.make_weights(w.model, w.weight_seed)))
    preds = oracle_preds(w.preds)

    def run(tab):
        t = _load(ctx, tab)
        r = ctx.run_select(t, m, preds, q.prefix, w.label_ids, agg=w.agg)
        ctx.free_table(t)
        return r

    full = shard.local_result(run(q.table), 0)
    parts = []
    for rank in range(world):
        lo, hi = shard.shard_range(q.table.n_rows, world, rank)
        parts.append(shard.local_result(run(_rows(q.table, lo, hi)), lo))
    ctx.free_model(m)
    assert sum(int(p["n_candidates"]) for p in parts) == int(full["n_candidates"]) > 0
    _check_merge(full, parts)


def test_join_shards_merge_to_the_unsharded_result(ctx):
    """The reviews (probe side) are sharded; the filtered movies (build side)
    are replicated on every replica, so group rows are global build rows."""
    w = replace(synth.C3_JOIN, name="c3_tiny_replicas", n_rows=4000, join_build_rows=500, model=synth.TINY,
                text=synth.TextRecipe("lognormal", 16, 120, median=40.0), prefix_len=16)
    q = synth.make_inputs(w)
    m = ctx.load_model(w.model, weights_list(w.model, synth.make_weights(w.model, w.weight_seed)))
    tb = ctx.load_table(q.build.cols, n_rows=q.build.n_rows)
    bp = oracle_preds(w.join_build_preds)

    def run(tab):
        tp = _load(ctx, tab)
        r = ctx.run_join_select(tb, "movie_id", bp, tp, "movie_id", m, [], q.prefix, w.label_ids,
                                agg=synth.AGG_GROUP_BUILD_KEY)
        ctx.free_table(tp)
        return r

    full = shard.local_result(run(q.table), 0)
    parts = []
    for rank in range(3):
        lo, hi = shard.shard_range(q.table.n_rows, 3, rank)
        parts.append(shard.local_result(run(_rows(q.table, lo, hi)), lo))
    ctx.free_table(tb)
    ctx.free_model(m)
    assert len(full["group_build_rows"]) > 0
    _check_merge(full, parts)


def _plan(ctx, run, q, world):
    """The ranks' row ranges, from the library's relational-only pass over the
    whole table (the first thing every rank does in the multi-GPU benchmark)."""
    cand = run([], aiq.FLAG_RELATIONAL_ONLY).cand_row_ids
    toks = len(q.prefix) + np.diff(q.table.offsets)[cand]
    return shard.token_balanced_ranges(q.table.n_rows, cand, toks, world)


@pytest.mark.parametrize("name", list(SELECT_CASES))
@pytest.mark.parametrize("world", [2, 4])
def test_row_range_terms_on_one_table_merge_to_the_unsharded_result(ctx, name, world):
    """The benchmark's multi-GPU step, one rank after another: every rank holds
    the whole table plus its row-id column, plans token-balanced ranges from a
    relational-only pass, runs the query restricted by the two row-id terms,
    and the merged results equal the unsharded query's."""
    w = SELECT_CASES[name]
    q = synth.make_inputs(w)
    m = ctx.load_model(w.model, weights_list(w.model, synth.make_weights(w.model, w.weight_seed)))
    t = ctx.load_table(shard.with_row_ids(q.table.cols, q.table.n_rows), (q.table.offsets, q.table.tokens))
    preds = oracle_preds(w.preds)

    def run(extra, flags=0):
        return ctx.run_select(t, m, preds + extra, q.prefix, w.label_ids, agg=w.agg, flags=flags)

    full = shard.local_result(run([]), 0)
    ranges = _plan(ctx, run, q, world)
    parts = [shard.local_result(run(shard.range_terms(lo, hi)), 0) for lo, hi in ranges]
    ctx.free_table(t)
    ctx.free_model(m)
    assert sum(int(p["n_candidates"]) for p in parts) == int(full["n_candidates"]) > 0
    _check_merge(full, parts)


def test_row_range_terms_on_the_join_probe_side(ctx):
    w = replace(synth.C3_JOIN, name="c3_tiny_ranges", n_rows=4000, join_build_rows=500, model=synth.TINY,
                text=synth.TextRecipe("lognormal", 16, 120, median=40.0), prefix_len=16)
    q = synth.make_inputs(w)
    m = ctx.load_model(w.model, weights_list(w.model, synth.make_weights(w.model, w.weight_seed)))
    tb = ctx.load_table(q.build.cols, n_rows=q.build.n_rows)
    tp = ctx.load_table(shard.with_row_ids(q.table.cols, q.table.n_rows), (q.table.offsets, q.table.tokens))
    bp = oracle_preds(w.join_build_preds)

    def run(extra, flags=0):
        return ctx.run_join_select(tb, "movie_id", bp, tp, "movie_id", 0 if flags else m, extra, q.prefix,
                                   w.label_ids, agg=synth.AGG_GROUP_BUILD_KEY, flags=flags)

    full = shard.local_result(run([]), 0)
    parts = [shard.local_result(run(shard.range_terms(lo, hi)), 0) for lo, hi in _plan(ctx, run, q, 3)]
    for h in (tb, tp):
        ctx.free_table(h)
    ctx.free_model(m)
    assert len(full["group_build_rows"]) > 0
    _check_merge(full, parts)
