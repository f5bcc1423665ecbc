"""Table 2 Q4 through the C-ABI: the key self-join's pairs formed on the device
(bit-exact against the oracle's nested loop, in ascending (a, b) order), the
AI_IF logits of every pair's prompt (prefix ++ text(a) ++ text(b)) within the
margin tolerance, and the aggregate equal to the oracle's aggregation of the
GPU's own decisions."""
import numpy as np
import pytest

import synth
from helpers import compare_logits, gpu_ctx, weights_list
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


def _table(n, n_keys, seed, empty_every=0, key_scale=1):
    rng = np.random.default_rng(seed)
    lens = rng.integers(1, 24, n)
    if empty_every:
        lens[::empty_every] = 0
    off = np.zeros(n + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    keys = (rng.integers(0, n_keys, n).astype(np.int64) - n_keys // 2) * key_scale
    cols = {"movie": keys, "score": rng.integers(0, 100, n).astype(np.int32)}
    return synth.Table(n, cols, off, rng.integers(0, synth.TINY.vocab, int(off[-1])).astype(np.int32))


@pytest.fixture(scope="module")
def model(ctx):
    W = synth.make_weights(synth.TINY, 4001)
    m = ctx.load_model(synth.TINY, weights_list(synth.TINY, W))
    yield W, m
    ctx.free_model(m)


@pytest.mark.parametrize("n,n_keys,key_scale,empty", [(300, 40, 1, 9), (700, 300, 2 ** 47 + 3, 0), (60, 1, 1, 5)])
def test_pair_select_matches_oracle(ctx, model, n, n_keys, key_scale, empty):
    W, m = model
    tab = _table(n, n_keys, n + n_keys, empty, key_scale)
    prefix = np.arange(5, 21, dtype=np.int32)
    preds = [("score", rel.LT, 60)]
    t = ctx.load_table(tab.cols, (tab.offsets, tab.tokens))
    r = ctx.run_pair_select(t, "movie", m, preds, prefix, [100, 101], agg=aiq.AGG_ROW_IDS, flags=aiq.FLAG_LOGITS)
    ctx.free_table(t)
    o = oq.run_pair_select(tab, "movie", preds, prefix, [100, 101], tf.Model(synth.TINY, W))
    assert r.n_candidates == len(o.pairs)
    assert np.array_equal(np.stack([r.cand_row_ids, r.cand_build_rows], 1), o.pairs.astype(np.int32))
    compare_logits(r.label_logits, o.logits, f"pairs n={n}")
    agg = oq.pair_aggregate(r.decisions, o.pairs)
    assert r.count == agg["count"]
    assert np.array_equal(np.stack([r.row_ids, r.row_ids_b], 1), agg["yes_pairs"].astype(np.int32))


def test_pair_select_self_join_at_scale_and_edges(ctx, model):
    W, m = model
    prefix = np.array([7, 8, 9], np.int32)
    # 6000 rows over 5000 keys (several radix-sort tiles), negative and > 2^32 keys: pairs exact
    tab = _table(6000, 5000, 11, 0, 2 ** 33 + 1)
    t = ctx.load_table(tab.cols, (tab.offsets, tab.tokens))
    r = ctx.run_pair_select(t, "movie", m, [], prefix, [100, 101], agg=aiq.AGG_COUNT, flags=aiq.FLAG_LOGITS)
    want = np.array(rel.self_join_pairs(tab.cols["movie"], np.arange(6000)), np.int32).reshape(-1, 2)
    assert np.array_equal(np.stack([r.cand_row_ids, r.cand_build_rows], 1), want)
    assert r.count == int(np.sum(r.decisions == 1))
    # nothing selected; every key distinct (no pair)
    e = ctx.run_pair_select(t, "movie", m, [("score", rel.GT, 1000)], prefix, [100, 101], agg=aiq.AGG_ROW_IDS)
    assert e.n_candidates == 0 and e.count == 0 and e.row_ids.size == 0
    ctx.free_table(t)
    u = _table(50, 10 ** 6, 3, 0, 1)
    u.cols["movie"] = np.arange(50, dtype=np.int64) * 7
    t = ctx.load_table(u.cols, (u.offsets, u.tokens))
    z = ctx.run_pair_select(t, "movie", m, [], prefix, [100, 101], agg=aiq.AGG_ROW_IDS)
    assert z.n_candidates == 0 and z.count == 0
    with pytest.raises(aiq.AiqError):
        ctx.run_pair_select(t, "score", m, [], prefix, [100, 101])   # the key must be INT64
    ctx.free_table(t)
