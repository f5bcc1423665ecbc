"""The N>1 host path on CPU: gloo ranks each hold the same table (plus the
row-id column), cut it into contiguous ranges of equal candidate prompt
tokens from a relational pass over the whole table, compute their part of the
query restricted by the two row-id terms, and all-gather the results; the
merge equals the unsharded answer bit-exactly.  The per-rank query here is
the oracle's relational part plus a fixed decision rule (no GPU is involved)."""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import synth
from oracle import query as oq
from oracle import relational as rel
from paper_2608_10139_gb300 import shard


class _Res:
    def __init__(self, **kw):
        self.__dict__.update(kw)


def _query(table, lo, hi, build_keys):
    """Candidates of rows [lo, hi): rating >= 3; decision: token sum parity."""
    sub = {k: v[lo:hi] for k, v in table.cols.items()}
    cand = rel.compact(rel.predicate_mask(sub, [("rating", rel.GE, 3)], hi - lo))
    dec = np.array([int(table.text(lo + c).sum()) % 2 for c in cand], np.int32)
    gb = (lo + cand) % len(build_keys)
    agg = oq.aggregate(oq.AGG_GROUP_BUILD_KEY, dec, cand, 2, gb, build_keys)
    rows, keys, counts = agg["group_build_rows"], agg["group_keys"], agg["group_counts"]
    return _Res(count=agg["count"], n_candidates=len(cand), row_ids=rel.yes_row_ids(dec, cand),
                label_counts=rel.group_label_counts(dec, 2), group_build_rows=rows, group_keys=keys,
                group_counts=counts)


PREDS = [("rating", rel.GE, 3)]


def _ranged_query(table, cols, terms, build_keys):
    """The toy query on the rows the terms select (row ids are global)."""
    cand = rel.compact(rel.predicate_mask(cols, terms, table.n_rows))
    dec = np.array([int(table.text(c).sum()) % 2 for c in cand], np.int32)
    gb = cand % len(build_keys)
    agg = oq.aggregate(oq.AGG_GROUP_BUILD_KEY, dec, cand, 2, gb, build_keys)
    return _Res(count=agg["count"], n_candidates=len(cand), row_ids=rel.yes_row_ids(dec, cand),
                label_counts=rel.group_label_counts(dec, 2), group_build_rows=agg["group_build_rows"],
                group_keys=agg["group_keys"], group_counts=agg["group_counts"])


def _plan(q, world, prefix_len=16):
    cols = shard.with_row_ids(q.table.cols, q.table.n_rows)
    cand = rel.compact(rel.predicate_mask(cols, PREDS, q.table.n_rows))
    toks = prefix_len + np.diff(q.table.offsets)[cand]
    return cols, cand, toks, shard.token_balanced_ranges(q.table.n_rows, cand, toks, world)


def _worker(rank, world, port, n, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    q = synth.make_inputs(synth.scaled(synth.C1_TINY, n))
    keys = np.arange(37, dtype=np.int64) * 1000 - 5
    cols, _, _, ranges = _plan(q, world)       # every rank plans alike from the whole table
    lo, hi = ranges[rank]
    part = _ranged_query(q.table, cols, PREDS + shard.range_terms(lo, hi), keys)
    merged = shard.gather_merge(shard.local_result(part, 0))
    if rank == 0:
        out_q.put({k: np.asarray(v).tolist() for k, v in merged.items()})
    dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("n,world", [(1001, 2), (4096, 2), (3000, 3)])
def test_token_balanced_ranks_merge_equals_unsharded(n, world):
    ctx = mp.get_context("spawn")
    q_out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, n, q_out)) for r in range(world)]
    for p in procs:
        p.start()
    merged = q_out.get(timeout=120)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    q = synth.make_inputs(synth.scaled(synth.C1_TINY, n))
    keys = np.arange(37, dtype=np.int64) * 1000 - 5
    full = shard.local_result(_query(q.table, 0, n, keys), 0)
    for k in full:
        assert np.array_equal(np.asarray(merged[k]), np.asarray(full[k])), k


@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_token_balanced_ranges_partition_and_balance(world):
    """The ranges partition the rows in order, and each rank's candidate
    prompt tokens are within the largest single prompt of total / world."""
    q = synth.make_inputs(synth.scaled(synth.C2_SELECT, 20_000))
    preds = [(p.column, p.op, p.value) for p in synth.C2_SELECT.preds]
    cand = rel.compact(rel.predicate_mask(q.table.cols, preds, q.table.n_rows))
    toks = 64 + np.diff(q.table.offsets)[cand]
    rs = shard.token_balanced_ranges(q.table.n_rows, cand, toks, world)
    assert rs[0][0] == 0 and rs[-1][1] == q.table.n_rows and len(rs) == world
    assert all(a[1] == b[0] and a[0] <= a[1] for a, b in zip(rs, rs[1:]))
    share = [int(toks[(cand >= lo) & (cand < hi)].sum()) for lo, hi in rs]
    assert sum(share) == int(toks.sum())
    assert max(abs(x - toks.sum() / world) for x in share) <= toks.max()
    assert rs == shard.token_balanced_ranges(q.table.n_rows, cand, toks, world)   # every rank plans alike


def test_token_balanced_ranges_edge_cases():
    assert shard.token_balanced_ranges(10, [], [], 3) == [shard.shard_range(10, 3, r) for r in range(3)]
    assert shard.token_balanced_ranges(0, [], [], 2) == [(0, 0), (0, 0)]
    # one heavy candidate: everything lands on one rank, the others get empty or row-only ranges
    rs = shard.token_balanced_ranges(100, [50], [1000], 4)
    assert rs[0][0] == 0 and rs[-1][1] == 100 and sum(1 for lo, hi in rs if lo <= 50 < hi) == 1
    with pytest.raises(ValueError):
        shard.token_balanced_ranges(10, [1], [1], 0)


def test_range_terms_select_exactly_the_range():
    cols = shard.with_row_ids({"x": np.arange(50, dtype=np.int32)}, 50)
    ids = rel.compact(rel.predicate_mask(cols, shard.range_terms(7, 19), 50))
    assert ids.tolist() == list(range(7, 19))


def test_shard_ranges_partition():
    for n in (0, 1, 7, 100):
        for world in (1, 2, 3, 8):
            rs = [shard.shard_range(n, world, r) for r in range(world)]
            assert rs[0][0] == 0 and rs[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
            assert max(h - l for l, h in rs) - min(h - l for l, h in rs) <= 1


def test_merge_keeps_a_count_that_the_aggregate_does_not_define():
    """K > 2 labels report count -1 (undefined); the merge keeps -1 instead of
    summing it, and sums label counts element-wise."""
    e = np.zeros(0, np.int64)
    parts = [{"count": np.int64(-1), "n_candidates": np.int64(n), "row_ids": e,
              "label_counts": np.array(lc, np.int64), "group_build_rows": e, "group_keys": e, "group_counts": e}
             for n, lc in ((3, [1, 0, 2, 0, 0]), (4, [0, 1, 1, 1, 1]))]
    m = shard.merge(parts)
    assert int(m["count"]) == -1 and int(m["n_candidates"]) == 7
    assert m["label_counts"].tolist() == [1, 1, 3, 1, 1]
