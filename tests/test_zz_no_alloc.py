"""The allocation-free filter entry point (aiq_filter_compact_static) against
the query path's own filter and compaction (aiq_run_select with
AIQ_FLAG_RELATIONAL_ONLY).

The allocation-free variant exists for callers that may not allocate device
memory while they run: a worker limited to a fixed device arena, or an
operator inside another engine's allocation-free loop.  It keeps its scratch
in a static device array, so the checks here are that two calls in a row (the
second reusing the scratch the first left behind) both return exactly the ids
the allocating path returns, that the array's full capacity works, that an
empty input gives a count of zero, and that sizes above the capacity are
refused.  This file sorts last so that a failure here never hides another
test's result."""
import numpy as np
import pytest

from helpers import gpu_ctx
from paper_2608_10139_gb300 import aiq

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ROWS = 1 << 24


def _static(terms, n, ids, count):
    torch.cuda.synchronize()
    aiq.filter_compact_static(terms, n, ids.data_ptr(), count.data_ptr(), 0)
    torch.cuda.synchronize()
    return int(count.item())


def test_static_filter_matches_query_path_on_two_calls():
    ctx = gpu_ctx()
    try:
        n = 300_001
        rng = np.random.default_rng(11)
        cols = {"a": rng.integers(0, 10, n).astype(np.int32),
                "b": rng.integers(-2**40, 2**40, n).astype(np.int64),
                "c": rng.standard_normal(n).astype(np.float32)}
        table = ctx.load_table(cols, n_rows=n)
        dev = {k: torch.from_numpy(v).cuda() for k, v in cols.items()}
        codes = {"a": aiq.INT32, "b": aiq.INT64, "c": aiq.FLOAT32}
        ids = torch.full((n,), -1, dtype=torch.int32, device="cuda")
        count = torch.full((1,), -1, dtype=torch.int64, device="cuda")
        queries = [
            [("a", aiq.GE, 5), ("b", aiq.GT, 0)],                 # about a quarter of the rows
            [("c", aiq.LE, -0.5), ("a", aiq.NE, 3)],              # a different, smaller set
        ]
        for preds in queries:
            want = ctx.run_select(table, 0, preds, [], [0, 1], flags=aiq.FLAG_RELATIONAL_ONLY).cand_row_ids
            terms = [(dev[c].data_ptr(), codes[c], op, v) for c, op, v in preds]
            k = _static(terms, n, ids, count)
            assert k == len(want)
            assert np.array_equal(ids[:k].cpu().numpy(), want)
        # no rows: the count is zero (written, not left at the previous call's value)
        count.fill_(-1)
        assert _static([(dev["a"].data_ptr(), aiq.INT32, aiq.GE, 5)], 0, ids, count) == 0
        with pytest.raises(aiq.AiqError) as e:
            aiq.filter_compact_static([], MAX_ROWS + 1, ids.data_ptr(), count.data_ptr(), 0)
        assert e.value.status == aiq.ERR_CAPACITY
        ctx.free_table(table)
    finally:
        ctx.close()


def test_static_filter_at_its_row_limit():
    """Exactly 2^24 rows, the array's capacity, twice in a row."""
    ctx = gpu_ctx()
    try:
        rng = np.random.default_rng(12)
        a = rng.integers(0, 1000, MAX_ROWS).astype(np.int32)
        table = ctx.load_table({"a": a}, n_rows=MAX_ROWS)
        dev = torch.from_numpy(a).cuda()
        ids = torch.full((MAX_ROWS,), -1, dtype=torch.int32, device="cuda")
        count = torch.full((1,), -1, dtype=torch.int64, device="cuda")
        for op, v in ((aiq.LT, 137), (aiq.GE, 500)):
            want = ctx.run_select(table, 0, [("a", op, v)], [], [0, 1],
                                  flags=aiq.FLAG_RELATIONAL_ONLY).cand_row_ids
            k = _static([(dev.data_ptr(), aiq.INT32, op, v)], MAX_ROWS, ids, count)
            assert k == len(want)
            assert np.array_equal(ids[:k].cpu().numpy(), want)
        ctx.free_table(table)
    finally:
        ctx.close()
