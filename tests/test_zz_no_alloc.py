"""The allocation-free filter entry point (aiq_filter_compact_static) against
the query path's own filter and compaction (aiq_run_select with
AIQ_FLAG_RELATIONAL_ONLY).

The allocation-free variant exists for callers that may not allocate device
memory while they run: work recorded into a CUDA graph, or a worker limited
to a fixed device arena.  It keeps its scratch in a static device array, so
the checks here are that two calls in a row (the second reusing the scratch
the first left behind) both return exactly the ids the allocating path
returns, and that sizes above the array's capacity are refused.  This file
sorts last so that a failure here never hides another test's result."""
import numpy as np
import pytest

from helpers import gpu_ctx
from paper_2608_10139_gb300 import aiq

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


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
            torch.cuda.synchronize()
            aiq.filter_compact_static(terms, n, ids.data_ptr(), count.data_ptr(), 0)
            torch.cuda.synchronize()
            k = int(count.item())
            assert k == len(want)
            assert np.array_equal(ids[:k].cpu().numpy(), want)
        with pytest.raises(aiq.AiqError) as e:
            aiq.filter_compact_static([], (1 << 24) + 1, ids.data_ptr(), count.data_ptr(), 0)
        assert e.value.status == aiq.ERR_CAPACITY
        ctx.free_table(table)
    finally:
        ctx.close()
