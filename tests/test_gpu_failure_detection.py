"""Device-side failure detection without a GPU fault: every pipelined kernel
waits on its mbarriers through one bounded wait.  The self-test kernel makes
that wait run out on a phase that nothing completes and checks that the call
reports it, that the CTA's abort flag releases the other waiting warp early,
and that the context keeps working afterwards."""
import time

import numpy as np
import pytest

import synth
from helpers import gpu_ctx, weights_list
from paper_2608_10139_gb300 import aiq

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = gpu_ctx()
    yield c
    c.close()


def _tiny_query(ctx):
    w = synth.C1_TINY
    q = synth.make_inputs(w)
    t = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
    m = ctx.load_model(w.model, weights_list(w.model, synth.make_weights(w.model, w.weight_seed)))
    preds = [(p.column, p.op, p.value) for p in w.preds]
    r = ctx.run_select(t, m, preds, q.prefix, w.label_ids, agg=aiq.AGG_ROW_IDS, flags=aiq.FLAG_LOGITS)
    ctx.free_model(m)
    ctx.free_table(t)
    return r


def test_expired_wait_is_reported_and_the_context_stays_usable(ctx):
    before = _tiny_query(ctx)
    limit = 100_000_000                        # 0.1 s; warp 1 alone would wait 0.4 s
    for _ in range(2):
        t0 = time.perf_counter()
        with pytest.raises(aiq.AiqError) as e:
            ctx.op_wait_expiry_selftest(limit)
        dt = time.perf_counter() - t0
        assert e.value.status == aiq.ERR_DEVICE_CHECK and "bounded wait expired" in str(e.value)
        assert limit * 1e-9 <= dt < 0.35, f"the self-test returned after {dt:.3f} s"
    # the device error word was cleared: the same query gives the same answer
    after = _tiny_query(ctx)
    assert after.count == before.count and np.array_equal(after.row_ids, before.row_ids)
    assert np.array_equal(after.label_logits, before.label_logits)


def test_selftest_rejects_out_of_range_limits(ctx):
    for bad in (0, 999, 1_000_000_001):
        with pytest.raises(aiq.AiqError) as e:
            ctx.op_wait_expiry_selftest(bad)
        assert e.value.status == aiq.ERR_INVALID_ARG
