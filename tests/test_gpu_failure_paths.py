"""Failure paths reported as statuses, with no GPU fault: the context's device
byte cap (AIQ_ERR_OOM), a weight outside the fp16 operand range
(AIQ_ERR_UNSUPPORTED at load), and an activation that leaves the fp16 range
inside the forward pass (the kernels' own range check sets the device error
word: AIQ_ERR_DEVICE_CHECK).  After each failure the same context answers the
normal query exactly as a fresh context does.

The overflowing activation is an ordinary input (embedding rows of 1e5, a
bf16 value), not a fault: every kernel it passes through only does arithmetic
on it; no index, loop bound or wait depends on activation values, and the
decision of a NaN logit pair is "no" (a strict comparison)."""
import os

import numpy as np
import pytest

import synth
from helpers import gpu_ctx, weights_list
from paper_2608_10139_gb300 import aiq

pytestmark = pytest.mark.gpu

W_TINY = synth.C1_TINY


@pytest.fixture(scope="module")
def inputs():
    q = synth.make_inputs(W_TINY)
    W = synth.make_weights(W_TINY.model, W_TINY.weight_seed)
    return q, W


def _query(ctx, q, W, weights=None):
    t = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
    m = None
    try:
        m = ctx.load_model(W_TINY.model, weights_list(W_TINY.model, weights if weights is not None else W))
        preds = [(p.column, p.op, p.value) for p in W_TINY.preds]
        return ctx.run_select(t, m, preds, q.prefix, W_TINY.label_ids, agg=aiq.AGG_ROW_IDS,
                              flags=aiq.FLAG_LOGITS)
    finally:
        if m is not None:
            ctx.free_model(m)
        ctx.free_table(t)


@pytest.fixture(scope="module")
def fresh(inputs):
    c = gpu_ctx()
    try:
        yield _query(c, *inputs)
    finally:
        c.close()


def _same(a, b):
    assert a.count == b.count and np.array_equal(a.row_ids, b.row_ids)
    assert np.array_equal(a.cand_row_ids, b.cand_row_ids)
    assert np.array_equal(a.label_logits, b.label_logits)


def test_byte_cap_option_gives_oom_then_the_context_recovers(inputs, fresh):
    ctx = gpu_ctx()
    try:
        q, W = inputs
        t = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
        m = ctx.load_model(W_TINY.model, weights_list(W_TINY.model, W))
        preds = [(p.column, p.op, p.value) for p in W_TINY.preds]
        ctx.set_option("device_bytes_max", 1)           # below what the table and model hold
        for _ in range(2):
            with pytest.raises(aiq.AiqError) as e:
                ctx.run_select(t, m, preds, q.prefix, W_TINY.label_ids, agg=aiq.AGG_ROW_IDS, flags=aiq.FLAG_LOGITS)
            assert e.value.status == aiq.ERR_OOM and "AIQ_DEVICE_BYTES_MAX" in str(e.value)
        ctx.set_option("device_bytes_max", 0)           # lift the cap
        r = ctx.run_select(t, m, preds, q.prefix, W_TINY.label_ids, agg=aiq.AGG_ROW_IDS, flags=aiq.FLAG_LOGITS)
        _same(r, fresh)
        ctx.free_model(m)
        ctx.free_table(t)
    finally:
        ctx.close()


def test_byte_cap_from_the_environment(inputs, fresh):
    q, W = inputs
    old = os.environ.get("AIQ_DEVICE_BYTES_MAX")
    os.environ["AIQ_DEVICE_BYTES_MAX"] = "4096"
    try:
        ctx = gpu_ctx()
    finally:
        if old is None:
            del os.environ["AIQ_DEVICE_BYTES_MAX"]
        else:
            os.environ["AIQ_DEVICE_BYTES_MAX"] = old
    try:
        with pytest.raises(aiq.AiqError) as e:
            ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
        assert e.value.status == aiq.ERR_OOM
        ctx.set_option("device_bytes_max", 0)
        _same(_query(ctx, q, W), fresh)
    finally:
        ctx.close()


def test_weight_outside_the_fp16_range_is_rejected_at_load(inputs, fresh):
    q, W = inputs
    bad = dict(W)
    wq = W["l1.wq"].copy()
    wq[3, 5] = synth.f32_to_bf16_bits(np.array([-1.0e5], np.float32))[0]   # |w| > 65504
    bad["l1.wq"] = wq
    ctx = gpu_ctx()
    try:
        with pytest.raises(aiq.AiqError) as e:
            ctx.load_model(W_TINY.model, weights_list(W_TINY.model, bad))
        assert e.value.status == aiq.ERR_UNSUPPORTED and "fp16 range" in str(e.value)
        _same(_query(ctx, q, W), fresh)
    finally:
        ctx.close()


def test_activation_overflow_is_reported_then_the_context_recovers(inputs, fresh):
    q, W = inputs
    bad = dict(W)
    emb = W["embed"].copy()
    # every prefix token's embedding row at 1e5: the residual stream's fp16
    # copy (the operand of the first QKV GEMM) cannot hold it
    emb[np.unique(q.prefix)] = synth.f32_to_bf16_bits(np.array([1.0e5], np.float32))[0]
    bad["embed"] = emb
    ctx = gpu_ctx()
    try:
        for _ in range(2):
            with pytest.raises(aiq.AiqError) as e:
                _query(ctx, q, W, bad)
            assert e.value.status == aiq.ERR_DEVICE_CHECK and "fp16 range" in str(e.value)
        _same(_query(ctx, q, W), fresh)
    finally:
        ctx.close()
