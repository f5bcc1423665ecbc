"""The CPU emulation of the GPU path's fp16 rounding points (precision_emulation.py)
is the evidence behind the precision analysis, so it is checked against the
oracle here: with no rounding point on, its reordered layer (norm gain applied
before the QKV product, 1/rms after it) is the oracle's decoder layer; every
rounding point perturbs the layer, and only by fp16-sized amounts."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import precision_emulation as pe  # noqa: E402
import synth  # noqa: E402
from oracle import transformer as tf  # noqa: E402

GQA = synth.ModelShape(n_layers=2, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32,
                       d_ffn=384, vocab=512)


@pytest.fixture(scope="module")
def setup():
    m = tf.Model(GQA, synth.make_weights(GQA, 77))
    rng = np.random.default_rng(5)
    x = m.embed_rows(rng.integers(0, GQA.vocab, 37))
    lw = {n: m.get(f"l0.{n}") for n in tf.LAYER_TENSORS}
    return m, x, lw


def test_no_rounding_point_is_the_oracle_layer(setup):
    m, x, lw = setup
    ref = tf.decoder_layer(x, m, 0, lw)
    got = pe.layer(x, GQA, lw, set())
    assert np.max(np.abs(got - ref)) <= 1e-12 * np.max(np.abs(ref))


@pytest.mark.parametrize("point", pe.POINTS)
def test_each_rounding_point_is_an_fp16_sized_perturbation(setup, point):
    m, x, lw = setup
    ref = tf.decoder_layer(x, m, 0, lw)
    got = pe.layer(x, GQA, lw, {point})
    err = np.max(np.abs(got - ref)) / np.max(np.abs(ref))
    assert 0 < err < 2e-3, (point, err)


def test_attention_without_rounding_is_the_oracle_attention():
    rng = np.random.default_rng(9)
    q = rng.standard_normal((19, 4, 16))
    k = rng.standard_normal((19, 2, 16))
    v = rng.standard_normal((19, 2, 16))
    ref = tf.causal_attention(q, k, v)
    assert np.allclose(pe.attention(q, k, v, False), ref, rtol=0, atol=1e-13)
    assert not np.array_equal(pe.attention(q, k, v, True), ref)


def test_variant_names():
    assert pe.parse_variant("all") == set(pe.POINTS)
    assert pe.parse_variant("none") == set()
    assert pe.parse_variant("mlpn+swiglu") == {"mlpn", "swiglu"}
    with pytest.raises(SystemExit):
        pe.parse_variant("qkv+bogus")
