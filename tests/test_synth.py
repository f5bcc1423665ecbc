"""The seeded input generator: determinism, recipe bounds and distributions."""
import numpy as np
import torch

import synth


def test_deterministic_and_bounds():
    w = synth.scaled(synth.C2_SELECT, 3000)
    a, b = synth.make_inputs(w), synth.make_inputs(w)
    assert np.array_equal(a.table.tokens, b.table.tokens)
    assert np.array_equal(a.table.cols["year"], b.table.cols["year"])
    lens = np.diff(a.table.offsets)
    assert lens.min() >= 16 and lens.max() <= 512
    assert 100 <= np.median(lens) <= 140            # lognormal median 120
    assert a.table.tokens.min() >= 0 and a.table.tokens.max() < w.model.vocab
    assert set(np.unique(a.table.cols["rating"])) <= set(range(1, 6))
    assert a.table.cols["year"].min() >= 1950 and a.table.cols["year"].max() <= 2024
    assert len(a.prefix) == 64


def test_zipf_head_frequency():
    rng = np.random.Generator(np.random.PCG64(0))
    s, v, n = 1.1, 4096, 400_000
    r = synth.zipf_ranks(rng, n, v, s)
    h = np.sum(np.arange(1, v + 1, dtype=np.float64) ** -s)
    for k in (1, 2, 10):
        assert abs(np.mean(r == k - 1) - k ** -s / h) < 4e-3


def test_join_tables():
    w = synth.scaled(synth.C3_JOIN, 20_000, join_build_rows=2000)
    q = synth.make_inputs(w)
    ids = q.build.cols["movie_id"]
    assert len(np.unique(ids)) == len(ids) and ids.min() >= 0
    assert np.isin(q.table.cols["movie_id"], ids).all()      # every FK has its movie
    _, counts = np.unique(q.table.cols["movie_id"], return_counts=True)
    assert counts.max() / len(q.table.cols["movie_id"]) > 0.05   # Zipf(1.05) head


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(1).standard_normal(10_000).astype(np.float32) * 3
    x[:4] = [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 0.0]   # ties to even
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(synth.f32_to_bf16_bits(x), want)


def test_weights_shapes_and_scale():
    s = synth.TINY
    w = synth.make_weights(s, 5)
    specs = synth.weight_specs(s)
    assert list(w) == [n for n, _, _ in specs]
    assert len(specs) == 1 + 9 * s.n_layers + 3
    e = synth.bf16_bits_to_f32(w["embed"])
    assert abs(e.std() - 0.02) < 1e-3
    g = synth.bf16_bits_to_f32(w["l0.attn_norm"])
    assert abs(g.mean() - 1.0) < 0.01
