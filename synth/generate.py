"""Seeded synthetic tables and random-init decoder weights.

Everything here is input generation: random draws in a fixed order from
numpy's PCG64, the bounded Zipf and lognormal recipes, and round-to-nearest-
even conversion of float32 draws to bfloat16 bit patterns.  Both the oracle
and the CUDA path consume these arrays; neither side's arithmetic lives here.

Draw order (fixed, so that a seed names one table):
  select table : int32 columns in ``Workload.columns`` order, text lengths,
                 token ids, then the prompt prefix.
  join tables  : build ``movie_id`` (distinct 63-bit), build ``year``,
                 probe foreign-key ranks, probe text lengths, probe tokens,
                 prefix; the rank -> build row permutation comes last.
  weights      : tensor i of ``weight_specs`` drawn from its own PCG64
                 stream, child i of SeedSequence(seed), as float32 standard
                 normals (so tensors can be generated in parallel).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np

from .configs import COLUMN_RANGES, ModelShape, PairWorkload, TextRecipe, Workload


# ---------------------------------------------------------------- tables ---

@dataclass
class Table:
    """Columnar table: fixed-width int columns plus one CSR token column."""
    n_rows: int
    cols: Dict[str, np.ndarray]
    offsets: Optional[np.ndarray] = None    # int64 [n_rows + 1]
    tokens: Optional[np.ndarray] = None     # int32 [offsets[-1]]

    def text(self, i: int) -> np.ndarray:
        return self.tokens[self.offsets[i]:self.offsets[i + 1]]

    def nbytes(self) -> int:
        b = sum(int(c.nbytes) for c in self.cols.values())
        if self.offsets is not None:
            b += int(self.offsets.nbytes) + int(self.tokens.nbytes)
        return b


@dataclass
class QueryInputs:
    """One workload's inputs: the table(s) and the prompt prefix."""
    table: Table                     # the select table, or the probe side
    prefix: np.ndarray               # int32 [P]
    build: Optional[Table] = None    # join build side (movies)


def zipf_ranks(rng: np.random.Generator, n: int, support: int, s: float) -> np.ndarray:
    """Bounded Zipf draws by inverse CDF: P(rank k) proportional to k**-s,
    k = 1..support.  Returns ``k - 1`` (0-based), int64."""
    w = np.arange(1, support + 1, dtype=np.float64) ** (-s)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    u = rng.random(n)
    k = np.searchsorted(cdf, u, side="right")
    return np.minimum(k, support - 1).astype(np.int64)


def text_lengths(rng: np.random.Generator, n: int, t: TextRecipe) -> np.ndarray:
    if t.kind == "uniform":
        return rng.integers(t.lo, t.hi + 1, n).astype(np.int64)
    if t.kind == "fixed":
        return np.full(n, t.lo, dtype=np.int64)
    if t.kind == "lognormal":
        x = np.exp(rng.normal(np.log(t.median), t.sigma, n))
        return np.clip(np.rint(x), t.lo, t.hi).astype(np.int64)
    raise ValueError(t.kind)


def _text_column(rng, n, t: TextRecipe, vocab: int):
    lens = text_lengths(rng, n, t)
    offsets = np.zeros(n + 1, dtype=np.int64)
    np.cumsum(lens, out=offsets[1:])
    tokens = zipf_ranks(rng, int(offsets[-1]), vocab, t.zipf_s).astype(np.int32)
    return offsets, tokens


def make_select_inputs(w: Workload) -> QueryInputs:
    rng = np.random.Generator(np.random.PCG64(w.data_seed))
    cols = {}
    for name in w.columns:
        lo, hi = COLUMN_RANGES[name]
        cols[name] = rng.integers(lo, hi + 1, w.n_rows).astype(np.int32)
    offsets, tokens = _text_column(rng, w.n_rows, w.text, w.model.vocab)
    prefix = rng.integers(0, w.model.vocab, w.prefix_len).astype(np.int32)
    return QueryInputs(Table(w.n_rows, cols, offsets, tokens), prefix)


def distinct_int63(rng: np.random.Generator, n: int) -> np.ndarray:
    """n distinct non-negative 63-bit integers (resampling collisions)."""
    out = rng.integers(0, 2 ** 63 - 1, n, dtype=np.int64)
    while True:
        _, first = np.unique(out, return_index=True)
        if len(first) == n:
            return out
        dup = np.ones(n, dtype=bool)
        dup[first] = False
        out[dup] = rng.integers(0, 2 ** 63 - 1, int(dup.sum()), dtype=np.int64)


def make_join_inputs(w: Workload) -> QueryInputs:
    """movies(movie_id int64 unique, year int32) and
    reviews(movie_id int64 FK with Zipf(join_zipf_s) skew, text)."""
    rng = np.random.Generator(np.random.PCG64(w.data_seed))
    m = w.join_build_rows
    movie_id = distinct_int63(rng, m)
    lo, hi = COLUMN_RANGES["year"]
    year = rng.integers(lo, hi + 1, m).astype(np.int32)
    ranks = zipf_ranks(rng, w.n_rows, m, w.join_zipf_s)
    offsets, tokens = _text_column(rng, w.n_rows, w.text, w.model.vocab)
    prefix = rng.integers(0, w.model.vocab, w.prefix_len).astype(np.int32)
    perm = rng.permutation(m)
    fk = movie_id[perm[ranks]]
    movies = Table(m, {"movie_id": movie_id, "year": year})
    reviews = Table(w.n_rows, {"movie_id": fk}, offsets, tokens)
    return QueryInputs(reviews, prefix, build=movies)


def make_pair_inputs(w: PairWorkload) -> QueryInputs:
    """reviews(movie_id int64 uniform over n_movies distinct 63-bit ids,
    score int32 uniform 0..99, text) for the Q4 self-join.  Draw order:
    movie ids, the movie of each review, scores, text lengths, tokens, prefix."""
    rng = np.random.Generator(np.random.PCG64(w.data_seed))
    movie_ids = distinct_int63(rng, w.n_movies)
    movie = movie_ids[rng.integers(0, w.n_movies, w.n_rows)]
    score = rng.integers(0, 100, w.n_rows).astype(np.int32)
    offsets, tokens = _text_column(rng, w.n_rows, w.text, w.model.vocab)
    prefix = rng.integers(0, w.model.vocab, w.prefix_len).astype(np.int32)
    return QueryInputs(Table(w.n_rows, {"movie_id": movie, "score": score}, offsets, tokens), prefix)


def make_inputs(w: Workload) -> QueryInputs:
    return make_join_inputs(w) if w.join_build_rows else make_select_inputs(w)


# --------------------------------------------------------------- weights ---

def weight_specs(s: ModelShape) -> List[Tuple[str, Tuple[int, ...], str]]:
    """Fixed tensor order of a model: (name, shape, init).  Linear weights are
    stored [out_features, in_features] (y = x W^T).  init "normal" is
    0.02 * N(0,1); "gain" is 1 + 0.02 * N(0,1)."""
    d, qd, kd, f = s.d_model, s.q_dim, s.kv_dim, s.d_ffn
    specs = [("embed", (s.vocab, d), "normal")]
    for l in range(s.n_layers):
        specs += [
            (f"l{l}.attn_norm", (d,), "gain"),
            (f"l{l}.wq", (qd, d), "normal"),
            (f"l{l}.wk", (kd, d), "normal"),
            (f"l{l}.wv", (kd, d), "normal"),
            (f"l{l}.wo", (d, qd), "normal"),
            (f"l{l}.mlp_norm", (d,), "gain"),
            (f"l{l}.wg", (f, d), "normal"),
            (f"l{l}.wu", (f, d), "normal"),
            (f"l{l}.wd", (d, f), "normal"),
        ]
    specs += [("final_norm", (d,), "gain"), ("lm_head", (s.vocab, d), "normal"),
              ("lm_bias", (s.vocab,), "normal")]
    return specs


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _draw_tensor(seed_seq, shape, init) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed_seq))
    n = int(np.prod(shape))
    bits = np.empty(n, dtype=np.uint16)
    step = 1 << 24
    for i in range(0, n, step):
        k = min(step, n - i)
        x = rng.standard_normal(k, dtype=np.float32)
        x *= np.float32(0.02)
        if init == "gain":
            x += np.float32(1.0)
        bits[i:i + k] = f32_to_bf16_bits(x)
    return bits.reshape(shape)


def make_weights(s: ModelShape, seed: int, zero: bool = False, threads: int = 0) -> Dict[str, np.ndarray]:
    """Random-init bf16 weights (uint16 bit patterns), keyed by spec name."""
    import concurrent.futures as cf
    import os
    specs = weight_specs(s)
    if zero:
        return {name: np.zeros(shape, dtype=np.uint16) for name, shape, _ in specs}
    children = np.random.SeedSequence(seed).spawn(len(specs))
    threads = threads or min(16, os.cpu_count() or 1)
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        arrays = list(ex.map(lambda a: _draw_tensor(*a),
                             [(c, shape, init) for c, (_, shape, init) in zip(children, specs)]))
    return {name: a for (name, _, _), a in zip(specs, arrays)}
