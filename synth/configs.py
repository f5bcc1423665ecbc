"""Workload shapes of the five synthetic AI-query configurations.

These are input recipes only: table sizes, value distributions, model shapes,
prompt prefix lengths, label token ids and the relational predicates.  They
hold none of the query's arithmetic.  The paper evaluates on SemBench Rotten
Tomatoes reviews joined with movies (Section 4, "Evaluation Queries and
Datasets") with Gemma-2B; seeded synthetic tables and random-init weights of
the shapes below stand in for both.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional, Tuple

# Comparison operators of a relational predicate ``column op constant``
# (Table 1, WHERE row; Table 2 Q2/Q3).  The numeric values are the C-ABI's.
LT, LE, GT, GE, EQ, NE = 0, 1, 2, 3, 4, 5
OP_NAMES = {LT: "<", LE: "<=", GT: ">", GE: ">=", EQ: "==", NE: "!="}

# Aggregate kinds applied after the semantic filter (Table 1, SELECT row).
AGG_COUNT, AGG_ROW_IDS, AGG_GROUP_LABEL, AGG_GROUP_BUILD_KEY = 0, 1, 2, 3


@dataclass(frozen=True)
class ModelShape:
    """Decoder-only Llama-style transformer shape (pre-norm, GQA, SwiGLU)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    rope_theta: float = 1.0e4
    rms_eps: float = 1.0e-5

    @property
    def q_dim(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    def layer_params(self) -> int:
        d = self.d_model
        return (2 * d + d * self.q_dim + 2 * d * self.kv_dim + self.q_dim * d
                + 3 * d * self.d_ffn)

    def linear_flops_per_token(self) -> int:
        """2 x (weights of the stack's linear layers) FLOPs for one token."""
        d = self.d_model
        per_layer = (d * (self.q_dim + 2 * self.kv_dim) + self.q_dim * d
                     + 3 * d * self.d_ffn)
        return 2 * per_layer * self.n_layers

    def attn_flops_per_pair(self) -> int:
        """QK^T and PV FLOPs for one causal (query, key) pair, all layers."""
        return 4 * self.n_heads * self.head_dim * self.n_layers


TINY = ModelShape(n_layers=2, d_model=128, n_heads=4, n_kv_heads=4, head_dim=32,
                  d_ffn=512, vocab=4096)
SHAPE_1B = ModelShape(n_layers=16, d_model=2048, n_heads=32, n_kv_heads=8,
                      head_dim=64, d_ffn=8192, vocab=32000)
SHAPE_8B = ModelShape(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=8,
                      head_dim=128, d_ffn=14336, vocab=128256)


@dataclass(frozen=True)
class TextRecipe:
    """Per-row token text: length distribution and Zipf token ids."""
    kind: str                 # "uniform" | "lognormal" | "fixed"
    lo: int
    hi: int
    median: float = 0.0       # lognormal median (tokens)
    sigma: float = 0.5        # lognormal sigma (the workloads leave it unstated)
    zipf_s: float = 1.1


@dataclass(frozen=True)
class Pred:
    column: str
    op: int
    value: int


@dataclass(frozen=True)
class Workload:
    name: str
    n_rows: int
    columns: Tuple[str, ...]            # int32 columns drawn uniform in their range
    text: TextRecipe
    preds: Tuple[Pred, ...]
    prefix_len: int
    model: ModelShape
    label_ids: Tuple[int, ...]
    agg: int
    data_seed: int
    weight_seed: int
    # join workloads: build side ("movies") filtered and joined on movie_id
    join_build_rows: int = 0
    join_build_preds: Tuple[Pred, ...] = ()
    join_zipf_s: float = 0.0


COLUMN_RANGES = {"rating": (1, 5), "year": (1950, 2024)}

YES_ID, NO_ID = 100, 101

C1_TINY = Workload(
    name="c1_tiny_select", n_rows=512, columns=("rating",),
    text=TextRecipe("uniform", 16, 48, zipf_s=1.1),
    preds=(Pred("rating", GE, 3),), prefix_len=16, model=TINY,
    label_ids=(YES_ID, NO_ID), agg=AGG_COUNT, data_seed=1001, weight_seed=2001)

C2_SELECT = Workload(
    name="c2_select_1b", n_rows=100_000, columns=("rating", "year"),
    text=TextRecipe("lognormal", 16, 512, median=120.0),
    preds=(Pred("rating", GE, 4), Pred("year", GE, 2000)), prefix_len=64,
    model=SHAPE_1B, label_ids=(YES_ID, NO_ID), agg=AGG_ROW_IDS,
    data_seed=1002, weight_seed=2002)

C3_JOIN = Workload(
    name="c3_join_1b", n_rows=500_000, columns=(),
    text=TextRecipe("lognormal", 16, 384, median=96.0),
    preds=(), prefix_len=64, model=SHAPE_1B, label_ids=(YES_ID, NO_ID),
    agg=AGG_GROUP_BUILD_KEY, data_seed=1003, weight_seed=2003,
    join_build_rows=50_000, join_build_preds=(Pred("year", GE, 2010),),
    join_zipf_s=1.05)

C4_MULTILABEL = Workload(
    name="c4_multilabel_8b", n_rows=20_000, columns=("rating",),
    text=TextRecipe("lognormal", 32, 1024, median=200.0),
    preds=(Pred("rating", LE, 2),), prefix_len=128, model=SHAPE_8B,
    label_ids=(100, 101, 102, 103, 104), agg=AGG_GROUP_LABEL,
    data_seed=1004, weight_seed=2004)

# Table 2 Q4 (pairwise AI_IF over the reviews self-joined on movie id): 20,000
# reviews spread uniformly over 2,000 movies (about 10 per movie; a skewed key
# would make the pair count quadratic in the head movie), score uniform 0..99,
# the filter score < 40 on both sides, the select workload's text recipe.
@dataclass(frozen=True)
class PairWorkload:
    name: str
    n_rows: int
    n_movies: int
    text: TextRecipe
    score_below: int
    prefix_len: int
    model: ModelShape
    label_ids: Tuple[int, ...]
    data_seed: int
    weight_seed: int


Q4_PAIRS = PairWorkload(
    name="q4_pairs_1b", n_rows=20_000, n_movies=2_000,
    text=TextRecipe("lognormal", 16, 512, median=120.0), score_below=40, prefix_len=64,
    model=SHAPE_1B, label_ids=(YES_ID, NO_ID), data_seed=1006, weight_seed=2002)


# Selectivity sweep thresholds ``rating >= R AND year >= Y`` on the c2 schema:
# P(rating>=R) * P(year>=Y) with rating uniform 1..5 and year uniform 1950..2024.
SWEEP_POINTS = {
    "1%": (5, 2021),    # 0.2 * 4/75  = 1.07 %
    "5%": (5, 2006),    # 0.2 * 19/75 = 5.07 %
    "25%": (4, 1978),   # 0.4 * 47/75 = 25.07 %
    "50%": (3, 1962),   # 0.6 * 63/75 = 50.4 %
    "100%": (1, 1950),  # everything
}


def sweep_workload(point: str, text_kind: str = "lognormal") -> Workload:
    r, y = SWEEP_POINTS[point]
    text = (TextRecipe("fixed", 64, 64) if text_kind == "fixed"
            else TextRecipe("lognormal", 16, 512, median=120.0))
    return Workload(
        name=f"c5_sweep_{point}_{text_kind}", n_rows=1_000_000,
        columns=("rating", "year"), text=text,
        preds=(Pred("rating", GE, r), Pred("year", GE, y)), prefix_len=64,
        model=SHAPE_1B, label_ids=(YES_ID, NO_ID), agg=AGG_ROW_IDS,
        data_seed=1005, weight_seed=2005)


WORKLOADS = {w.name: w for w in (C1_TINY, C2_SELECT, C3_JOIN, C4_MULTILABEL)}


def scaled(w: Workload, n_rows: int, model: Optional[ModelShape] = None,
           join_build_rows: Optional[int] = None) -> Workload:
    """Same recipe at another size (parity cases smaller than the workload)."""
    from dataclasses import replace
    kw = dict(n_rows=n_rows, name=f"{w.name}_n{n_rows}")
    if model is not None:
        kw["model"] = model
    if join_build_rows is not None:
        kw["join_build_rows"] = join_build_rows
    return replace(w, **kw)
