"""Oracle, whole query: the unified AI query's result from its plain definition.

TEST INFRASTRUCTURE ONLY (tests, smoke check, benchmark CPU-baseline leg).

``run_select`` follows Table 2 Q1/Q2 with Fig. 2's decision: WHERE relational
terms AND AI_IF(text) = 1, then the aggregate.  ``run_transform`` follows
Table 2 Q3 (SELECT AI_TRANSFORM(text) ... WHERE relational terms: greedy
generation for every candidate row) and Q5 (COUNT(*) of the rows whose
generated text is LIKE '%pattern%', with the matching rows' outputs as the
debug payload).  ``run_pair_select`` follows Q4: the selected rows are
self-joined on a key (A.id = B.id AND A.review_id < B.review_id) and every
pair gets one AI_IF call on prefix ++ text(A) ++ text(B).  ``run_join_select`` adds the
reviews-movies equi-join on movie id of Section 4's datasets paragraph, with
the build-side (movies) predicate, and groups the yes rows by movie.

With ``sample`` set, the relational results are computed in full and the
transformer only for the sampled candidate positions; the aggregate of a
sampled run is then the caller's business (``aggregate`` applied to a full
decision vector).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import relational as rel
from . import transformer as tf

AGG_COUNT, AGG_ROW_IDS, AGG_GROUP_LABEL, AGG_GROUP_BUILD_KEY, AGG_SUM = 0, 1, 2, 3, 4


@dataclass
class OracleResult:
    cand_rows: np.ndarray            # probe/select rows that reach the LM, ascending
    cand_build_rows: Optional[np.ndarray]  # joins: matching build row per candidate
    sample: np.ndarray               # candidate positions the LM was run on
    logits: np.ndarray               # [len(sample), K] float64
    decision: np.ndarray             # decisions of the sampled candidates
    agg: Optional[dict]              # aggregate (only when every candidate ran)


def prompts(prefix: np.ndarray, offsets: np.ndarray, tokens: np.ndarray,
            rows: Sequence[int]) -> List[np.ndarray]:
    """Each row's prompt: shared prefix followed by the row's tokens."""
    return [np.concatenate([prefix, tokens[offsets[r]:offsets[r + 1]]]).astype(np.int64)
            for r in rows]


def aggregate(agg: int, decision: np.ndarray, cand_rows: np.ndarray, k: int,
              cand_build_rows: Optional[np.ndarray] = None,
              build_keys: Optional[np.ndarray] = None,
              sum_values: Optional[np.ndarray] = None) -> dict:
    """Masked aggregate over a full decision vector (Table 1, SELECT row)."""
    out = {}
    if k == 2:
        out["count"] = rel.count_yes(decision)
    if agg == AGG_SUM:
        out["sum"] = rel.masked_sum(decision, cand_rows, sum_values)
    elif agg == AGG_ROW_IDS:
        out["row_ids"] = rel.yes_row_ids(decision, cand_rows)
    elif agg == AGG_GROUP_LABEL:
        out["label_counts"] = rel.group_label_counts(decision, k)
    elif agg == AGG_GROUP_BUILD_KEY:
        rows, keys, counts = rel.group_build_counts(decision, cand_build_rows, build_keys)
        out["group_build_rows"], out["group_keys"], out["group_counts"] = rows, keys, counts
    return out


def _finish(model, prefix, table, cand_rows, cand_build_rows, labels, agg,
            sample, build_keys):
    n = len(cand_rows)
    sample = np.arange(n) if sample is None else np.asarray(sample, dtype=np.int64)
    seqs = prompts(prefix, table.offsets, table.tokens, cand_rows[sample])
    logits = tf.label_logits(model, seqs, labels)
    decision = rel.decide(logits) if len(seqs) else np.zeros(0, np.int32)
    full = len(sample) == n and np.array_equal(sample, np.arange(n))
    res = None
    if full:
        res = aggregate(agg, decision, cand_rows, len(labels), cand_build_rows, build_keys)
    return OracleResult(cand_rows, cand_build_rows, sample, logits, decision, res)


def run_select(table, prefix, preds, labels, agg, model: tf.Model,
               sample: Optional[np.ndarray] = None) -> OracleResult:
    """preds: (column name, op, constant) triples, conjoined."""
    mask = rel.predicate_mask(table.cols, preds, table.n_rows)
    cand = rel.compact(mask)
    return _finish(model, prefix, table, cand, None, labels, agg, sample, None)


def join_candidates(probe, build, probe_key: str, build_key: str, probe_preds,
                    build_preds, brute_force: bool = False):
    """Joined (probe row, build row) pairs after both sides' predicates,
    ascending probe row."""
    pm = rel.predicate_mask(probe.cols, probe_preds, probe.n_rows)
    bm = rel.predicate_mask(build.cols, build_preds, build.n_rows)
    join = rel.nested_loop_join if brute_force else rel.dict_join
    pairs = join(probe.cols[probe_key], rel.compact(pm), build.cols[build_key], rel.compact(bm))
    cand = np.array([p for p, _ in pairs], dtype=np.int32)
    cand_b = np.array([m for _, m in pairs], dtype=np.int32)
    return cand, cand_b


def run_join_select(probe, build, probe_key: str, build_key: str, probe_preds,
                    build_preds, prefix, labels, agg, model: tf.Model,
                    sample: Optional[np.ndarray] = None,
                    brute_force: bool = False) -> OracleResult:
    cand, cand_b = join_candidates(probe, build, probe_key, build_key, probe_preds,
                                   build_preds, brute_force)
    return _finish(model, prefix, probe, cand, cand_b, labels, agg, sample,
                   build.cols[build_key])


@dataclass
class TransformResult:
    cand_rows: np.ndarray          # rows that reach the LM, ascending
    sample: np.ndarray             # candidate positions the LM was run on
    tokens: np.ndarray             # [len(sample), n_new] generated ids (pad after eos)
    text_len: np.ndarray           # [len(sample)] tokens before the eos
    match: Optional[np.ndarray]    # LIKE result per sampled candidate (None: no LIKE)
    agg: Optional[dict]            # LIKE: count and matching row ids, when every candidate ran


def like_aggregate(match: np.ndarray, cand_rows: np.ndarray) -> dict:
    """Table 2 Q5: COUNT(*) of the LIKE matches and their row ids (ascending)."""
    match = np.asarray(match, dtype=bool)
    return {"count": int(match.sum()), "row_ids": np.asarray(cand_rows)[match].astype(np.int32)}


def run_transform(table, prefix, preds, model: tf.Model, n_new: int, eos: int = -1,
                  pad: int = 0, like: Optional[Sequence[int]] = None,
                  sample: Optional[np.ndarray] = None) -> TransformResult:
    """WHERE ``preds``, then greedy AI_TRANSFORM of each candidate's prompt
    (prefix ++ row tokens), then the optional LIKE '%like%' filter applied to
    each output's text (the tokens before its eos)."""
    cand = rel.compact(rel.predicate_mask(table.cols, preds, table.n_rows))
    n = len(cand)
    sample = np.arange(n) if sample is None else np.asarray(sample, dtype=np.int64)
    seqs = prompts(prefix, table.offsets, table.tokens, cand[sample])
    toks = np.zeros((len(seqs), n_new), dtype=np.int64)
    lens = np.zeros(len(seqs), dtype=np.int64)
    for i, q in enumerate(seqs):
        toks[i], lens[i] = tf.greedy_generate(model, q, n_new, eos, pad)
    match = None
    agg = None
    if like is not None:
        match = np.array([rel.like_contains(toks[i, :lens[i]], like) for i in range(len(seqs))], dtype=bool)
        if len(sample) == n and np.array_equal(sample, np.arange(n)):
            agg = like_aggregate(match, cand)
    return TransformResult(cand, sample, toks, lens, match, agg)


def pair_prompts(prefix: np.ndarray, offsets: np.ndarray, tokens: np.ndarray,
                 pairs: Sequence[Tuple[int, int]]) -> List[np.ndarray]:
    """Q4's prompt for a pair: the shared prefix, then A's text, then B's."""
    return [np.concatenate([prefix, tokens[offsets[a]:offsets[a + 1]],
                            tokens[offsets[b]:offsets[b + 1]]]).astype(np.int64) for a, b in pairs]


@dataclass
class PairResult:
    pairs: np.ndarray          # [n_pairs, 2] (a, b), ascending
    sample: np.ndarray         # pair positions the LM was run on
    logits: np.ndarray         # [len(sample), K]
    decision: np.ndarray       # decisions of the sampled pairs
    agg: Optional[dict]        # COUNT and the yes pairs, when every pair ran


def pair_aggregate(decision: np.ndarray, pairs: np.ndarray) -> dict:
    """COUNT(*) of the pairs decided yes and those pairs, ascending."""
    yes = np.asarray(decision) == 1
    return {"count": int(yes.sum()), "yes_pairs": np.asarray(pairs).reshape(-1, 2)[yes]}


def run_pair_select(table, key: str, preds, prefix, labels, model: tf.Model,
                    sample: Optional[np.ndarray] = None) -> PairResult:
    """WHERE ``preds`` on both sides (the predicate filters the relation before
    it is joined with itself), the key self-join, then AI_IF per pair."""
    cand = rel.compact(rel.predicate_mask(table.cols, preds, table.n_rows))
    pairs = np.array(rel.self_join_pairs(table.cols[key], cand), dtype=np.int64).reshape(-1, 2)
    n = len(pairs)
    sample = np.arange(n) if sample is None else np.asarray(sample, dtype=np.int64)
    seqs = pair_prompts(prefix, table.offsets, table.tokens, [tuple(p) for p in pairs[sample]])
    logits = tf.label_logits(model, seqs, labels)
    decision = rel.decide(logits) if len(seqs) else np.zeros(0, np.int32)
    agg = None
    if len(sample) == n and np.array_equal(sample, np.arange(n)):
        agg = pair_aggregate(decision, pairs)
    return PairResult(pairs, sample, logits, decision, agg)
