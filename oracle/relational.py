"""Oracle, relational half: predicate, compaction, join, pack, decision, aggregate.

TEST INFRASTRUCTURE ONLY.  This module is the plain, slow, obviously correct
definition of what the unified AI query computes.  Only the tests, the
smoke check and the benchmark's CPU-baseline leg may import it; the product
path never does.  It shares no code with the CUDA path.

Every function restates a passage of the paper:
  * Table 1, WHERE row: a predicate is a vectorised boolean mask of
    ``column op constant`` terms; Table 2 Q2 conjoins it with AI_IF.
  * Table 1, FROM row and Fig. 2: the selected rows' text enters the language
    model; here each row's prompt is the shared prefix followed by its tokens.
  * Fig. 2: the decision compares the "yes" and "no" label logits at the
    last position with a strict greater-than.
  * Table 1, SELECT row and Fig. 2: the aggregate is a masked reduction over
    the decision mask (COUNT, the selected ids, or a GROUP BY count).
  * Section 4, datasets paragraph: reviews joined with movies on movie id.
  * Table 2 Q4: the self-join A.id = B.id AND A.review_id < B.review_id whose
    row pairs each get one AI_IF call on the concatenated texts.
"""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

import numpy as np

LT, LE, GT, GE, EQ, NE = 0, 1, 2, 3, 4, 5


def compare(values: np.ndarray, op: int, const) -> np.ndarray:
    """Element-wise ``values op const`` (Table 1, WHERE row)."""
    if op == LT:
        return values < const
    if op == LE:
        return values <= const
    if op == GT:
        return values > const
    if op == GE:
        return values >= const
    if op == EQ:
        return values == const
    if op == NE:
        return values != const
    raise ValueError(f"unknown comparison {op}")


def predicate_mask(cols: Dict[str, np.ndarray], preds: Sequence[Tuple[str, int, object]],
                   n_rows: int) -> np.ndarray:
    """Conjunction of ``column op constant`` terms; no terms selects every row."""
    mask = np.ones(n_rows, dtype=bool)
    for name, op, const in preds:
        mask &= compare(cols[name], op, const)
    return mask


def compact(mask: np.ndarray) -> np.ndarray:
    """Ids of the surviving rows in ascending row order (int32)."""
    return np.array([i for i in range(len(mask)) if mask[i]], dtype=np.int32) \
        if len(mask) <= 4096 else np.flatnonzero(mask).astype(np.int32)


def nested_loop_join(probe_keys: np.ndarray, probe_rows: np.ndarray,
                     build_keys: np.ndarray, build_rows: np.ndarray) -> List[Tuple[int, int]]:
    """Equi-join by brute force: every (probe row, build row) pair with equal
    keys, probe rows ascending then build rows ascending.  Tiny inputs only."""
    out = []
    for r in probe_rows:
        for m in build_rows:
            if probe_keys[r] == build_keys[m]:
                out.append((int(r), int(m)))
    return out


def dict_join(probe_keys: np.ndarray, probe_rows: np.ndarray,
              build_keys: np.ndarray, build_rows: np.ndarray) -> List[Tuple[int, int]]:
    """The same equi-join through a Python dict from key to build rows; used at
    sizes where the nested loop is too slow.  Same output order."""
    table: Dict[int, List[int]] = {}
    for m in build_rows:
        table.setdefault(int(build_keys[m]), []).append(int(m))
    out = []
    for r in probe_rows:
        for m in table.get(int(probe_keys[r]), ()):
            out.append((int(r), m))
    return out


def pack(prefix: np.ndarray, offsets: np.ndarray, tokens: np.ndarray,
         rows: np.ndarray):
    """Concatenate each selected row's prompt ``prefix ++ text`` in row order.

    Returns (packed token ids int32 [T], cu_seqlens int32 [S+1], positions
    int32 [T], last index int32 [S]).  Positions restart at 0 for every row;
    a row's last index is the packed position of its final token.
    """
    seqs = [np.concatenate([prefix, tokens[offsets[r]:offsets[r + 1]]]) for r in rows]
    lens = np.array([len(s) for s in seqs], dtype=np.int64)
    cu = np.zeros(len(rows) + 1, dtype=np.int64)
    cu[1:] = np.cumsum(lens)
    packed = np.concatenate(seqs).astype(np.int32) if seqs else np.zeros(0, np.int32)
    pos = np.concatenate([np.arange(n) for n in lens]).astype(np.int32) if seqs \
        else np.zeros(0, np.int32)
    last = (cu[1:] - 1).astype(np.int32)
    return packed, cu.astype(np.int32), pos, last


def decide(logits: np.ndarray) -> np.ndarray:
    """Per-row decision from label logits [S, K] (Fig. 2).

    K == 2: label 0 ("yes") wins only when strictly greater than label 1
    ("no"); a tie is "no".  Returns 1 for yes, 0 for no.
    K > 2 : index of the largest logit, the lowest index on ties.
    """
    logits = np.asarray(logits)
    s, k = logits.shape
    out = np.zeros(s, dtype=np.int32)
    for i in range(s):
        if k == 2:
            out[i] = 1 if logits[i, 0] > logits[i, 1] else 0
        else:
            best = 0
            for j in range(1, k):
                if logits[i, j] > logits[i, best]:
                    best = j
            out[i] = best
    return out


def margins(logits: np.ndarray, ref_decision: np.ndarray | None = None) -> np.ndarray:
    """K == 2: z_yes - z_no per row.  K > 2: z_k - z_{k*} for every k, with k*
    the reference argmax (``ref_decision``) or this logits' own argmax."""
    logits = np.asarray(logits, dtype=np.float64)
    if logits.shape[1] == 2:
        return logits[:, 0] - logits[:, 1]
    k_star = decide(logits) if ref_decision is None else ref_decision
    return logits - logits[np.arange(len(logits)), k_star][:, None]


def count_yes(decision: np.ndarray) -> int:
    """SELECT COUNT(*) ... WHERE AI_IF(...) = 1."""
    n = 0
    for d in decision:
        if d == 1:
            n += 1
    return n


def yes_row_ids(decision: np.ndarray, cand_rows: np.ndarray) -> np.ndarray:
    """Ids of the candidate rows whose decision is yes, ascending."""
    return np.array([int(r) for r, d in zip(cand_rows, decision) if d == 1], dtype=np.int32)


def masked_sum(decision: np.ndarray, cand_rows: np.ndarray, values: np.ndarray):
    """Fig. 2 / Table 1 SELECT row: SUM(values) over the rows decided yes (the
    masked reduction ``where(filter, values, 0).sum()``).  Integer columns sum
    exactly (Python integers); float columns are summed with correct rounding
    (math.fsum of the exact float64 values)."""
    import math
    picked = [values[int(r)] for r, d in zip(cand_rows, decision) if d == 1]
    if np.issubdtype(np.asarray(values).dtype, np.integer):
        return sum(int(v) for v in picked)
    return math.fsum(float(v) for v in picked)


def group_label_counts(decision: np.ndarray, k: int) -> np.ndarray:
    """GROUP BY label COUNT(*), all K labels including empty ones."""
    counts = np.zeros(k, dtype=np.int64)
    for d in decision:
        counts[d] += 1
    return counts


def group_build_counts(decision: np.ndarray, cand_build_rows: np.ndarray,
                       build_keys: np.ndarray):
    """GROUP BY build key COUNT(*) over the yes rows.  Groups with no yes row
    do not exist (the semantic filter is part of WHERE).  Output in ascending
    build-row order: (build rows int32, keys int64, counts int64)."""
    counts: Dict[int, int] = {}
    for d, m in zip(decision, cand_build_rows):
        if d == 1:
            counts[int(m)] = counts.get(int(m), 0) + 1
    rows = sorted(counts)
    return (np.array(rows, dtype=np.int32),
            np.array([build_keys[m] for m in rows], dtype=np.int64),
            np.array([counts[m] for m in rows], dtype=np.int64))


def like_contains(text: Sequence[int], pattern: Sequence[int]) -> bool:
    """SQL ``text LIKE '%pattern%'`` on token sequences (Table 2 Q5): true iff
    ``pattern`` occurs as a contiguous run of ``text``; an empty pattern
    matches every text, the empty one included."""
    t, p = list(text), list(pattern)
    if not p:
        return True
    return any(t[i:i + len(p)] == p for i in range(len(t) - len(p) + 1))


def self_join_pairs(keys: np.ndarray, rows: Sequence[int]) -> List[Tuple[int, int]]:
    """Table 2 Q4's self-join over the selected rows: every (a, b) with
    keys[a] == keys[b] and a < b (the row index is the review id), each
    unordered pair once, in ascending (a, b) order.  Nested loop."""
    rows = sorted(int(r) for r in rows)
    out = []
    for i, a in enumerate(rows):
        for b in rows[i + 1:]:
            if keys[a] == keys[b]:
                out.append((a, b))
    return out
