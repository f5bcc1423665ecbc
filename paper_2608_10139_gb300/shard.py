"""Row-range sharding of one AI query over replicas (one process per GPU).

Rows are independent and the model is replicated, as in the paper's
horizontal-scaling experiment (Table 5: one table split over the devices,
the same program on each).  Every rank holds the whole table (and, for a
join, the whole build side) and runs the query on a contiguous range of the
probe table's rows, expressed as two more conjunctive terms on an int32
row-id column.  The ranges are cut where the running count of the
candidates' prompt tokens (the prefill work, the query's cost) crosses
r / world of its total, from a relational-only pass that every rank runs
alike.  The only exchange is the merge of the small results at the end
(counts summed, row ids concatenated in rank order, group counts summed per
build row), never on the data path.
"""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

import numpy as np


def shard_range(n_rows: int, world: int, rank: int) -> Tuple[int, int]:
    """Contiguous, balanced [lo, hi) of rank `rank` out of `world`."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    base, extra = divmod(n_rows, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


ROW_ID = "row_id"
GE, LT = 3, 0   # comparison codes of the C-ABI (aiq_cmp)


def token_balanced_ranges(n_rows: int, cand_rows: np.ndarray, cand_tokens: np.ndarray,
                          world: int) -> List[Tuple[int, int]]:
    """Contiguous [lo, hi) ranges, one per rank, covering [0, n_rows) in order.

    cand_rows are the candidate rows (ascending) that reach the language model
    and cand_tokens their prompt tokens.  Rank r's range ends just after the
    first candidate at which the running token count reaches (r + 1) / world
    of the total, so every rank's share is within one row's tokens of
    total / world.  Without candidates the rows are split evenly."""
    if world <= 0:
        raise ValueError("world must be positive")
    cand_rows = np.asarray(cand_rows, np.int64)
    cum = np.cumsum(np.asarray(cand_tokens, np.int64))
    if len(cum) == 0 or cum[-1] <= 0:
        return [shard_range(n_rows, world, r) for r in range(world)]
    total = int(cum[-1])
    cuts = [0]
    for r in range(1, world):
        i = int(np.searchsorted(cum * world, total * r, side="left"))   # first cum >= total * r / world
        cuts.append(max(cuts[-1], min(n_rows, int(cand_rows[i]) + 1) if i < len(cum) else n_rows))
    cuts.append(n_rows)
    return [(cuts[r], cuts[r + 1]) for r in range(world)]


def range_terms(lo: int, hi: int):
    """The two conjunctive terms that restrict a query to rows [lo, hi) of a
    table carrying the int32 row-id column (column name, op, constant)."""
    return [(ROW_ID, GE, int(lo)), (ROW_ID, LT, int(hi))]


def with_row_ids(cols: Dict[str, np.ndarray], n_rows: int) -> Dict[str, np.ndarray]:
    """The table's columns plus the int32 row-id column the range terms read."""
    out = dict(cols)
    out[ROW_ID] = np.arange(n_rows, dtype=np.int32)
    return out


def local_result(res, row_offset: int) -> Dict[str, np.ndarray]:
    """The mergeable part of one rank's query result, with row ids made global."""
    return {
        "count": np.int64(res.count),
        "n_candidates": np.int64(res.n_candidates),
        "row_ids": res.row_ids.astype(np.int64) + row_offset,
        "label_counts": res.label_counts.astype(np.int64),
        "group_build_rows": res.group_build_rows.astype(np.int64),
        "group_keys": res.group_keys.astype(np.int64),
        "group_counts": res.group_counts.astype(np.int64),
    }


def merge(parts: Sequence[Dict[str, np.ndarray]]) -> Dict[str, np.ndarray]:
    """Merge rank results given in rank order (rank r covers rows below rank r+1)."""
    counts = [int(p["count"]) for p in parts]
    out = {
        # a negative count means "not defined for this aggregate" (e.g. K > 2 labels)
        "count": np.int64(-1 if any(c < 0 for c in counts) else sum(counts)),
        "n_candidates": np.int64(sum(int(p["n_candidates"]) for p in parts)),
        "row_ids": np.concatenate([p["row_ids"] for p in parts]) if parts else np.zeros(0, np.int64),
    }
    lcs = [p["label_counts"] for p in parts if len(p["label_counts"])]
    out["label_counts"] = np.sum(lcs, axis=0) if lcs else np.zeros(0, np.int64)
    groups: Dict[int, Tuple[int, int]] = {}
    for p in parts:
        for r, k, c in zip(p["group_build_rows"], p["group_keys"], p["group_counts"]):
            key, prev = int(r), groups.get(int(r), (int(k), 0))
            groups[key] = (prev[0], prev[1] + int(c))
    rows = sorted(groups)
    out["group_build_rows"] = np.array(rows, np.int64)
    out["group_keys"] = np.array([groups[r][0] for r in rows], np.int64)
    out["group_counts"] = np.array([groups[r][1] for r in rows], np.int64)
    return out


def gather_merge(part: Dict[str, np.ndarray], group=None) -> Dict[str, np.ndarray]:
    """All-gather every rank's part (torch.distributed, any backend) and merge."""
    import torch.distributed as dist
    parts: List[Dict[str, np.ndarray]] = [None] * dist.get_world_size(group)
    dist.all_gather_object(parts, part, group=group)
    return merge(parts)
