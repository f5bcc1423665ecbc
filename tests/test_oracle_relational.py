"""Pins of the oracle's relational half against hand-worked cases, brute force
and invariants (CPU only)."""
import operator
import os

import numpy as np
import pytest

from oracle import relational as rel
from oracle import query as oq

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read(name):
    rows = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        k, *v = line.split()
        rows.setdefault(k, []).append([int(x) if x.lstrip("-").isdigit() else float(x) for x in v])
    return rows


def test_where_and_hand_worked():
    g = _read("where_and.txt")
    cols = {"rating": np.array(g["rating"][0], np.int32), "year": np.array(g["year"][0], np.int32)}
    mask = rel.predicate_mask(cols, [("rating", rel.GE, 4), ("year", rel.GE, 2000)], 10)
    assert rel.compact(mask).tolist() == g["expect"][0]


@pytest.mark.parametrize("op,pyop", [(rel.LT, operator.lt), (rel.LE, operator.le),
                                     (rel.GT, operator.gt), (rel.GE, operator.ge),
                                     (rel.EQ, operator.eq), (rel.NE, operator.ne)])
def test_compare_ops_match_python(op, pyop):
    vals = np.array([-3, 0, 2, 2, 7], np.int64)
    got = rel.compare(vals, op, 2)
    assert got.tolist() == [pyop(int(v), 2) for v in vals]


@pytest.mark.parametrize("n", [0, 1, 31, 32, 33, 1000, 4096, 4097, 100_003])
def test_compaction_brute_force(n):
    rng = np.random.default_rng(n)
    cols = {"a": rng.integers(0, 10, n).astype(np.int32), "b": rng.integers(-5, 5, n).astype(np.int64)}
    preds = [("a", rel.GE, 4), ("b", rel.NE, 0)]
    ids = rel.compact(rel.predicate_mask(cols, preds, n))
    brute = [i for i in range(n) if cols["a"][i] >= 4 and cols["b"][i] != 0]
    assert ids.tolist() == brute
    mask = rel.predicate_mask(cols, preds, n)
    assert len(ids) == int(mask.sum())                      # size == popcount
    assert np.all(np.diff(ids) > 0)                         # order preserved
    assert rel.compact(np.zeros(n, bool)).size == 0          # nothing survives
    assert rel.compact(np.ones(n, bool)).tolist() == list(range(n))  # everything


def test_no_predicate_selects_all():
    assert rel.predicate_mask({}, [], 5).all()


def test_join_hand_worked():
    g = _read("join_small.txt")
    bkeys = np.array([m[1] for m in g["movie"]], np.int64)
    byear = np.array([m[2] for m in g["movie"]], np.int32)
    pkeys = np.array([r[1] for r in g["review"]], np.int64)
    bm = rel.compact(rel.predicate_mask({"year": byear}, [("year", rel.GE, 2010)], len(bkeys)))
    pr = np.arange(len(pkeys), dtype=np.int32)
    want = [tuple(p) for p in g["pair"]]
    assert rel.nested_loop_join(pkeys, pr, bkeys, bm) == want
    assert rel.dict_join(pkeys, pr, bkeys, bm) == want


@pytest.mark.parametrize("seed", range(5))
def test_dict_join_equals_nested_loop_with_orphans_and_duplicates(seed):
    rng = np.random.default_rng(seed)
    bkeys = rng.integers(0, 30, 25).astype(np.int64)   # duplicate build keys too
    pkeys = rng.integers(0, 40, 60).astype(np.int64)   # orphans (no match) and repeats
    br = np.flatnonzero(rng.random(25) < 0.7).astype(np.int32)
    pr = np.flatnonzero(rng.random(60) < 0.8).astype(np.int32)
    nl = rel.nested_loop_join(pkeys, pr, bkeys, br)
    assert rel.dict_join(pkeys, pr, bkeys, br) == nl
    # cardinality closed form: sum over probe rows of matching build rows
    card = sum(int(np.sum(bkeys[br] == pkeys[r])) for r in pr)
    assert len(nl) == card


def test_pack_layout():
    prefix = np.array([7, 8], np.int32)
    offsets = np.array([0, 3, 3 + 1, 3 + 1 + 2], np.int64)
    tokens = np.array([1, 2, 3, 4, 5, 6], np.int32)
    packed, cu, pos, last = rel.pack(prefix, offsets, tokens, np.array([0, 2], np.int32))
    assert packed.tolist() == [7, 8, 1, 2, 3, 7, 8, 5, 6]
    assert cu.tolist() == [0, 5, 9]
    assert pos.tolist() == [0, 1, 2, 3, 4, 0, 1, 2, 3]
    assert last.tolist() == [4, 8]
    e = rel.pack(prefix, offsets, tokens, np.zeros(0, np.int32))
    assert e[0].size == 0 and e[1].tolist() == [0] and e[3].size == 0


def test_decide_strict_and_ties():
    z = np.array([[1.0, 0.5], [0.5, 0.5], [-1.0, -2.0], [0.0, 1e-30]])
    assert rel.decide(z).tolist() == [1, 0, 1, 0]          # strict >, tie -> no
    z5 = np.array([[0, 3, 3, 1, 2], [5, 5, 5, 5, 5], [-1, -2, -3, -4, -0.5]], float)
    assert rel.decide(z5).tolist() == [1, 0, 4]             # first index on ties


def test_aggregate_invariants():
    rng = np.random.default_rng(3)
    s = 200
    dec = rng.integers(0, 2, s).astype(np.int32)
    cand = np.sort(rng.choice(10_000, s, replace=False)).astype(np.int32)
    bro = rng.integers(0, 20, s).astype(np.int32)
    bkeys = rng.integers(-100, 100, 20).astype(np.int64)
    a = oq.aggregate(oq.AGG_ROW_IDS, dec, cand, 2)
    assert a["count"] == len(a["row_ids"]) == int(dec.sum())
    assert np.all(np.diff(a["row_ids"]) > 0)
    g = oq.aggregate(oq.AGG_GROUP_BUILD_KEY, dec, cand, 2, bro, bkeys)
    assert int(g["group_counts"].sum()) == g["count"]       # groups sum to yes count
    assert np.all(g["group_counts"] > 0)                   # non-empty groups only
    assert np.all(np.diff(g["group_build_rows"]) > 0)       # ascending build row
    assert g["group_keys"].tolist() == bkeys[g["group_build_rows"]].tolist()
    dec5 = rng.integers(0, 5, s).astype(np.int32)
    lc = oq.aggregate(oq.AGG_GROUP_LABEL, dec5, cand, 5)["label_counts"]
    assert lc.sum() == s and lc.tolist() == [int(np.sum(dec5 == k)) for k in range(5)]


def test_masked_sum_hand_cases_and_exactness():
    dec = np.array([1, 0, 1, 1], np.int32)
    cand = np.array([0, 2, 3, 5], np.int32)
    vals = np.array([10, 20, 30, 40, 50, 60], np.int32)
    assert rel.masked_sum(dec, cand, vals) == 10 + 40 + 60
    assert rel.masked_sum(np.zeros(4, np.int32), cand, vals) == 0
    big = np.array([2 ** 62, 2 ** 62, -5], np.int64)                       # exact beyond float64
    assert rel.masked_sum(np.ones(3, np.int32), np.arange(3), big) == 2 ** 63 - 5
    f = np.array([1e16, 1.0, -1e16, 1.0], np.float32)                       # cancellation: exact sum 2
    assert rel.masked_sum(np.ones(4, np.int32), np.arange(4), f) == 2.0
    r = np.random.default_rng(5).standard_normal(1000).astype(np.float32)
    exact = rel.masked_sum(np.ones(1000, np.int32), np.arange(1000), r)
    assert abs(exact - float(np.sum(np.sort(r.astype(np.float64))))) < 1e-9
    agg = oq.aggregate(oq.AGG_SUM, dec, cand, 2, sum_values=vals)
    assert agg == {"count": 3, "sum": 110}


def test_margins_hand_worked():
    """K = 2: z_yes - z_no.  K = 5: z_k - z_{k*} for every k, with k* the
    reference decision when one is given (else the first argmax)."""
    z2 = np.array([[2.0, 0.5], [-1.0, 3.0], [0.25, 0.25]])
    assert rel.margins(z2).tolist() == [1.5, -4.0, 0.0]
    z5 = np.array([[1.0, 3.5, 3.5, -2.0, 0.25],
                   [0.0, -1.0, -2.0, -3.0, 4.0]])
    # own argmax: row 0 -> label 1 (first of the tied maxima), row 1 -> label 4
    assert rel.margins(z5).tolist() == [[-2.5, 0.0, 0.0, -5.5, -3.25],
                                        [-4.0, -5.0, -6.0, -7.0, 0.0]]
    # a reference decision that is not this row's own argmax is used as given
    assert rel.margins(z5, np.array([4, 0])).tolist() == [[0.75, 3.25, 3.25, -2.25, 0.0],
                                                          [0.0, -1.0, -2.0, -3.0, 4.0]]


def test_parity_comparison_rule_on_hand_cases():
    """The tests' margin comparison (tolerance 2e-2 * max(1, |ref|), decisions
    equal on clear rows) accepts and rejects the cases it should."""
    from helpers import compare_logits
    ref = np.array([[1.0, 3.5, 3.49, -2.0, 0.25],       # runner-up 0.01 below: not clear
                    [0.0, -1.0, -2.0, -3.0, 4.0]])      # clear
    ok = ref + np.array([[0.0, 0.0, 0.015, 0.0, 0.0],   # flips the near tie within 0.02: allowed
                         [0.01, 0.0, 0.0, 0.0, -0.05]])  # within 2e-2 * |margin| (4 -> 0.08)
    compare_logits(ok, ref)
    bad = ref + np.array([[0.0, 0.0, 0.0, 0.0, 0.0], [0.0, 0.0, 0.0, 0.0, -0.2]])
    with pytest.raises(AssertionError):
        compare_logits(bad, ref)                        # margin error 0.2 > 0.08
    ref2 = np.array([[0.3, 0.0], [0.01, 0.0]])
    compare_logits(np.array([[0.29, 0.0], [-0.005, 0.0]]), ref2)  # |0.01| <= 0.1: may flip
    with pytest.raises(AssertionError):
        compare_logits(np.array([[0.3, 0.31], [0.01, 0.0]]), ref2)  # clear row flipped
