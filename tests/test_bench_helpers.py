"""The benchmark's reporting arithmetic (CPU): the algorithmic attention FLOPs
of a select query and the per-kernel roofline classification."""
import importlib.util
import os

import numpy as np

import synth
from helpers import ROOT
from oracle import relational as rel


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_attention_flops_counts_causal_pairs_with_the_prefix():
    b = _bench()
    w = synth.C1_TINY
    q = synth.make_inputs(w)
    preds = [(p.column, p.op, p.value) for p in w.preds]
    cand = rel.compact(rel.predicate_mask(q.table.cols, preds, q.table.n_rows))
    P = w.prefix_len
    # brute force: every row token attends the P prefix keys and its own earlier tokens
    pairs = 0
    for r in cand:
        n = int(q.table.offsets[r + 1] - q.table.offsets[r])
        pairs += sum(P + j + 1 for j in range(n))
    pairs += P * (P + 1) // 2                      # the prefix pass, once per query
    s = w.model
    assert b.attention_flops_host(w, q) == 4.0 * s.n_heads * s.head_dim * s.n_layers * pairs


def test_kernel_rooflines_bounds_and_fractions():
    b = _bench()
    pk = {"hbm_gbs": 6000.0, "bf16_tflops": 2000.0, "bf16_tflops_sustained": 1500.0}
    stats = {"gemm_a": {"total_ms": 2.0, "flops": 3.0e12, "bytes": 0.0},
             "rmsnorm": {"total_ms": 1.0, "flops": 0.0, "bytes": 3.0e9},
             "attention": {"total_ms": 4.0, "flops": 0.0, "bytes": 0.0},
             "pack_chunk": {"total_ms": 0.5, "flops": 0.0, "bytes": 0.0}}
    k = b.kernel_rooflines(stats, 2, pk, attn_flops=1.2e12)
    assert k["gemm_a"]["bound"] == "tensor" and np.isclose(k["gemm_a"]["achieved"], 1500.0)
    assert np.isclose(k["gemm_a"]["frac"], 1.0)
    assert k["rmsnorm"]["bound"] == "hbm" and np.isclose(k["rmsnorm"]["frac"], 0.5)
    assert k["attention"]["bound"] == "tensor" and np.isclose(k["attention"]["achieved"], 300.0)
    assert k["pack_chunk"] == {"ms_per_step": 0.25}


def test_reference_arm_json_line_on_the_tiny_workload():
    """`bench.py --impl reference` (the oracle, on the host cores) prints one
    JSON line with the contract's keys, describing the workload it ran."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                        "c1_tiny_select", "--steps", "2", "--warmup", "1"], capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == "AI-query input rows/s" and d["unit"] == "rows/s"
    assert d["steps"] == 2 and d["warmup"] == 1 and d["higher_is_better"] is True and d["value"] > 0
    assert d["config"]["workload"] == "c1_tiny_select" and d["config"]["rows"] == synth.C1_TINY.n_rows
    assert d["config"]["model"].startswith(f"decoder d{synth.C1_TINY.model.d_model} L{synth.C1_TINY.model.n_layers} ")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_runs_the_join_workload():
    """The reference arm times the oracle's join (movies year >= 2010, reviews
    joined on movie id) on a scaled-down reviews-movies workload."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                        "c3_join_1b", "--rows", "2000", "--steps", "1", "--warmup", "1",
                        "--cpu-sample-candidates", "1"], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    d = json.loads([ln for ln in r.stdout.splitlines() if ln.startswith("{")][0])
    assert d["config"]["workload"] == "c3_join_1b_n2000" and d["value"] > 0
    assert "of the" in d["cpu_baseline"]["sample"] and d["cpu_baseline"]["cores"] >= 1


def test_stratified_sample_spans_the_length_distribution():
    b = _bench()
    lens = np.random.default_rng(3).lognormal(np.log(120), 0.5, 5000)
    pos = b.stratified_sample(lens, 16, 9)
    assert len(pos) == 16 and len(set(pos.tolist())) == 16 and np.all(np.diff(pos) > 0)
    # one pick per sixteenth of the sorted lengths
    ranks = np.argsort(np.argsort(lens, kind="stable"), kind="stable")[pos]
    assert sorted((ranks * 16) // 5000) == list(range(16))
    assert np.array_equal(pos, b.stratified_sample(lens, 16, 9))          # seeded
    assert len(b.stratified_sample(lens[:5], 16, 9)) == 5                  # fewer candidates than strata
    assert len(b.stratified_sample(lens[:0], 16, 9)) == 0


def test_blas_threads_reports_a_positive_count():
    b = _bench()
    assert b.blas_threads() >= 1
