"""Benchmark of the unified AI query on GB300.

Default workload: the select AI query at scale (100,000 rows; predicate
rating >= 4 AND year >= 2000; lognormal text of median 120 tokens behind a
64-token shared prefix; random-init 1B-shape decoder: d=2048, 16 layers,
32/8 heads, head_dim 64, SwiGLU 8192, vocab 32000; yes/no decision; output the
selected row ids and their count).  One step = one whole query over the
resident table: predicate, compaction, packing, prefill, decision, aggregate.

Prints one JSON line.  `value` is input rows/s over the device-timed steps
(table and model resident in HBM); `e2e` repeats the metric through the C-ABI
with host buffers (table upload, query, result download per step).
`--impl reference` times the CPU oracle instead, on a bounded sample.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

# The CPU oracle (the reference arm and the cpu_baseline leg) runs numpy BLAS on
# every host core.  torchrun sets OMP_NUM_THREADS=1 for each rank, which would
# pin the reference arm's rank 0 to one thread: give every BLAS flavour the
# host's cores before numpy loads it.
if "reference" in sys.argv and os.environ.get("OMP_NUM_THREADS") == "1":
    for _k in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "OMP_NUM_THREADS"):
        os.environ[_k] = str(os.cpu_count() or 1)

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_BYTES = 129 * 1024 * 1024

# DRAM traffic of one tcgen05 GEMM launch from an ncu capture, valid only for the
# GEMM source it was measured on (sha256 prefix of csrc/gemm_tcgen05.cu followed
# by csrc/common.cuh, the device helpers it includes).
GEMM_TRAFFIC = {"source_sha": "e6d25c1d18b681c0", "bytes_per_launch": 3.708e9}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="c2_select_1b")
    p.add_argument("--rows", type=int, default=0, help="override the table size (testing)")
    p.add_argument("--token-budget", type=int, default=0,
                   help="prefill tokens per chunk (0: the library default); small values keep profiler captures small")
    p.add_argument("--e2e-steps", type=int, default=2)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-sample-candidates", type=int, default=16,
                   help="CPU oracle: LM candidates per step (stratified by prompt length)")
    p.add_argument("--relational-micro-rows", type=int, default=1 << 28,
                   help="rows of the predicate + compaction micro-measurement in the default line (0: skip)")
    p.add_argument("--micro", default="", choices=["", "relational", "attention"],
                   help="relational: predicate + compaction alone on a 2^28-row table, against HBM bandwidth; "
                        "attention: one prefill chunk's varlen GQA attention launch (select-query shape)")
    p.add_argument("--micro-rows", type=int, default=1 << 28)
    p.add_argument("--sweep", default="", help="selectivity sweep: 'fixed', 'lognormal' or 'both'")
    p.add_argument("--transform", type=int, default=0,
                   help="AI_TRANSFORM: greedy tokens per candidate row (0: the AI_IF query)")
    p.add_argument("--like", default="", help="AI_TRANSFORM ... LIKE pattern, comma-separated token ids")
    p.add_argument("--decode-rows", type=int, default=0, help="AI_TRANSFORM rows per decode batch (0: library default)")
    p.add_argument("--pairs", action="store_true", help="Table 2 Q4: AI_IF over the reviews self-joined on movie id")
    return p.parse_args()


def workload(args):
    w = synth.WORKLOADS[args.workload]
    if args.rows:
        w = synth.scaled(w, args.rows, join_build_rows=(max(1, args.rows // 10) if w.join_build_rows else None))
    return w


def make_step(ctx, w, q, model, aiq, world=1, rank=0):
    """One whole query on the resident tables: the select form, or the
    reviews-movies join form with GROUP BY movie.

    With world > 1 every rank holds the whole table (plus a row-id column) and
    one step is the query over one table split across the ranks: a
    relational-only pass gives the candidates, the rows are cut into
    contiguous ranges of equal candidate prompt tokens, this rank runs the
    query on its range (two more terms on the row-id column) and the small
    results are merged over the process group."""
    from paper_2608_10139_gb300 import shard
    preds = [(p.column, p.op, p.value) for p in w.preds]
    cols = q.table.cols if world == 1 else shard.with_row_ids(q.table.cols, q.table.n_rows)
    table = ctx.load_table(cols, (q.table.offsets, q.table.tokens))
    tables = [table]
    if not w.join_build_rows:
        def run(terms, flags=0):
            return ctx.run_select(table, model, terms, q.prefix, w.label_ids, agg=w.agg, flags=flags)
    else:
        build = ctx.load_table(q.build.cols, n_rows=q.build.n_rows)
        tables.append(build)
        bpreds = [(p.column, p.op, p.value) for p in w.join_build_preds]

        def run(terms, flags=0):
            return ctx.run_join_select(build, "movie_id", bpreds, table, "movie_id", model if not flags else 0,
                                       terms, q.prefix, w.label_ids, agg=w.agg, flags=flags)
    if world == 1:
        return (lambda: run(preds)), tables
    text_len = np.diff(q.table.offsets)

    def step():
        plan = run(preds, aiq.FLAG_RELATIONAL_ONLY)
        cand = plan.cand_row_ids
        lo, hi = shard.token_balanced_ranges(q.table.n_rows, cand, len(q.prefix) + text_len[cand], world)[rank]
        r = run(preds + shard.range_terms(lo, hi))
        r.merged = shard.gather_merge(shard.local_result(r, 0))
        r.n_launches += plan.n_launches
        r.shard_range = (lo, hi)
        return r
    return step, tables


def blas_threads() -> int:
    """Threads the CPU oracle's BLAS actually runs on: threadpoolctl's report
    where it is installed, else OpenBLAS's own answer through the library
    numpy has loaded, else the environment's setting."""
    try:
        from threadpoolctl import threadpool_info
        n = [int(p["num_threads"]) for p in threadpool_info() if p.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    try:
        import ctypes
        libs = set()
        with open("/proc/self/maps") as fh:
            for line in fh:
                path = line.split()[-1] if "/" in line else ""
                if "openblas" in os.path.basename(path).lower():
                    libs.add(path)
        for path in sorted(libs):
            lib = ctypes.CDLL(path)
            for sym in ("scipy_openblas_get_num_threads64_", "openblas_get_num_threads64_",
                        "openblas_get_num_threads"):
                f = getattr(lib, sym, None)
                if f is not None:
                    f.restype = ctypes.c_int
                    n = int(f())
                    if n > 0:
                        return n
    except Exception:
        pass
    for k in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "OMP_NUM_THREADS"):
        v = os.environ.get(k, "")
        if v.isdigit() and int(v) > 0:
            return int(v)
    return os.cpu_count() or 1


def model_desc(m) -> str:
    return (f"decoder d{m.d_model} L{m.n_layers} {m.n_heads}/{m.n_kv_heads} heads hd{m.head_dim} "
            f"ffn{m.d_ffn} V{m.vocab}, random init")


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return d, "measured"
    return PEAKS_FALLBACK, "fallback"


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


def gemm_source_sha():
    h = hashlib.sha256()
    for name in ("gemm_tcgen05.cu", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2608_10139_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


# ------------------------------------------------------------ CPU oracle ---

def oracle_candidates(w, q):
    """The oracle's relational phase on the whole table (the join for the
    reviews-movies workload): candidate rows that reach the LM, ascending."""
    from oracle import query as oq
    from oracle import relational as rel
    if w.join_build_rows:
        bp = [(p.column, p.op, p.value) for p in w.join_build_preds]
        pp = [(p.column, p.op, p.value) for p in w.preds]
        return oq.join_candidates(q.table, q.build, "movie_id", "movie_id", pp, bp)[0]
    preds = [(p.column, p.op, p.value) for p in w.preds]
    return rel.compact(rel.predicate_mask(q.table.cols, preds, q.table.n_rows))


def stratified_sample(lens: np.ndarray, m: int, seed: int) -> np.ndarray:
    """m candidate positions, one from each of m equal-count strata of the
    candidates sorted by prompt length (seeded pick inside each stratum), so
    that every sample spans the length distribution."""
    n = len(lens)
    if n == 0:
        return np.zeros(0, np.int64)
    m = min(m, n)
    order = np.argsort(lens, kind="stable")
    edges = np.linspace(0, n, m + 1).astype(np.int64)
    rng = np.random.default_rng(seed)
    pick = [order[rng.integers(edges[i], edges[i + 1])] for i in range(m) if edges[i + 1] > edges[i]]
    return np.sort(np.array(pick, dtype=np.int64))


def cpu_oracle_step(w, q, model, m: int, seed: int):
    """One bounded step of the CPU oracle as it stands: its relational phase
    on the whole table, then its fp64 transformer on m stratified candidates.
    The query's time is extrapolated from the sample by prompt tokens (the
    transformer's cost is linear in them up to the small attention term).
    Returns (step seconds, extrapolated query seconds, candidates, sample size)."""
    from oracle import query as oq
    from oracle import relational as rel
    from oracle import transformer as tf
    t0 = time.perf_counter()
    cand = oracle_candidates(w, q)
    t_rel = time.perf_counter() - t0
    lens = (np.diff(q.table.offsets)[cand] + len(q.prefix)).astype(np.float64)
    pos = stratified_sample(lens, m, seed)
    t1 = time.perf_counter()
    if len(pos):
        z = tf.label_logits(model, oq.prompts(q.prefix, q.table.offsets, q.table.tokens, cand[pos]), w.label_ids)
        rel.decide(z)
    t_lm = time.perf_counter() - t1
    scale = float(lens.sum() / lens[pos].sum()) if len(pos) else 0.0
    return t_rel + t_lm, t_rel + t_lm * scale, len(cand), len(pos)


def attention_flops_host(w, q) -> float:
    """Algorithmic FLOPs of the prefill attention of one select query:
    4 Hq hd per causal (query, key) pair per layer, every row attending the
    shared prefix and its own earlier tokens, plus the prefix pass itself.
    (Host arithmetic for the report only; 0 for the join workloads.)"""
    if w.join_build_rows:
        return 0.0
    mask = np.ones(w.n_rows, dtype=bool)
    ops = {0: np.less, 1: np.less_equal, 2: np.greater, 3: np.greater_equal, 4: np.equal, 5: np.not_equal}
    for p in w.preds:
        mask &= ops[p.op](q.table.cols[p.column].astype(np.int64), p.value)
    lens = np.diff(q.table.offsets)[mask].astype(np.float64)
    P = float(w.prefix_len)
    pairs = float(np.sum(lens * P + lens * (lens + 1) / 2)) + (P * (P + 1) / 2 if mask.any() else 0.0)
    s = w.model
    return 4.0 * s.n_heads * s.head_dim * s.n_layers * pairs


def kernel_rooflines(stats, steps, pk, attn_flops) -> dict:
    """Per kernel class: device ms per step and the achieved rate against its
    bound (tensor: TFLOP/s vs the sustained dense peak; HBM: GB/s vs the copy peak)."""
    out = {}
    tens = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    for name, v in sorted(stats.items()):
        ms = v["total_ms"]
        if ms <= 0:
            continue
        e = {"ms_per_step": round(ms / steps, 3)}
        flops = v["flops"] if v["flops"] else (attn_flops if name == "attention" else 0.0)
        if flops:
            a = flops / (ms / 1000.0) / 1e12
            e.update(bound="tensor", achieved=round(a, 1), unit="TFLOP/s", frac=round(a / tens, 3))
        elif v["bytes"]:
            a = v["bytes"] / (ms / 1000.0) / 1e9
            e.update(bound="hbm", achieved=round(a, 1), unit="GB/s", frac=round(a / pk["hbm_gbs"], 3))
        out[name] = e
    return out


def reference_arm(args):
    """The CPU oracle as it stands, timed on this host's cores (rank 0 only):
    each step runs the relational phase on the whole table and the fp64
    transformer on a stratified sample of candidates (a different seeded
    sample per step), and the query's rows/s is extrapolated from it."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from oracle import transformer as tf
    w = workload(args)
    q = synth.make_inputs(w)
    model = tf.Model(w.model, synth.make_weights(w.model, w.weight_seed))
    m = args.cpu_sample_candidates
    for i in range(args.warmup):            # warm-up steps: one candidate each
        cpu_oracle_step(w, q, model, 1, w.data_seed + 100 + i)
    steps, extrap, n_cand, n_sampled = [], [], 0, 0
    for k in range(args.steps):
        s, e, n_cand, ns = cpu_oracle_step(w, q, model, m, w.data_seed + k)
        steps.append(s)
        extrap.append(e)
        n_sampled += ns
    value = w.n_rows / statistics.mean(extrap)
    threads = blas_threads()
    sample = (f"per step: relational phase on all {w.n_rows} rows, fp64 transformer on {m} of the {n_cand} "
              f"LM candidates (one per prompt-length stratum, new seed each step; {n_sampled} in all), "
              f"query time extrapolated by prompt tokens")
    line = {"impl": "reference", "metric": "AI-query input rows/s", "value": value, "unit": "rows/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000 * statistics.mean(steps), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "rows": w.n_rows, "model": model_desc(w.model),
                       "sample_candidates_per_step": m},
            "extrapolated_query_s": statistics.mean(extrap),
            "cpu_baseline": {"value": value, "unit": "rows/s", "cores": threads, "host_cores": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------- GPU arm ---

def ours(args):
    import torch
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    # one process compiles (an up-to-date library is left alone); the others wait for it
    if local == 0:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    w = workload(args)
    q = synth.make_inputs(w)      # every rank: the same table (one query split over the ranks)
    W = synth.make_weights(w.model, w.weight_seed)
    tensors = [W[n] for n, _, _ in synth.weight_specs(w.model)]
    preds = [(p.column, p.op, p.value) for p in w.preds]
    ctx = aiq.Context(local)
    if args.token_budget:
        ctx.set_option("token_budget", args.token_budget)
    model = ctx.load_model(w.model, tensors)
    step, tables = make_step(ctx, w, q, model, aiq, world, rank)
    stream = torch.cuda.ExternalStream(ctx.stream())
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    for _ in range(args.warmup):
        step()
    clocks = ClockSampler(local)
    ctx.reset_kernel_stats()
    ctx.set_option("profile", 1)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    ms, launches, res = [], 0, None
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    t_wall = time.perf_counter()
    for k in range(args.steps):
        flush.add_(1.0)                    # write 2x L2 between steps
        torch.cuda.synchronize()
        ev[k][0].record(stream)
        res = step()
        ev[k][1].record(stream)
        launches += res.n_launches
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_wall
    barrier()
    clk = clocks.stop()
    ctx.set_option("profile", 0)
    ms = [a.elapsed_time(b) for a, b in ev]
    stats = ctx.kernel_stats()
    total_ms = sum(ms)
    if world > 1:
        t = torch.tensor([total_ms], device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_per_step = total_ms / args.steps
    value = w.n_rows / (ms_per_step / 1000.0)     # one table's rows over the slowest rank's time

    # dominant kernel: the tcgen05 GEMM (all four epilogue variants, one kernel template)
    g = [v for k, v in stats.items() if k.startswith("gemm_")]
    gemm_ms = sum(v["total_ms"] for v in g)
    gemm_launches = sum(v["launches"] for v in g)
    gemm_flops = sum(v["flops"] for v in g)
    pk, src = peaks()
    peak = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    achieved = gemm_flops / (gemm_ms / 1000.0) / 1e12 if gemm_ms else 0.0
    traffic = GEMM_TRAFFIC["bytes_per_launch"] if GEMM_TRAFFIC["source_sha"] == gemm_source_sha() else None
    step_ms = {k: round(v["total_ms"] / args.steps, 3) for k, v in sorted(stats.items())}
    kernels = kernel_rooflines(stats, args.steps, pk, attention_flops_host(w, q) * args.steps)

    # end to end through the C-ABI with host buffers: upload table(s), query, download results
    e2e_ms, h2d, d2h = [], q.table.nbytes() + (q.build.nbytes() if q.build else 0), 0
    for t in tables:
        ctx.free_table(t)
    for _ in range(args.e2e_steps):
        barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        step_e, tabs = make_step(ctx, w, q, model, aiq, world, rank)
        r = step_e()
        for t in tabs:
            ctx.free_table(t)
        torch.cuda.synchronize()
        e2e_ms.append(1000 * (time.perf_counter() - t0))
        d2h = (4 * len(r.row_ids) + 8 * len(r.label_counts) + 8 + 20 * len(r.group_keys))
    e2e_per = statistics.median(e2e_ms) if e2e_ms else float("nan")
    if world > 1:
        t = torch.tensor([e2e_per], device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        e2e_per = float(t.item())

    micro = None
    if rank == 0 and world == 1 and args.relational_micro_rows > 0:
        micro = relational_micro(ctx, aiq, args.relational_micro_rows, 5, 2)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import transformer as tf
        m = args.cpu_sample_candidates
        s, e, n_cand, ns = cpu_oracle_step(w, q, tf.Model(w.model, W), m, w.data_seed)
        cpu = {"value": w.n_rows / e, "unit": "rows/s", "cores": blas_threads(), "host_cores": os.cpu_count(),
               "kind": "oracle", "seconds": round(s, 1),
               "sample": f"relational phase on all {w.n_rows} rows, fp64 transformer on {ns} of the {n_cand} "
                         f"LM candidates (one per prompt-length stratum, seed {w.data_seed}); query time "
                         f"extrapolated by prompt tokens"}

    if rank == 0:
        line = {
            "metric": "AI-query input rows/s", "value": value, "unit": "rows/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "strong", "vs_baseline": None,
            "dtype": "f16xf16->f32 (bf16 model values)", "data": "synthetic",
            "config": {"workload": w.name, "rows": w.n_rows, "candidates": res.n_candidates,
                       "tokens": res.n_tokens, "prefill_tokens": res.n_prefill_tokens, "chunks": res.n_chunks,
                       "model": model_desc(w.model),
                       "l2": "2x L2 written between timed steps; weights and activations exceed L2",
                       "parallelism": ("one GPU" if world == 1 else
                                       f"one table over {world} ranks: row ranges of equal candidate prompt "
                                       f"tokens, results merged over the process group")},
            "p50_latency_ms": statistics.median(ms),
            "wall_ms_per_step": 1000 * wall / args.steps,
            "prefill_tflops": res.prefill_flops / (res.ms_prefill / 1000.0) / 1e12 if res.ms_prefill else None,
            "prompt_tokens_per_s": res.n_tokens / (res.ms_prefill / 1000.0) if res.ms_prefill else None,
            "phase_ms": {"relational": res.ms_relational, "prefill": res.ms_prefill,
                         "aggregate": res.ms_aggregate},
            "kernel_ms_per_step": step_ms,
            "kernels": kernels,
            "roofline": {"kernel": "gemm_tcgen05 (QKV+RoPE, O+residual, gate/up+SwiGLU, down+residual)",
                         "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                         "frac": achieved / peak if peak else None, "traffic": traffic,
                         "peak_source": f"{src} bf16_tflops_sustained (fp16 dense rate = bf16)",
                         "launches": gemm_launches},
            "cpu_baseline": cpu,
            "relational_micro": micro,
            "e2e": ({"value": w.n_rows / (e2e_per / 1000.0), "unit": "rows/s",
                     "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_per}
                    if e2e_ms else None),
            "gpu_launches": launches,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    ctx.close()
    if world > 1:
        torch.distributed.destroy_process_group()


def relational_micro(ctx, aiq, n: int, steps: int, warmup: int) -> dict:
    """Predicate (rating >= 4 AND year >= 2000) + order-preserving compaction
    over an n-row table of two int32 columns (rating uniform 1..5, year
    uniform 1950..2024), each kernel timed with CUDA events on the library's
    stream, against the measured HBM copy bandwidth.  The table is far larger
    than L2, so every step reads it from HBM."""
    rng = np.random.Generator(np.random.PCG64(7))
    cols = {"rating": rng.integers(1, 6, n, dtype=np.int32), "year": rng.integers(1950, 2025, n, dtype=np.int32)}
    preds = [("rating", aiq.GE, 4), ("year", aiq.GE, 2000)]
    t = ctx.load_table(cols, n_rows=n)
    del cols
    for _ in range(warmup):
        ctx.run_select(t, 0, preds, [], [0, 1], flags=aiq.FLAG_RELATIONAL_ONLY)
    ctx.reset_kernel_stats()
    ctx.set_option("profile", 1)
    totals = []
    for _ in range(steps):
        r = ctx.run_select(t, 0, preds, [], [0, 1], flags=aiq.FLAG_RELATIONAL_ONLY)
        totals.append(r.ms_relational)
    ctx.set_option("profile", 0)
    st = ctx.kernel_stats()
    ctx.free_table(t)
    S = r.n_candidates
    pk, src = peaks()
    mask_ms = st["predicate_mask"]["total_ms"] / steps
    comp_ms = st["compact"]["total_ms"] / steps
    mask_bytes = 8.0 * n + n / 8          # two int32 columns read, 1 bit/row written
    comp_bytes = n / 8 + 4.0 * S          # bitmask read, survivor ids written
    return {"rows": n, "survivors": S, "steps": steps, "warmup": warmup,
            "predicate_mask": {"ms": mask_ms, "GB/s": mask_bytes / mask_ms / 1e6,
                               "frac": mask_bytes / mask_ms / 1e6 / pk["hbm_gbs"]},
            "compact": {"ms": comp_ms, "GB/s": comp_bytes / comp_ms / 1e6,
                        "frac": comp_bytes / comp_ms / 1e6 / pk["hbm_gbs"]},
            "combined": {"ms": mask_ms + comp_ms, "GB/s": (mask_bytes + comp_bytes) / (mask_ms + comp_ms) / 1e6,
                         "frac": (mask_bytes + comp_bytes) / (mask_ms + comp_ms) / 1e6 / pk["hbm_gbs"]},
            "query_relational_ms_p50": statistics.median(totals),
            "peak": {"hbm_gbs": pk["hbm_gbs"], "source": f"{src} hbm_gbs"}}


def micro_relational(args):
    """`--micro relational`: the relational micro-measurement alone, one JSON line."""
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build
    _build.build()
    ctx = aiq.Context(0)
    clocks = ClockSampler(0)
    clocks.start()
    d = relational_micro(ctx, aiq, args.micro_rows, args.steps, args.warmup)
    d = {"metric": "relational predicate + compaction HBM throughput", **d, "clocks": clocks.stop()}
    print(json.dumps(d), flush=True)
    ctx.close()


def attention_micro(args):
    """`--micro attention`: one launch of the library's varlen GQA attention
    (aiq_op_attention) on a chunk of the select workload's shape: 970 rows of
    lognormal length (median 120, sigma 0.5, clipped 16..512; 125,560 tokens),
    each behind the same 64-token prefix, 32 query / 8 key-value heads of
    head_dim 64, fp16 q/k/v of N(0, 0.25).  CUDA events around each launch on
    the library's stream; median of `steps` launches after `warmup`.  FLOPs:
    4 * Hq * hd per causal (query, key) pair, prefix keys included."""
    import torch
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build
    _build.build()
    rng = np.random.default_rng(7)
    lens = np.clip(np.round(np.exp(rng.normal(np.log(120.0), 0.5, 970))), 16, 512).astype(np.int64)
    T = int(lens.sum())
    ss = np.zeros(len(lens) + 1, np.int32)
    np.cumsum(lens, out=ss[1:])
    Hq, Hkv, hd, P = 32, 8, 64, 64
    ctx = aiq.Context(0)
    qkv = (torch.randn(T, (Hq + 2 * Hkv) * hd, device="cuda") * 0.5).half()
    pkv = (torch.randn(P, 2 * Hkv * hd, device="cuda") * 0.5).half()
    out = torch.empty(T, Hq * hd, device="cuda", dtype=torch.half)
    sst = torch.as_tensor(ss).cuda()
    torch.cuda.synchronize()
    stream = torch.cuda.ExternalStream(ctx.stream())

    def run():
        ctx.op_attention(qkv.data_ptr(), T, sst.data_ptr(), len(lens), Hq, Hkv, hd, out.data_ptr(), pkv.data_ptr(), P)

    for _ in range(max(args.warmup, 1)):
        run()
    clocks = ClockSampler(0)
    clocks.start()
    ms = []
    for _ in range(max(args.steps, 1)):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        run()
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    clk = clocks.stop()
    med = statistics.median(ms)
    pairs = float((lens * P + lens * (lens + 1) // 2).sum())
    flops = 4.0 * Hq * hd * pairs
    pk, src = peaks()
    print(json.dumps({"metric": "attention launch time", "tokens": T, "rows": len(lens), "prefix": P,
                      "heads": [Hq, Hkv], "head_dim": hd, "us_median": med * 1e3, "us_min": min(ms) * 1e3,
                      "TFLOP/s": flops / (med * 1e-3) / 1e12,
                      "frac": flops / (med * 1e-3) / 1e12 / pk["bf16_tflops"],
                      "peak": {"bf16_tflops": pk["bf16_tflops"], "source": f"{src} bf16_tflops"},
                      "steps": len(ms), "clocks": clk}), flush=True)
    ctx.close()


def sweep(args):
    """Selectivity sweep on the 1M-row table: rows/s, p50 latency and the
    relational / prefill time split at each point (one JSON line per point)."""
    import torch
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build
    _build.build()
    kinds = ["fixed", "lognormal"] if args.sweep == "both" else [args.sweep]
    base = synth.sweep_workload("1%", kinds[0])
    W = synth.make_weights(base.model, base.weight_seed)
    ctx = aiq.Context(0)
    model = ctx.load_model(base.model, [W[n] for n, _, _ in synth.weight_specs(base.model)])
    for kind in kinds:
        q = synth.make_inputs(synth.sweep_workload("1%", kind))   # one table per text kind
        table = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
        for i, point in enumerate(synth.SWEEP_POINTS):
            w = synth.sweep_workload(point, kind)
            preds = [(p.column, p.op, p.value) for p in w.preds]
            runs = args.steps if point in ("1%", "5%", "25%") else max(1, min(args.steps, 3))
            if i == 0:   # one warm-up per table: workspaces grow to the token budget here
                ctx.run_select(table, model, preds, q.prefix, w.label_ids, agg=w.agg)
            res = [ctx.run_select(table, model, preds, q.prefix, w.label_ids, agg=w.agg) for _ in range(runs)]
            tot = [r.ms_total for r in res]
            r = res[-1]
            line = {"metric": "AI-query input rows/s", "workload": w.name, "point": point, "text": kind,
                    "rows": w.n_rows, "candidates": r.n_candidates, "prefill_tokens": r.n_prefill_tokens,
                    "runs": runs, "p50_latency_ms": statistics.median(tot),
                    "rows_per_s": w.n_rows / (statistics.median(tot) / 1000.0),
                    "relational_ms": statistics.median([x.ms_relational for x in res]),
                    "prefill_ms": statistics.median([x.ms_prefill for x in res]),
                    "aggregate_ms": statistics.median([x.ms_aggregate for x in res]),
                    "prefill_tflops": r.prefill_flops / (r.ms_prefill / 1000.0) / 1e12 if r.ms_prefill else None,
                    "count": r.count}
            print(json.dumps(line), flush=True)
        ctx.free_table(table)
    ctx.close()


def transform_bench(args):
    """AI_TRANSFORM over the workload's candidate rows (Table 2 Q3; Q5 with
    --like): greedy decoding of --transform tokens per row after the chunked
    prefill, everything on the device.  One JSON line with generated tokens/s
    and the decode kernels' rooflines; not the headline metric."""
    import torch
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build
    _build.build()
    w = workload(args)
    q = synth.make_inputs(w)
    W = synth.make_weights(w.model, w.weight_seed)
    ctx = aiq.Context(0)
    model = ctx.load_model(w.model, [W[n] for n, _, _ in synth.weight_specs(w.model)])
    table = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
    preds = [(p.column, p.op, p.value) for p in w.preds]
    like = [int(x) for x in args.like.split(",")] if args.like else None
    if args.decode_rows:
        ctx.set_option("decode_rows", args.decode_rows)
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")

    def run():
        return ctx.run_transform(table, model, preds, q.prefix, args.transform, like=like)

    for _ in range(args.warmup):
        run()
    clocks = ClockSampler(0)
    ctx.reset_kernel_stats()
    ctx.set_option("profile", 1)
    clocks.start()
    res = []
    for _ in range(args.steps):
        flush.add_(1.0)
        torch.cuda.synchronize()
        res.append(run())
    clk = clocks.stop()
    ctx.set_option("profile", 0)
    stats = ctx.kernel_stats()
    r = res[-1]
    ms = statistics.median([x.ms_total for x in res])
    dec_ms = statistics.median([x.ms_decode for x in res])
    gen_tokens = r.n_candidates * args.transform
    pk, src = peaks()
    att = stats.get("decode_attention", {"total_ms": 0, "bytes": 0, "launches": 0})
    att_gbs = att["bytes"] / (att["total_ms"] / 1000.0) / 1e9 if att["total_ms"] else None
    dg = [v for k, v in stats.items() if k.startswith("dec_gemm_") or k == "gemm_lm_argmax"]
    dg_ms = sum(v["total_ms"] for v in dg)
    dg_tf = sum(v["flops"] for v in dg) / (dg_ms / 1000.0) / 1e12 if dg_ms else None
    line = {"metric": "AI_TRANSFORM generated tokens/s", "value": gen_tokens / (ms / 1000.0), "unit": "tokens/s",
            "higher_is_better": True, "steps": args.steps, "warmup": args.warmup, "dtype": "f16xf16->f32",
            "data": "synthetic",
            "config": {"workload": w.name, "rows": w.n_rows, "candidates": r.n_candidates,
                       "max_new_tokens": args.transform, "like": like, "chunks": r.n_chunks,
                       "decode_rows": args.decode_rows or 4096},
            "input_rows_per_s": w.n_rows / (ms / 1000.0), "p50_latency_ms": ms, "decode_ms_p50": dec_ms,
            "prefill_ms_p50": statistics.median([x.ms_prefill - x.ms_decode for x in res]),
            "decode_tflops": r.decode_flops / (dec_ms / 1000.0) / 1e12 if dec_ms else None,
            "like_count": r.count,
            "kernel_ms_per_step": {k: round(v["total_ms"] / args.steps, 3) for k, v in sorted(stats.items())},
            "roofline": {
                "decode_attention": {"bound": "hbm", "achieved": att_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                                     "frac": att_gbs / pk["hbm_gbs"] if att_gbs else None,
                                     "launches": att["launches"], "peak_source": f"{src} hbm_gbs"},
                "decode_gemms": {"bound": "tensor", "achieved": dg_tf,
                                 "peak": pk.get("bf16_tflops_sustained", pk["bf16_tflops"]), "unit": "TFLOP/s",
                                 "frac": dg_tf / pk.get("bf16_tflops_sustained", pk["bf16_tflops"]) if dg_tf else None,
                                 "peak_source": f"{src} bf16_tflops_sustained"}},
            "clocks": clk}
    print(json.dumps(line), flush=True)
    ctx.free_table(table)
    ctx.close()


def pairs_bench(args):
    """Table 2 Q4 on the q4_pairs_1b workload: the self-join's pairs formed on
    the device, AI_IF on each pair's prompt.  One JSON line (pairs/s, the
    prefill GEMM roofline, and the host->device bytes against the bytes the
    pair prompts would take if they were formed on the host)."""
    import torch
    from paper_2608_10139_gb300 import aiq
    from paper_2608_10139_gb300 import build as _build
    _build.build()
    w = synth.Q4_PAIRS
    q = synth.make_pair_inputs(w)
    W = synth.make_weights(w.model, w.weight_seed)
    ctx = aiq.Context(0)
    model = ctx.load_model(w.model, [W[n] for n, _, _ in synth.weight_specs(w.model)])
    table = ctx.load_table(q.table.cols, (q.table.offsets, q.table.tokens))
    preds = [("score", 0, w.score_below)]   # LT
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")

    def run():
        return ctx.run_pair_select(table, "movie_id", model, preds, q.prefix, w.label_ids, agg=aiq.AGG_ROW_IDS)

    for _ in range(args.warmup):
        run()
    clocks = ClockSampler(0)
    ctx.reset_kernel_stats()
    ctx.set_option("profile", 1)
    clocks.start()
    res = []
    for _ in range(args.steps):
        flush.add_(1.0)
        torch.cuda.synchronize()
        res.append(run())
    clk = clocks.stop()
    ctx.set_option("profile", 0)
    stats = ctx.kernel_stats()
    r = res[-1]
    ms = statistics.median([x.ms_total for x in res])
    g = [v for k, v in stats.items() if k.startswith("gemm_")]
    g_ms = sum(v["total_ms"] for v in g)
    g_tf = sum(v["flops"] for v in g) / (g_ms / 1000.0) / 1e12 if g_ms else None
    pk, src = peaks()
    peak = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    line = {"metric": "Q4 pairs/s", "value": r.n_candidates / (ms / 1000.0), "unit": "pairs/s",
            "higher_is_better": True, "steps": args.steps, "warmup": args.warmup, "dtype": "f16xf16->f32",
            "data": "synthetic",
            "config": {"workload": w.name, "rows": w.n_rows, "movies": w.n_movies, "pairs": r.n_candidates,
                       "yes_pairs": r.count},
            "input_rows_per_s": w.n_rows / (ms / 1000.0), "p50_latency_ms": ms,
            "relational_ms_p50": statistics.median([x.ms_relational for x in res]),
            "prefill_tflops": r.prefill_flops / (r.ms_prefill / 1000.0) / 1e12 if r.ms_prefill else None,
            "h2d_table_bytes": int(q.table.nbytes()),
            "host_pair_prompt_bytes": int(4 * r.n_tokens),
            "kernel_ms_per_step": {k: round(v["total_ms"] / args.steps, 3) for k, v in sorted(stats.items())},
            "roofline": {"kernel": "gemm_tcgen05", "bound": "tensor", "achieved": g_tf, "peak": peak,
                         "unit": "TFLOP/s", "frac": g_tf / peak if g_tf else None,
                         "peak_source": f"{src} bf16_tflops_sustained"},
            "clocks": clk}
    print(json.dumps(line), flush=True)
    ctx.free_table(table)
    ctx.close()


def main():
    args = parse()
    if args.impl == "reference":
        reference_arm(args)
    elif args.micro == "relational":
        micro_relational(args)
    elif args.micro == "attention":
        attention_micro(args)
    elif args.sweep:
        sweep(args)
    elif args.transform:
        transform_bench(args)
    elif args.pairs:
        pairs_bench(args)
    else:
        ours(args)


if __name__ == "__main__":
    main()
