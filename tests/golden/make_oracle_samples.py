"""Write the fp64 oracle's label logits for a seeded sample of candidates of
each full-size workload, for the full-size parity tests to compare against.

Imports only ``oracle/`` (the query's definition) and ``synth/`` (the seeded
inputs); nothing here touches the CUDA path.  Every stored number is the
oracle's: each sampled candidate's prompt (shared prefix ++ row text) is run
through the fp64 decoder on its own, and the K label logits at its last
position are written out (Fig. 2: ``logits[:, -1, :]`` at the label ids).

Each output file ``oracle_logits_<workload>.json`` is keyed by the workload's
name and seeds and by the sha256 of the oracle's and the input generator's
sources; the tests refuse a file whose key no longer matches, so a change to
either side's source calls for a re-run of this script.

Usage (a few CPU-hours for the whole set on 8 cores; resumable):
    python tests/golden/make_oracle_samples.py                 # every workload
    python tests/golden/make_oracle_samples.py --only c2_select_1b
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402
from oracle import query as oq  # noqa: E402
from oracle import relational as rel  # noqa: E402
from oracle import transformer as tf  # noqa: E402

ORACLE_FILES = ("oracle/relational.py", "oracle/transformer.py", "oracle/query.py")
SYNTH_FILES = ("synth/configs.py", "synth/generate.py")

# (workload, sampled candidates besides the shortest and the longest prompt)
PLAN = (
    ("c2_select_1b", 512),
    ("c3_join_1b", 512),
    ("c5_sweep_100%_fixed", 512),
    ("c5_sweep_25%_lognormal", 512),
    ("c4_multilabel_8b", 128),
)


def sources_sha256(files) -> str:
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(f.encode() + b"\0" + fh.read())
    return h.hexdigest()


def workload(name: str):
    if name.startswith("c5_sweep_"):
        point, kind = name[len("c5_sweep_"):].split("_")
        return synth.sweep_workload(point, kind)
    return synth.WORKLOADS[name]


def sample_positions(n_cand: int, k: int, seed: int, lens: np.ndarray) -> np.ndarray:
    """k seeded candidate positions plus the shortest and the longest prompt."""
    rng = np.random.default_rng(seed)
    pick = set(rng.choice(n_cand, size=min(k, n_cand), replace=False).tolist())
    if n_cand:
        pick |= {int(np.argmin(lens)), int(np.argmax(lens))}
    return np.array(sorted(pick), dtype=np.int64)


def candidates(w, q):
    """Candidate rows that reach the LM (and, for the join, their build rows)."""
    if w.join_build_rows:
        bp = [(p.column, p.op, p.value) for p in w.join_build_preds]
        return oq.join_candidates(q.table, q.build, "movie_id", "movie_id", [], bp)
    preds = [(p.column, p.op, p.value) for p in w.preds]
    return rel.compact(rel.predicate_mask(q.table.cols, preds, q.table.n_rows)), None


def key_of(w, k):
    return {"workload": w.name, "data_seed": w.data_seed, "weight_seed": w.weight_seed,
            "sample_seed": w.data_seed, "sample_k": k,
            "oracle_sha256": sources_sha256(ORACLE_FILES),
            "synth_sha256": sources_sha256(SYNTH_FILES)}


def run(name: str, k: int, out_dir: str, work_dir: str, chunk: int) -> str:
    w = workload(name)
    key = key_of(w, k)
    out = os.path.join(out_dir, f"oracle_logits_{name}.json")
    if os.path.exists(out):
        with open(out) as fh:
            old = json.load(fh)
        if all(old.get(a) == b for a, b in key.items()):
            print(f"{name}: up to date", flush=True)
            return out
    q = synth.make_inputs(w)
    cand, _ = candidates(w, q)
    lens = np.diff(q.table.offsets)[cand]
    pos = sample_positions(len(cand), k, key["sample_seed"], lens)
    rows = cand[pos]
    prompts = oq.prompts(q.prefix, q.table.offsets, q.table.tokens, rows)
    print(f"{name}: {len(cand)} candidates, sampling {len(pos)}; "
          f"{sum(len(p) for p in prompts)} prompt tokens", flush=True)

    os.makedirs(work_dir, exist_ok=True)
    part = os.path.join(work_dir, f"{name}.partial.json")
    done = {}
    if os.path.exists(part):
        with open(part) as fh:
            p = json.load(fh)
        if p.get("key") == key:
            done = {int(a): b for a, b in p["logits"].items()}
    t0 = time.time()
    W = synth.make_weights(w.model, w.weight_seed)
    model = tf.Model(w.model, W)
    print(f"{name}: weights ready in {time.time() - t0:.0f} s; {len(done)} rows resumed", flush=True)
    todo = [i for i in range(len(pos)) if i not in done]
    cpu_s = 0.0
    for s in range(0, len(todo), chunk):
        idx = todo[s:s + chunk]
        t1 = time.time()
        z = tf.label_logits(model, [prompts[i] for i in idx], w.label_ids)
        cpu_s += time.time() - t1
        for i, zi in zip(idx, z):
            done[i] = [float(v) for v in zi]
        with open(part + ".tmp", "w") as fh:
            json.dump({"key": key, "logits": {str(a): b for a, b in done.items()}}, fh)
        os.replace(part + ".tmp", part)
        print(f"{name}: {len(done)}/{len(pos)} rows, {time.time() - t1:.0f} s for {len(idx)}", flush=True)

    rec = dict(key)
    rec.update({
        "labels": list(w.label_ids),
        "n_candidates": int(len(cand)),
        "positions": [int(v) for v in pos],
        "row_ids": [int(v) for v in rows],
        "prompt_lens": [int(len(p)) for p in prompts],
        "logits": [done[i] for i in range(len(pos))],
        "made_with": {"python": platform.python_version(), "numpy": np.__version__,
                      "machine": platform.machine(),
                      "seconds_this_run": round(cpu_s, 1)},
    })
    with open(out + ".tmp", "w") as fh:
        json.dump(rec, fh, indent=0)
        fh.write("\n")
    os.replace(out + ".tmp", out)
    print(f"{name}: wrote {out}", flush=True)
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--only", default="", help="comma-separated workload names")
    ap.add_argument("--out-dir", default=HERE)
    ap.add_argument("--work-dir", default=os.path.join("/tmp", "aiq_oracle_samples"),
                    help="checkpoints of partly computed samples")
    ap.add_argument("--chunk", type=int, default=32, help="rows per checkpoint")
    a = ap.parse_args(argv)
    only = set(filter(None, a.only.split(",")))
    for name, k in PLAN:
        if only and name not in only:
            continue
        run(name, k, a.out_dir, a.work_dir, a.chunk)


if __name__ == "__main__":
    main()
