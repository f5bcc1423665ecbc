"""CPU emulation of where the GPU path rounds to fp16, for the precision
analysis of the multi-label (8B-shape) workload.  Test infrastructure: it runs
the oracle's decoder in float64 and rounds chosen intermediate values to fp16
exactly where the GPU's kernels store them, then compares the label-logit
margins with the stored fp64 oracle sample (tests/golden/oracle_logits_*.json).

Rounding points (each can be switched on alone or together):
  resg    the QKV GEMM's input, fp16(residual * attention-norm gain)
  qkv     q, k (after the rotary embedding) and v
  p       the attention probabilities
  attn    the attention output (the O projection's input)
  mlpn    the MLP-side RMSNorm output (the gate/up GEMM's input)
  swiglu  the SwiGLU output (the down projection's input)

On the 8B shape the library writes the two MLP activations as two fp16 terms
by default, so "mlpn" and "swiglu" there stand for the one-term mode
(mlp_split 0).  With no point on, the script reproduces the stored oracle
logits exactly, which checks the reordering of the norm (gain before the GEMM,
1/rms after it) against the oracle's.

Usage (about 20 s per layer per variant and row on 8 cores for the 8B shape):
    python tests/precision_emulation.py --rows 10,40,70,100 --variants all,qkv,mlpn
A variant is "all", "none" or a '+'-joined set of points ("mlpn+swiglu")."""
from __future__ import annotations

import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402
from oracle import query as oq  # noqa: E402
from oracle import relational as rel  # noqa: E402
from oracle import transformer as tf  # noqa: E402

POINTS = ("resg", "qkv", "p", "attn", "mlpn", "swiglu")


def f16(a: np.ndarray) -> np.ndarray:
    return a.astype(np.float16).astype(np.float64)


def attention(q, k, v, round_p):
    """Causal GQA attention; with round_p the probabilities enter P V as fp16
    (the row sums stay unrounded, as on the GPU)."""
    t, hq, hd = q.shape
    group = hq // k.shape[1]
    out = np.empty_like(q)
    future = np.triu(np.ones((t, t), dtype=bool), 1)
    for h in range(hq):
        kv = h // group
        s = (q[:, h, :] @ k[:, kv, :].T) / np.sqrt(hd)
        s[future] = -np.inf
        p = np.exp(s - s.max(axis=1, keepdims=True))
        l = p.sum(axis=1, keepdims=True)
        out[:, h, :] = ((f16(p) if round_p else p) @ v[:, kv, :]) / l
    return out


def layer(x, s, lw, on):
    t = x.shape[0]
    pos = np.arange(t)
    g = lw["attn_norm"]
    inv = 1.0 / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + s.rms_eps)
    xg = x * g[None, :]
    W = np.concatenate([lw["wq"], lw["wk"], lw["wv"]])
    qkv = ((f16(xg) if "resg" in on else xg) @ W.T) * inv
    kd = s.n_kv_heads * s.head_dim
    q = tf.rope(qkv[:, :s.q_dim].reshape(t, s.n_heads, s.head_dim), pos, s.rope_theta)
    k = tf.rope(qkv[:, s.q_dim:s.q_dim + kd].reshape(t, s.n_kv_heads, s.head_dim), pos, s.rope_theta)
    v = qkv[:, s.q_dim + kd:].reshape(t, s.n_kv_heads, s.head_dim)
    if "qkv" in on:
        q, k, v = f16(q), f16(k), f16(v)
    a = attention(q, k, v, "p" in on).reshape(t, s.q_dim)
    if "attn" in on:
        a = f16(a)
    x = x + a @ lw["wo"].T
    h = tf.rmsnorm(x, lw["mlp_norm"], s.rms_eps)
    if "mlpn" in on:
        h = f16(h)
    y = tf.silu(h @ lw["wg"].T) * (h @ lw["wu"].T)
    if "swiglu" in on:
        y = f16(y)
    return x + y @ lw["wd"].T


def parse_variant(v: str):
    if v == "all":
        return set(POINTS)
    if v == "none":
        return set()
    pts = set(v.split("+"))
    bad = pts - set(POINTS)
    if bad:
        raise SystemExit(f"unknown rounding point(s): {sorted(bad)}")
    return pts


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="c4_multilabel_8b")
    ap.add_argument("--rows", default="10,40,70,100", help="positions in the stored sample")
    ap.add_argument("--variants", default="all,qkv,mlpn,swiglu,attn")
    a = ap.parse_args(argv)
    w = synth.WORKLOADS[a.workload]
    path = os.path.join(ROOT, "tests", "golden", f"oracle_logits_{a.workload}.json")
    d = json.load(open(path))
    idx = [int(i) for i in a.rows.split(",")]
    variants = [(v, parse_variant(v)) for v in a.variants.split(",")]
    q = synth.make_inputs(w)
    model = tf.Model(w.model, synth.make_weights(w.model, w.weight_seed))
    s = w.model
    seqs = oq.prompts(q.prefix, q.table.offsets, q.table.tokens, [d["row_ids"][i] for i in idx])
    xs = {name: [model.embed_rows(np.asarray(sq, np.int64)) for sq in seqs] for name, _ in variants}
    for l in range(s.n_layers):
        lw = {n: model.get(f"l{l}.{n}") for n in tf.LAYER_TENSORS}
        for name, on in variants:
            xs[name] = [layer(x, s, lw, on) for x in xs[name]]
        print(f"layer {l + 1}/{s.n_layers}", flush=True)
    gfin = model.get("final_norm")
    wl, bl = model.label_head(w.label_ids)
    ref = np.asarray(d["logits"], np.float64)[idx]
    mr = rel.margins(ref, rel.decide(ref))
    tol = 2e-2 * np.maximum(1.0, np.abs(mr))
    for name, _ in variants:
        z = np.array([wl @ tf.rmsnorm(x[-1], gfin, s.rms_eps) + bl for x in xs[name]])
        ratio = np.abs(rel.margins(z, rel.decide(ref)) - mr) / tol
        ratio = ratio.max(axis=1) if ratio.ndim == 2 else ratio
        print(f"{name:>24}: margin error / tolerance per row {np.round(ratio, 3).tolist()}, "
              f"largest logit error per row {np.round(np.abs(z - ref).max(axis=1), 4).tolist()}", flush=True)


if __name__ == "__main__":
    main()
