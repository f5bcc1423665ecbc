"""Shared test helpers: GPU availability, library handles, oracle comparisons."""
from __future__ import annotations

import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# Margin tolerance and decision rule of the parity bar: label-logit margins
# within 2e-2 * max(1, |ref|); decisions must agree wherever |ref margin| > 0.1.
MARGIN_RTOL = 2e-2
DECISION_MARGIN = 0.1


def header_symbols():
    syms = set()
    for name in os.listdir(os.path.join(ROOT, "include")):
        if name.endswith(".h"):
            src = open(os.path.join(ROOT, "include", name)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            syms |= set(re.findall(r"\b(aiq_\w+)\s*\(", src))
    return sorted(syms)


def gpu_ctx():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_10139_gb300 import aiq
    return aiq.Context(0)


def weights_list(shape, W):
    import synth
    return [W[n] for n, _, _ in synth.weight_specs(shape)]


def oracle_preds(preds):
    return [(p.column, p.op, p.value) for p in preds]


def margin_ratios(gpu_logits, ref_logits):
    """Per row, the largest |margin error| / tolerance of K-label logits (rows
    aligned), and whether the decisions agree on every clear row."""
    from oracle import relational as rel
    gpu = np.asarray(gpu_logits, np.float64)
    ref = np.asarray(ref_logits, np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    if len(ref) == 0:
        return np.zeros(0), True
    ref_dec = rel.decide(ref)
    mr = rel.margins(ref, ref_dec)
    mg = rel.margins(gpu, ref_dec)
    tol = MARGIN_RTOL * np.maximum(1.0, np.abs(mr))
    ratio = np.abs(mg - mr) / tol
    if ratio.ndim == 2:  # K > 2: every label's margin to k*
        ratio = ratio.max(axis=1)
    gdec = rel.decide(gpu)
    if ref.shape[1] == 2:
        clear = np.abs(mr) > DECISION_MARGIN
    else:
        # the runner-up margin decides: clear when every other label is > 0.1 below k*
        others = np.where(np.arange(ref.shape[1])[None, :] == ref_dec[:, None], -np.inf, mr)
        clear = others.max(axis=1) < -DECISION_MARGIN
    return ratio, bool(np.array_equal(gdec[clear], ref_dec[clear]))


def compare_logits(gpu_logits, ref_logits, what=""):
    """Margin parity of K-label logits (rows aligned)."""
    ratio, decisions_ok = margin_ratios(gpu_logits, ref_logits)
    if len(ratio) == 0:
        return 0.0
    worst = float(ratio.max())
    assert worst <= 1.0, f"{what} margin error above tolerance on {int((ratio > 1).sum())} rows (worst ratio {worst:.3f})"
    assert decisions_ok, f"{what} decision mismatch on clear rows"
    return worst


def check_greedy(model, prompts, toks, text_len, eos, pad, what=""):
    """Teacher-forced validity of GPU greedy outputs; returns (worst gap
    ratio, number of steps where the oracle's own argmax differs)."""
    worst, flips = 0.0, 0
    n_new = toks.shape[1]
    for i, p in enumerate(prompts):
        y = [int(v) for v in toks[i]]
        L = int(text_len[i])
        steps = min(L + 1, n_new)                  # decisions taken: the text, then the eos
        if L < n_new:
            assert y[L] == eos, f"{what} row {i}: text_len {L} but token {y[L]} is not the eos"
            assert all(v == pad for v in y[L + 1:]), f"{what} row {i}: no pad after the eos"
        assert eos not in y[:L], f"{what} row {i}: eos before text_len"
        seq = np.concatenate([p, np.asarray(y[:steps - 1], np.int64)])
        z = _tf().vocab_logits(model, [seq])[len(p) - 1:]
        for t in range(steps):
            zt = z[t]
            top = float(zt.max())
            gap = top - float(zt[y[t]])
            ratio = gap / (MARGIN_RTOL * max(1.0, abs(top)))
            worst = max(worst, ratio)
            flips += int(_tf().first_argmax(zt) != y[t])
            assert ratio <= 1.0, f"{what} row {i} step {t}: token {y[t]} is {gap:.4g} below the max"
    return worst, flips


def _tf():
    from oracle import transformer as tf
    return tf
