"""Oracle, neural half: fp64 forward of a decoder-only causal LM, one row at a time.

TEST INFRASTRUCTURE ONLY: imported by tests, the smoke check and the
benchmark's CPU-baseline leg, never by the product path.  Shares no code
with the CUDA path.

The paper runs a causal-LM forward pass over each selected row and reads the
label-token logits at the row's last position (Table 1, AI_IF row; Fig. 2).
It names Gemma-2B but fixes no architecture, so the decoder follows the
common Llama-style reading:
  * pre-norm residual blocks, RMSNorm(x) = x / sqrt(mean(x^2) + eps) * g;
  * rotary embeddings on q and k, half-split pairs (i, i + hd/2),
    inv_freq_i = theta^(-2i/hd), positions restarting at 0 for every row;
  * causal grouped-query attention, scale 1/sqrt(hd), query head h reads
    key/value head h // (H_q / H_kv);
  * SwiGLU MLP W_d(silu(W_g x) * W_u x); no biases except the LM-head bias;
  * untied LM head; AI_IF needs only its label rows (Fig. 2 slices the last
    position's logits at the label ids), AI_TRANSFORM (Table 1) its full
    vocabulary for greedy decoding.
Weights arrive as bf16 bit patterns and are upcast exactly; all arithmetic is
float64.  Each row is run alone: no packing, no padding.
"""
from __future__ import annotations

from typing import Dict, List, Sequence

import numpy as np


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact upcast of bfloat16 bit patterns (uint16) to float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope(x: np.ndarray, positions: np.ndarray, theta: float) -> np.ndarray:
    """Rotate each (i, i + hd/2) pair of every head by angle pos * inv_freq_i.
    x: [T, H, hd]."""
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-(2.0 * np.arange(half, dtype=np.float64)) / hd)
    ang = positions.astype(np.float64)[:, None] * inv_freq[None, :]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Softmax(q k^T / sqrt(hd)) v with a causal mask, grouped-query heads.
    q: [T, Hq, hd]; k, v: [T, Hkv, hd] -> [T, Hq, hd]."""
    t, hq, hd = q.shape
    hkv = k.shape[1]
    group = hq // hkv
    out = np.empty_like(q)
    future = np.triu(np.ones((t, t), dtype=bool), 1)
    for h in range(hq):
        kv = h // group
        s = (q[:, h, :] @ k[:, kv, :].T) / np.sqrt(hd)
        s[future] = -np.inf
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, kv, :]
    return out


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


class Model:
    """Upcast view of a bf16 weight dict (names as in the input generator's
    tensor order).  Layers are upcast on demand so that the 8B shape fits."""

    def __init__(self, shape, weights: Dict[str, np.ndarray], cache_layers: bool = False):
        self.s = shape
        self.w = weights
        self._cache: Dict[str, np.ndarray] = {}
        self.cache_layers = cache_layers

    def get(self, name: str) -> np.ndarray:
        if name in self._cache:
            return self._cache[name]
        a = bf16_to_f64(self.w[name])
        if self.cache_layers:
            self._cache[name] = a
        return a

    def embed_rows(self, ids: np.ndarray) -> np.ndarray:
        return bf16_to_f64(self.w["embed"][ids])

    def label_head(self, labels: Sequence[int]):
        return bf16_to_f64(self.w["lm_head"][list(labels)]), \
            bf16_to_f64(self.w["lm_bias"][list(labels)])


def decoder_layer(x: np.ndarray, m: Model, l: int, lw: Dict[str, np.ndarray]) -> np.ndarray:
    """One pre-norm block on one row's hidden states x [T, d]."""
    s = m.s
    t = x.shape[0]
    pos = np.arange(t)
    h = rmsnorm(x, lw["attn_norm"], s.rms_eps)
    q = (h @ lw["wq"].T).reshape(t, s.n_heads, s.head_dim)
    k = (h @ lw["wk"].T).reshape(t, s.n_kv_heads, s.head_dim)
    v = (h @ lw["wv"].T).reshape(t, s.n_kv_heads, s.head_dim)
    q = rope(q, pos, s.rope_theta)
    k = rope(k, pos, s.rope_theta)
    a = causal_attention(q, k, v).reshape(t, s.q_dim)
    x = x + a @ lw["wo"].T
    h = rmsnorm(x, lw["mlp_norm"], s.rms_eps)
    x = x + (silu(h @ lw["wg"].T) * (h @ lw["wu"].T)) @ lw["wd"].T
    return x


LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")


def hidden_states(m: Model, seqs: List[np.ndarray], n_layers: int | None = None) -> List[np.ndarray]:
    """Residual stream after ``n_layers`` blocks (all by default) for each
    token sequence, every sequence run on its own.  Layer weights are upcast
    once per layer and reused across the sequences."""
    xs = [m.embed_rows(np.asarray(q, dtype=np.int64)) for q in seqs]
    for l in range(m.s.n_layers if n_layers is None else n_layers):
        lw = {n: m.get(f"l{l}.{n}") for n in LAYER_TENSORS}
        xs = [decoder_layer(x, m, l, lw) for x in xs]
    return xs


def label_logits(m: Model, seqs: List[np.ndarray], labels: Sequence[int]) -> np.ndarray:
    """Logits of the label tokens at each sequence's last position [S, K]:
    final RMSNorm of the last hidden state, dot the label rows of the LM
    head, plus the LM-head bias (Fig. 2: logits[:, -1, :] at the label ids)."""
    out = np.zeros((len(seqs), len(labels)), dtype=np.float64)
    if not seqs:
        return out
    g = m.get("final_norm")
    w_lab, b_lab = m.label_head(labels)
    for i, x in enumerate(hidden_states(m, seqs)):
        h = rmsnorm(x[-1], g, m.s.rms_eps)
        out[i] = w_lab @ h + b_lab
    return out


def vocab_logits(m: Model, seqs: List[np.ndarray]) -> np.ndarray:
    """Full-vocabulary logits at every position of one sequence [T, V]:
    final RMSNorm of each hidden state, times the whole LM head, plus its
    bias.  Row t is the next-token distribution after seq[:t+1] (causal)."""
    assert len(seqs) == 1
    x = hidden_states(m, seqs)[0]
    h = rmsnorm(x, m.get("final_norm"), m.s.rms_eps)
    return h @ bf16_to_f64(m.w["lm_head"]).T + bf16_to_f64(m.w["lm_bias"])


def first_argmax(z: np.ndarray) -> int:
    """Index of the largest value; the lowest index among equal maxima."""
    return int(np.flatnonzero(z == z.max())[0])


def greedy_generate(m: Model, prompt: np.ndarray, n_new: int, eos: int = -1,
                    pad: int = 0):
    """AI_TRANSFORM (Table 1: causal-LM forward with generative decoding,
    output masked with a pad id): ``n_new`` greedy steps, each one a full
    forward over prompt ++ tokens generated so far (no key/value cache) and
    the first argmax of the last position's vocabulary logits.  Once the
    model emits ``eos`` the remaining positions hold ``pad``.

    Returns (tokens [n_new] int64, text_len): text_len counts the tokens
    before the eos (n_new when none was emitted)."""
    seq = [int(t) for t in prompt]
    out = np.full(n_new, pad, dtype=np.int64)
    text_len = n_new
    for t in range(n_new):
        z = vocab_logits(m, [np.asarray(seq, dtype=np.int64)])[-1]
        y = first_argmax(z)
        out[t] = y
        if y == eos:
            text_len = t
            break
        seq.append(y)
    return out, text_len
