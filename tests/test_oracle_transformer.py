"""Pins of the oracle's fp64 decoder against closed forms, invariants, a
hand-worked block and library routines (torch CPU), CPU only."""
import os
from dataclasses import replace

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import transformer as tf

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")

SMALL = synth.ModelShape(n_layers=2, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16,
                         d_ffn=96, vocab=300)


def _bf16(a):
    return synth.f32_to_bf16_bits(np.asarray(a, np.float32))


def test_bf16_upcast_exact():
    x = np.array([1.0, -2.5, 3.140625, 1e-3, 0.0], np.float32)
    b = _bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(tf.bf16_to_f64(b), ref)


def test_rmsnorm_constant_row_and_torch():
    g = np.array([1.0, 2.0, -0.5, 3.0])
    x = np.full((1, 4), -2.0)
    eps = 1e-5
    want = -2.0 / np.sqrt(4.0 + eps) * g
    assert np.allclose(tf.rmsnorm(x, g, eps), want, rtol=0, atol=1e-15)
    r = np.random.default_rng(0).standard_normal((5, 33))
    gg = np.random.default_rng(1).standard_normal(33)
    lib = F.rms_norm(torch.from_numpy(r), (33,), torch.from_numpy(gg), eps).numpy()
    assert np.allclose(tf.rmsnorm(r, gg, eps), lib, rtol=1e-12, atol=1e-12)


def test_silu_matches_torch():
    z = np.linspace(-20, 20, 101)
    assert np.allclose(tf.silu(z), F.silu(torch.from_numpy(z)).numpy(), rtol=1e-13, atol=1e-15)


def test_swiglu_block_hand_worked():
    vals = {}
    for line in open(os.path.join(GOLDEN, "swiglu_rmsnorm_d2.txt")):
        if line.strip() and not line.startswith("#"):
            k, *v = line.split()
            vals[k] = np.array([float(t) for t in v])
    x = vals["x"][None, :]
    h = tf.rmsnorm(x, vals["g"], 0.0)
    wg, wu, wd = np.array([[1.0, 0.0]]), np.array([[0.0, 1.0]]), np.array([[1.0], [-1.0]])
    out = x + (tf.silu(h @ wg.T) * (h @ wu.T)) @ wd.T
    assert np.allclose(out[0], vals["out"], rtol=0, atol=1e-14)


def test_rope_half_split_pairs_closed_form():
    # hd = 4: pairs (0, 2) and (1, 3); inv_freq = (1, theta^-0.5)
    theta = 100.0
    for p in [0, 1, 5]:
        x = np.array([[[1.0, 0.0, 0.0, 0.0]]])
        y = tf.rope(x, np.array([p]), theta)[0, 0]
        assert np.allclose(y, [np.cos(p), 0.0, np.sin(p), 0.0], atol=1e-15)
        x = np.array([[[0.0, 1.0, 0.0, 0.0]]])
        y = tf.rope(x, np.array([p]), theta)[0, 0]
        a = p * theta ** -0.5
        assert np.allclose(y, [0.0, np.cos(a), 0.0, np.sin(a)], atol=1e-15)


def test_rope_position_zero_identity_norm_and_relative():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 1, 32))
    k = rng.standard_normal((1, 1, 32))
    assert np.array_equal(tf.rope(q, np.array([0]), 1e4), q)
    for p in [3, 700]:
        assert np.isclose(np.linalg.norm(tf.rope(q, np.array([p]), 1e4)), np.linalg.norm(q))
    def score(m, n):
        return float(np.sum(tf.rope(q, np.array([m]), 1e4) * tf.rope(k, np.array([n]), 1e4)))
    assert np.isclose(score(10, 4), score(106, 100), rtol=1e-10, atol=1e-12)
    assert not np.isclose(score(10, 4), score(10, 5))


def test_attention_matches_torch_sdpa():
    rng = np.random.default_rng(4)
    t, hq, hkv, hd = 9, 6, 2, 8
    q, k, v = (rng.standard_normal((t, h, hd)) for h in (hq, hkv, hkv))
    got = tf.causal_attention(q, k, v)
    rep = hq // hkv
    kt = torch.from_numpy(k).repeat_interleave(rep, dim=1)
    vt = torch.from_numpy(v).repeat_interleave(rep, dim=1)
    lib = F.scaled_dot_product_attention(torch.from_numpy(q).transpose(0, 1), kt.transpose(0, 1),
                                         vt.transpose(0, 1), is_causal=True).transpose(0, 1)
    assert np.allclose(got, lib.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_identical_keys_is_prefix_mean_and_length_one():
    rng = np.random.default_rng(5)
    t, hd = 7, 4
    q = rng.standard_normal((t, 2, hd))
    k = np.tile(rng.standard_normal((1, 1, hd)), (t, 1, 1))
    v = rng.standard_normal((t, 1, hd))
    out = tf.causal_attention(q, k, v)
    for i in range(t):
        assert np.allclose(out[i, 0], v[: i + 1, 0].mean(0), atol=1e-14)
        assert np.allclose(out[i, 1], v[: i + 1, 0].mean(0), atol=1e-14)
    one = tf.causal_attention(q[:1], k[:1], v[:1])
    assert np.allclose(one[0, 0], v[0, 0]) and np.allclose(one[0, 1], v[0, 0])


def test_gqa_head_mapping():
    # kv head j carries the constant value j+1; query head h must read kv head h // (Hq/Hkv)
    t, hq, hkv, hd = 5, 8, 2, 4
    rng = np.random.default_rng(6)
    q = rng.standard_normal((t, hq, hd))
    k = rng.standard_normal((t, hkv, hd))
    v = np.stack([np.full((t, hd), j + 1.0) for j in range(hkv)], axis=1)
    out = tf.causal_attention(q, k, v)
    for h in range(hq):
        assert np.allclose(out[:, h], h // (hq // hkv) + 1.0)


def _weights(shape, seed, **overrides):
    w = synth.make_weights(shape, seed)
    for name, val in overrides.items():
        w[name] = val
    return w


def test_zero_weights_give_lm_bias():
    s = SMALL
    w = synth.make_weights(s, 0, zero=True)
    w["lm_bias"] = _bf16(np.random.default_rng(7).standard_normal(s.vocab))
    m = tf.Model(s, w)
    seqs = [np.array([1, 2, 3]), np.array([299])]
    labels = [100, 101, 5]
    z = tf.label_logits(m, seqs, labels)
    b = tf.bf16_to_f64(w["lm_bias"][labels])
    assert np.array_equal(z, np.tile(b, (2, 1)))


def test_identity_layers_closed_form():
    # W_o = W_d = 0 makes every block the identity: logits come from the last token's embedding
    s = SMALL
    w = synth.make_weights(s, 11)
    for l in range(s.n_layers):
        w[f"l{l}.wo"] = np.zeros_like(w[f"l{l}.wo"])
        w[f"l{l}.wd"] = np.zeros_like(w[f"l{l}.wd"])
    m = tf.Model(s, w)
    seq = np.array([5, 17, 42, 9])
    labels = [100, 101]
    z = tf.label_logits(m, [seq], labels)[0]
    e = tf.bf16_to_f64(w["embed"][9])
    g = tf.bf16_to_f64(w["final_norm"])
    h = e * g / np.sqrt(np.dot(e, e) / s.d_model + s.rms_eps)
    want = [np.dot(tf.bf16_to_f64(w["lm_head"][j]), h) + tf.bf16_to_f64(w["lm_bias"][j:j + 1])[0]
            for j in labels]
    assert np.allclose(z, want, rtol=1e-13, atol=1e-13)


def test_uniform_attention_layer_closed_form():
    # One layer, W_q = 0 (all scores zero: uniform causal attention, RoPE irrelevant),
    # W_d = 0: x_out[i] = x[i] + (mean_{j<=i} rmsnorm(x_j) W_v^T) W_o^T   (Hq = Hkv)
    s = replace(SMALL, n_layers=1, n_kv_heads=4)
    w = synth.make_weights(s, 12)
    w["l0.wq"] = np.zeros_like(w["l0.wq"])
    w["l0.wd"] = np.zeros_like(w["l0.wd"])
    m = tf.Model(s, w)
    seq = np.array([3, 1, 4, 1, 5, 9])
    x = tf.bf16_to_f64(w["embed"][seq])
    xo = tf.hidden_states(m, [seq])[0]
    g = tf.bf16_to_f64(w["l0.attn_norm"])
    wv = tf.bf16_to_f64(w["l0.wv"])
    wo = tf.bf16_to_f64(w["l0.wo"])
    for i in range(len(seq)):
        vs = []
        for j in range(i + 1):
            xj = x[j]
            vs.append(wv @ (xj * g / np.sqrt(np.dot(xj, xj) / s.d_model + s.rms_eps)))
        want = x[i] + wo @ np.mean(vs, axis=0)
        assert np.allclose(xo[i], want, rtol=1e-12, atol=1e-12)


def test_causality_prefix_truncation():
    s = SMALL
    m = tf.Model(s, synth.make_weights(s, 13))
    seq = np.random.default_rng(8).integers(0, s.vocab, 12)
    full = tf.hidden_states(m, [seq])[0]
    for n in (1, 5, 12):
        part = tf.hidden_states(m, [seq[:n]])[0]
        assert np.allclose(part[-1], full[n - 1], rtol=1e-12, atol=1e-12)


def test_gqa_duplicated_kv_heads_equivalent():
    # A GQA model and the MHA model whose K/V head blocks are duplicated per query group agree.
    s = SMALL
    w = synth.make_weights(s, 14)
    s2 = replace(s, n_kv_heads=s.n_heads)
    w2 = dict(w)
    rep = s.n_heads // s.n_kv_heads
    for l in range(s.n_layers):
        for n in ("wk", "wv"):
            blocks = w[f"l{l}.{n}"].reshape(s.n_kv_heads, s.head_dim, s.d_model)
            w2[f"l{l}.{n}"] = np.repeat(blocks, rep, axis=0).reshape(s2.kv_dim, s.d_model)
    seqs = [np.array([1, 2, 3, 4, 5]), np.array([7])]
    a = tf.label_logits(tf.Model(s, w), seqs, [100, 101])
    b = tf.label_logits(tf.Model(s2, w2), seqs, [100, 101])
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)


def test_label_logits_match_torch_reference_forward():
    # An independent forward written with torch library layers (F.rms_norm,
    # F.scaled_dot_product_attention, F.silu) on the same weights.
    s = SMALL
    w = synth.make_weights(s, 15)
    seq = np.random.default_rng(9).integers(0, s.vocab, 10)
    T = lambda n: torch.from_numpy(tf.bf16_to_f64(w[n]))
    x = T("embed")[torch.from_numpy(seq)]
    t = len(seq)
    half = s.head_dim // 2
    inv = torch.tensor(s.rope_theta, dtype=torch.float64) ** (-torch.arange(0, s.head_dim, 2, dtype=torch.float64) / s.head_dim)
    ang = torch.arange(t, dtype=torch.float64)[:, None] * inv[None, :]
    cos = torch.cat([ang.cos(), ang.cos()], -1)[:, None, :]
    sin = torch.cat([ang.sin(), ang.sin()], -1)[:, None, :]
    rot = lambda u: torch.cat([-u[..., half:], u[..., :half]], -1)
    for l in range(s.n_layers):
        h = F.rms_norm(x, (s.d_model,), T(f"l{l}.attn_norm"), s.rms_eps)
        q = (h @ T(f"l{l}.wq").T).view(t, s.n_heads, s.head_dim)
        k = (h @ T(f"l{l}.wk").T).view(t, s.n_kv_heads, s.head_dim)
        v = (h @ T(f"l{l}.wv").T).view(t, s.n_kv_heads, s.head_dim)
        q, k = q * cos + rot(q) * sin, k * cos + rot(k) * sin
        rep = s.n_heads // s.n_kv_heads
        a = F.scaled_dot_product_attention(q.transpose(0, 1), k.repeat_interleave(rep, 1).transpose(0, 1),
                                           v.repeat_interleave(rep, 1).transpose(0, 1), is_causal=True)
        x = x + a.transpose(0, 1).reshape(t, -1) @ T(f"l{l}.wo").T
        h = F.rms_norm(x, (s.d_model,), T(f"l{l}.mlp_norm"), s.rms_eps)
        x = x + (F.silu(h @ T(f"l{l}.wg").T) * (h @ T(f"l{l}.wu").T)) @ T(f"l{l}.wd").T
    h = F.rms_norm(x[-1], (s.d_model,), T("final_norm"), s.rms_eps)
    lab = [100, 101]
    want = (T("lm_head")[lab] @ h + T("lm_bias")[lab]).numpy()
    got = tf.label_logits(tf.Model(s, w), [seq], lab)[0]
    assert np.allclose(got, want, rtol=1e-11, atol=1e-11)
