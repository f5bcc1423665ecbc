"""AI_TRANSFORM (greedy generation) and the LIKE filter through the C-ABI,
against the fp64 oracle (Table 1 AI_TRANSFORM row; Table 2 Q3 and Q5).

Greedy decoding turns floating point into integers at every step, and two
correct implementations may pick different tokens where the two largest
logits are within rounding of each other.  So each generated sequence is
checked by teacher forcing: the oracle runs the prompt followed by the GPU's
own tokens and every GPU token must be an argmax of the oracle's logits
within the parity tolerance (2e-2 * max(1, |max logit|)); where the oracle's
top two logits are further apart than that, this forces the same token.
The eos / pad masking, the LIKE matches, the count and the ids are compared
exactly (the oracle's LIKE applied to the GPU's tokens)."""
from dataclasses import replace

import numpy as np
import pytest

import synth
from helpers import check_greedy, gpu_ctx, weights_list
from oracle import query as oq
from oracle import relational as rel
from oracle import transformer as tf
from paper_2608_10139_gb300 import aiq

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = gpu_ctx()
    yield c
    c.close()


def _tiny_inputs(shape=synth.TINY, n_rows=96, seed=5, empty_every=0):
    rng = np.random.default_rng(seed)
    lens = rng.integers(1, 40, n_rows)
    if empty_every:
        lens[::empty_every] = 0
    off = np.zeros(n_rows + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = rng.integers(0, shape.vocab, int(off[-1])).astype(np.int32)
    cols = {"r": rng.integers(0, 10, n_rows).astype(np.int32)}
    prefix = rng.integers(0, shape.vocab, 16).astype(np.int32)
    return synth.Table(n_rows, cols, off, toks), prefix


def _run(ctx, shape, W, table, prefix, preds, max_new, eos=-1, pad=0, like=None, match_tokens=False, budget=None):
    m = ctx.load_model(shape, weights_list(shape, W))
    t = ctx.load_table(table.cols, (table.offsets, table.tokens))
    if budget:   # small chunks, so that several decode batches run
        ctx.set_option("token_budget", budget)
        ctx.set_option("decode_rows", 8)
    try:
        return ctx.run_transform(t, m, preds, prefix, max_new, eos=eos, pad=pad, like=like,
                                 match_tokens=match_tokens)
    finally:
        ctx.set_option("token_budget", 131072)
        ctx.set_option("decode_rows", 4096)
        ctx.free_table(t)
        ctx.free_model(m)


SHAPES = {
    "tiny_mha_hd32": synth.TINY,
    "gqa4_hd64": replace(synth.TINY, d_model=256, n_heads=8, n_kv_heads=2, head_dim=64, d_ffn=512),
    "gqa8_hd128": replace(synth.TINY, d_model=256, n_heads=8, n_kv_heads=1, head_dim=128, d_ffn=384),
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_transform_greedy_matches_oracle(ctx, name):
    shape = SHAPES[name]
    W = synth.make_weights(shape, 3001)
    table, prefix = _tiny_inputs(shape, seed=7, empty_every=11)
    preds = [("r", rel.GE, 4)]
    r = _run(ctx, shape, W, table, prefix, preds, 8, budget=400)   # several chunks
    cand = rel.compact(rel.predicate_mask(table.cols, preds, table.n_rows))
    assert np.array_equal(r.gen_row_ids, cand)
    assert r.count == -1 and r.gen_tokens.shape == (len(cand), 8)
    assert np.all(r.gen_text_len == 8)
    prompts = oq.prompts(prefix, table.offsets, table.tokens, cand)
    worst, flips = check_greedy(tf.Model(shape, W), prompts, r.gen_tokens, r.gen_text_len, -1, 0, name)
    print(f"{name}: worst gap ratio {worst:.3f}, near-tie flips {flips}")


def test_transform_permutation_model_exact(ctx):
    # identity embedding, zero blocks, unit gains, permutation LM head: y_t = pi^(t+1)(last prompt token)
    v = 128
    shape = replace(synth.TINY, d_model=v, vocab=v, n_heads=4, n_kv_heads=4, head_dim=32, d_ffn=128)
    W = synth.make_weights(shape, 0, zero=True)
    W["embed"] = synth.f32_to_bf16_bits(np.eye(v, dtype=np.float32))
    perm = np.random.default_rng(9).permutation(v)
    head = np.zeros((v, v), np.float32)
    head[perm, np.arange(v)] = 1.0
    W["lm_head"] = synth.f32_to_bf16_bits(head)
    one = synth.f32_to_bf16_bits(np.ones(v, np.float32))
    for l in range(shape.n_layers):
        W[f"l{l}.attn_norm"] = one
        W[f"l{l}.mlp_norm"] = one
    W["final_norm"] = one
    table, prefix = _tiny_inputs(shape, n_rows=40, seed=2, empty_every=7)
    r = _run(ctx, shape, W, table, prefix, [], 12)
    last = [int(table.tokens[table.offsets[i + 1] - 1]) if table.offsets[i + 1] > table.offsets[i]
            else int(prefix[-1]) for i in range(table.n_rows)]
    want = np.zeros((table.n_rows, 12), np.int64)
    for i, x in enumerate(last):
        for t in range(12):
            x = int(perm[x])
            want[i, t] = x
    assert np.array_equal(r.gen_tokens, want)
    # eos = the third token of row 0: that row stops there, every row pads after its first eos
    eos = int(want[0, 2])
    r2 = _run(ctx, shape, W, table, prefix, [], 12, eos=eos, pad=5)
    for i in range(table.n_rows):
        hits = np.flatnonzero(want[i] == eos)
        L = int(hits[0]) if len(hits) else 12
        assert r2.gen_text_len[i] == L
        assert np.array_equal(r2.gen_tokens[i, :L], want[i, :L])
        if L < 12:
            assert r2.gen_tokens[i, L] == eos and np.all(r2.gen_tokens[i, L + 1:] == 5)


def test_transform_eos_like_and_match_tokens(ctx):
    shape = SHAPES["gqa4_hd64"]
    W = synth.make_weights(shape, 3002)
    table, prefix = _tiny_inputs(shape, seed=8)
    preds = [("r", rel.LT, 7)]
    base = _run(ctx, shape, W, table, prefix, preds, 10)
    cand = base.gen_row_ids
    # an eos the model actually emits: the most frequent token at step 3
    vals, cnt = np.unique(base.gen_tokens[:, 3], return_counts=True)
    eos = int(vals[np.argmax(cnt)])
    r = _run(ctx, shape, W, table, prefix, preds, 10, eos=eos, pad=1)
    prompts = oq.prompts(prefix, table.offsets, table.tokens, cand)
    check_greedy(tf.Model(shape, W), prompts, r.gen_tokens, r.gen_text_len, eos, 1, "eos")
    assert np.any(r.gen_text_len < 10)
    # LIKE: a bigram taken from one row's text, then an unmatchable pattern, then the empty pattern
    row = int(np.argmax(r.gen_text_len))
    pat = [int(x) for x in r.gen_tokens[row, 1:3]]
    lk = _run(ctx, shape, W, table, prefix, preds, 10, eos=eos, pad=1, like=pat, match_tokens=True)
    match = np.array([rel.like_contains(r.gen_tokens[i, :r.gen_text_len[i]], pat) for i in range(len(cand))])
    want = oq.like_aggregate(match, cand)
    assert lk.count == want["count"] >= 1
    assert np.array_equal(lk.row_ids, want["row_ids"])
    assert np.array_equal(lk.gen_row_ids, want["row_ids"])
    assert np.array_equal(lk.gen_tokens, r.gen_tokens[match])
    assert np.array_equal(lk.gen_text_len, r.gen_text_len[match])
    none = _run(ctx, shape, W, table, prefix, preds, 10, eos=eos, pad=1, like=[eos])   # eos is never text
    assert none.count == 0 and none.row_ids.size == 0 and none.gen_tokens.shape[0] == 0
    every = _run(ctx, shape, W, table, prefix, preds, 10, eos=eos, pad=1, like=[])
    assert every.count == len(cand) and np.array_equal(every.row_ids, cand)
    assert every.gen_tokens.shape[0] == 0          # tokens only with match_tokens


def test_transform_single_step_and_empty_selection(ctx):
    shape = synth.TINY
    W = synth.make_weights(shape, 3003)
    table, prefix = _tiny_inputs(shape, n_rows=30, seed=9, empty_every=4)
    r = _run(ctx, shape, W, table, prefix, [], 1)      # LM head on the prefill output only
    prompts = oq.prompts(prefix, table.offsets, table.tokens, np.arange(30))
    check_greedy(tf.Model(shape, W), prompts, r.gen_tokens, r.gen_text_len, -1, 0, "max_new=1")
    e = _run(ctx, shape, W, table, prefix, [("r", rel.GT, 100)], 4, like=[1, 2])
    assert e.n_candidates == 0 and e.count == 0 and e.row_ids.size == 0


def test_transform_rejects_bad_specs(ctx):
    shape = synth.TINY
    W = synth.make_weights(shape, 3004)
    table, prefix = _tiny_inputs(shape, n_rows=8, seed=1)
    for kw in (dict(max_new=0), dict(max_new=5000), dict(max_new=4, pad=shape.vocab),
               dict(max_new=4, eos=shape.vocab), dict(max_new=4, like=[shape.vocab])):
        n = kw.pop("max_new")
        with pytest.raises(aiq.AiqError) as ei:
            _run(ctx, shape, W, table, prefix, [], n, **kw)
        assert ei.value.status == aiq.ERR_INVALID_ARG


@pytest.mark.parametrize("hd,hq,hkv", [(32, 4, 4), (64, 8, 2), (128, 8, 1), (64, 32, 8), (128, 32, 8), (64, 16, 8)])
def test_op_decode_attention_matches_fp32_reference(ctx, hd, hq, hkv):
    torch = pytest.importorskip("torch")
    dev = "cuda"
    g = torch.Generator(device="cpu").manual_seed(hd + hq)
    R, P, cap, slot = 5, 7, 6, 3
    lens = torch.tensor([0, 3, 40, 1, 70])
    seq_start = torch.zeros(R + 1, dtype=torch.int32)
    seq_start[1:] = torch.cumsum(lens, 0)
    kd = hkv * hd
    qkv = torch.randn(R, (hq + 2 * hkv) * hd, generator=g).half()
    pkv = torch.randn(P, 2 * kd, generator=g).half()
    own = torch.randn(int(lens.sum()), 2 * kd, generator=g).half()
    gen = torch.randn(R, cap, 2 * kd, generator=g).half()
    d = {k: v.to(dev) for k, v in dict(qkv=qkv, pkv=pkv, own=own, gen=gen.clone(), ss=seq_start).items()}
    out = torch.empty(R, hq * hd, dtype=torch.float16, device=dev)
    ctx.op_decode_attention(d["qkv"].data_ptr(), R, hq, hkv, hd, d["own"].data_ptr(), d["ss"].data_ptr(),
                            d["gen"].data_ptr(), cap, slot, out.data_ptr(), prefix_kv=d["pkv"].data_ptr(), P=P)
    torch.cuda.synchronize()
    gen_after = d["gen"].cpu()
    want_gen = gen.clone()
    want_gen[:, slot, :kd] = qkv[:, hq * hd:(hq + hkv) * hd]
    want_gen[:, slot, kd:] = qkv[:, (hq + hkv) * hd:]
    assert torch.equal(gen_after, want_gen)            # the new key/value landed in the slot, bit for bit
    ref = torch.empty(R, hq * hd, dtype=torch.float32)
    for r in range(R):
        st, n = int(seq_start[r]), int(lens[r])
        keys = torch.cat([pkv, own[st:st + n], want_gen[r, :slot + 1]]).float()
        q = qkv[r, :hq * hd].float().view(hq, hd)
        for h in range(hq):
            kv = h // (hq // hkv)
            k = keys[:, kv * hd:(kv + 1) * hd]
            v = keys[:, kd + kv * hd:kd + (kv + 1) * hd]
            p = torch.softmax(q[h] @ k.T / hd ** 0.5, dim=0)
            ref[r, h * hd:(h + 1) * hd] = p @ v
    got = out.float().cpu()
    assert torch.allclose(got, ref, rtol=2e-3, atol=2e-3), (got - ref).abs().max()
