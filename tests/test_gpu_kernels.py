"""Step-level parity of the prefill kernels (tcgen05 GEMM with each fused
epilogue, RoPE table, RMSNorm, varlen GQA attention) against the oracle's
fp64 definitions, through the C-ABI (aiq_ops.h)."""
import numpy as np
import pytest

from helpers import gpu_ctx
from oracle import transformer as tf

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = gpu_ctx()
    yield c
    c.close()


def _h(a):
    t = torch.as_tensor(np.ascontiguousarray(a)).cuda()
    torch.cuda.synchronize()
    return t


def _np64(t):
    torch.cuda.synchronize()
    return t.float().cpu().numpy().astype(np.float64)


def _close(got, ref, rtol, atol, what):
    err = np.abs(got - ref)
    bound = atol + rtol * np.abs(ref)
    bad = err > bound
    assert not bad.any(), f"{what}: {bad.sum()} of {bad.size} outside tol, max err {err.max():.3g}"


GEMM_CASES = [  # M, N, K, bn
    (1, 128, 64, 128),
    (130, 384, 128, 128),
    (257, 512, 192, 256),
    (1000, 256, 2048, 256),
    (8192, 1024, 512, 256),   # more tiles than SMs: persistent loop, both accumulators
    (3000, 768, 1024, 128),
]


@pytest.mark.parametrize("M,N,K,bn", GEMM_CASES)
def test_gemm_f16_store(ctx, M, N, K, bn):
    rng = np.random.default_rng(M + N + K)
    A = rng.standard_normal((M, K)).astype(np.float16)
    B = (rng.standard_normal((N, K)) * 0.05).astype(np.float16)
    dA, dB = _h(A), _h(B)
    out = torch.zeros((M, N), dtype=torch.float16, device="cuda")
    ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, bn, 0, out.data_ptr(), N)
    ref = A.astype(np.float64) @ B.astype(np.float64).T
    _close(_np64(out), ref, 2e-3, 2e-3 * np.sqrt(K) * 0.05, f"f16 M{M} N{N} K{K}")


@pytest.mark.parametrize("epi", [2, 5])   # residual add in the epilogue threads / by TMA reduce-add tiles
@pytest.mark.parametrize("M,N,K,bn", GEMM_CASES[:4] + [GEMM_CASES[5]])
def test_gemm_residual_add(ctx, M, N, K, bn, epi):
    rng = np.random.default_rng(7 * M + N)
    A = rng.standard_normal((M, K)).astype(np.float16)
    B = (rng.standard_normal((N, K)) * 0.05).astype(np.float16)
    R = rng.standard_normal((M, N)).astype(np.float32)
    guard = rng.standard_normal((M + 40, N)).astype(np.float32)     # rows past M must stay untouched
    guard[:M] = R
    dA, dB, dR = _h(A), _h(B), _h(guard)
    ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, bn, epi, dR.data_ptr(), N)
    ref = R.astype(np.float64) + A.astype(np.float64) @ B.astype(np.float64).T
    got = _np64(dR)
    _close(got[:M], ref, 1e-5, 2e-6 * np.sqrt(K), f"resid{epi} M{M} N{N} K{K}")
    assert np.array_equal(got[M:], guard[M:].astype(np.float64))


@pytest.mark.parametrize("M,f,K,bn", [(130, 256, 128, 256), (700, 512, 256, 128), (2049, 1024, 512, 256)])
def test_gemm_swiglu(ctx, M, f, K, bn):
    rng = np.random.default_rng(M + f)
    A = rng.standard_normal((M, K)).astype(np.float16)
    Wg = (rng.standard_normal((f, K)) * 0.05).astype(np.float16)
    Wu = (rng.standard_normal((f, K)) * 0.05).astype(np.float16)
    ib = bn // 2
    inter = np.concatenate([np.concatenate([Wg[b:b + ib], Wu[b:b + ib]]) for b in range(0, f, ib)])
    dA, dB = _h(A), _h(inter)
    out = torch.zeros((M, f), dtype=torch.float16, device="cuda")
    ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, 2 * f, K, bn, 3, out.data_ptr(), f)
    a = A.astype(np.float64)
    ref = tf.silu(a @ Wg.astype(np.float64).T) * (a @ Wu.astype(np.float64).T)
    _close(_np64(out), ref, 3e-3, 3e-3 * K * 0.0025, f"swiglu M{M} f{f}")


def test_rope_table(ctx):
    max_pos, hd, theta = 1200, 64, 1.0e4
    cs = torch.zeros((max_pos, hd // 2), dtype=torch.float32, device="cuda")
    sn = torch.zeros_like(cs)
    ctx.op_rope_table(cs.data_ptr(), sn.data_ptr(), max_pos, hd, theta)
    ang = np.arange(max_pos)[:, None] * theta ** (-(2.0 * np.arange(hd // 2)) / hd)[None, :]
    assert np.allclose(cs.cpu().numpy(), np.cos(ang), rtol=0, atol=1.2e-7)
    assert np.allclose(sn.cpu().numpy(), np.sin(ang), rtol=0, atol=1.2e-7)


@pytest.mark.parametrize("hd,Hq,Hkv,bn", [(32, 4, 4, 128), (64, 32, 8, 256), (128, 8, 2, 256)])
def test_gemm_qkv_rope(ctx, hd, Hq, Hkv, bn):
    rng = np.random.default_rng(hd)
    M, K = 300, 256
    N = (Hq + 2 * Hkv) * hd
    if N % bn:
        bn = 128
    A = rng.standard_normal((M, K)).astype(np.float16)
    B = (rng.standard_normal((N, K)) * 0.05).astype(np.float16)
    pos = rng.integers(0, 1100, M).astype(np.int32)
    max_pos = 1200
    cs = torch.zeros((max_pos, hd // 2), dtype=torch.float32, device="cuda")
    sn = torch.zeros_like(cs)
    ctx.op_rope_table(cs.data_ptr(), sn.data_ptr(), max_pos, hd, 1.0e4)
    dA, dB, dP = _h(A), _h(B), _h(pos)
    out = torch.zeros((M, N), dtype=torch.float16, device="cuda")
    rope_cols = (Hq + Hkv) * hd
    ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, bn, 1, out.data_ptr(), N, dP.data_ptr(),
                cs.data_ptr(), sn.data_ptr(), rope_cols, hd)
    y = A.astype(np.float64) @ B.astype(np.float64).T
    qk = y[:, :rope_cols].reshape(M, Hq + Hkv, hd)
    ref = np.concatenate([tf.rope(qk, pos, 1.0e4).reshape(M, rope_cols), y[:, rope_cols:]], axis=1)
    _close(_np64(out), ref, 2e-3, 2e-3 * np.sqrt(K) * 0.05, f"rope hd{hd}")


@pytest.mark.parametrize("d", [128, 2048, 4096])
def test_rmsnorm(ctx, d):
    rng = np.random.default_rng(d)
    T = 333
    x = (rng.standard_normal((T, d)) * 3).astype(np.float32)
    import synth
    gb = synth.f32_to_bf16_bits((1 + 0.02 * rng.standard_normal(d)).astype(np.float32))
    dx, dg = _h(x), _h(gb.view(np.int16))
    out = torch.zeros((T, d), dtype=torch.float16, device="cuda")
    ctx.op_rmsnorm(dx.data_ptr(), T, d, dg.data_ptr(), 1e-5, out.data_ptr())
    ref = tf.rmsnorm(x.astype(np.float64), tf.bf16_to_f64(gb), 1e-5)
    _close(_np64(out), ref, 1.5e-3, 1e-4, f"rmsnorm d{d}")


@pytest.mark.parametrize("hd,Hq,Hkv", [(32, 4, 4), (64, 8, 2), (128, 4, 1), (64, 8, 8), (64, 4, 2), (128, 16, 2)])
def test_attention_varlen(ctx, hd, Hq, Hkv):
    rng = np.random.default_rng(hd + Hq)
    lens = [1, 5, 64, 65, 130, 300, 17]
    T = sum(lens)
    W = (Hq + 2 * Hkv) * hd
    qkv = rng.standard_normal((T, W)).astype(np.float16)
    starts = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    dq, ds = _h(qkv), _h(starts)
    out = torch.zeros((T, Hq * hd), dtype=torch.float16, device="cuda")
    ctx.op_attention(dq.data_ptr(), T, ds.data_ptr(), len(lens), Hq, Hkv, hd, out.data_ptr())
    got = _np64(out)
    q64 = qkv.astype(np.float64)
    for i, n in enumerate(lens):
        s = starts[i]
        seg = q64[s:s + n]
        q = seg[:, :Hq * hd].reshape(n, Hq, hd)
        k = seg[:, Hq * hd:(Hq + Hkv) * hd].reshape(n, Hkv, hd)
        v = seg[:, (Hq + Hkv) * hd:].reshape(n, Hkv, hd)
        ref = tf.causal_attention(q, k, v).reshape(n, Hq * hd)
        _close(got[s:s + n], ref, 4e-3, 4e-3, f"attention seq {i} len {n} hd {hd}")


@pytest.mark.parametrize("hd,Hq,Hkv,P", [(32, 4, 4, 16), (64, 8, 2, 64), (64, 8, 2, 70), (128, 4, 1, 130),
                                         (64, 32, 8, 64), (128, 32, 8, 128)])
def test_attention_with_shared_prefix(ctx, hd, Hq, Hkv, P):
    """Rows attend a shared prefix's keys/values plus their own: the output at
    each row token equals the oracle's attention over prefix ++ row at that position."""
    rng = np.random.default_rng(P + hd)
    lens = [1, 5, 64, 65, 130, 17]
    T = sum(lens)
    W = (Hq + 2 * Hkv) * hd
    pre = rng.standard_normal((P, W)).astype(np.float16)
    rows = rng.standard_normal((T, W)).astype(np.float16)
    pkv = np.ascontiguousarray(pre[:, Hq * hd:])            # [P, 2 Hkv hd]: keys then values
    starts = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    dq, ds, dp = _h(rows), _h(starts), _h(pkv)
    out = torch.zeros((T, Hq * hd), dtype=torch.float16, device="cuda")
    ctx.op_attention(dq.data_ptr(), T, ds.data_ptr(), len(lens), Hq, Hkv, hd, out.data_ptr(), dp.data_ptr(), P)
    got = _np64(out)
    for i, n in enumerate(lens):
        seq = np.concatenate([pre, rows[starts[i]:starts[i] + n]]).astype(np.float64)
        m = P + n
        q = seq[:, :Hq * hd].reshape(m, Hq, hd)
        k = seq[:, Hq * hd:(Hq + Hkv) * hd].reshape(m, Hkv, hd)
        v = seq[:, (Hq + Hkv) * hd:].reshape(m, Hkv, hd)
        ref = tf.causal_attention(q, k, v).reshape(m, Hq * hd)[P:]
        _close(got[starts[i]:starts[i] + n], ref, 4e-3, 4e-3, f"prefix attention P{P} seq {i} len {n}")


@pytest.mark.parametrize("pair", [0, 1])
@pytest.mark.parametrize("M,N,K,epi", [(512, 256, 128, 0), (1000, 512, 2048, 0), (4099, 1536, 512, 2),
                                       (4099, 1536, 512, 5), (3000, 2048, 256, 3), (70000, 1024, 256, 0),
                                       (1024, 512, 8192, 2),   # the down projection's depth
                                       (600, 256, 192, 0)])    # K % 128 != 0: CTA pairs fall back to one CTA
def test_gemm_cta_pair_vs_single(ctx, pair, M, N, K, epi):
    """256 x 256 tiles on CTA pairs (tcgen05 cta_group::2) and 128 x 256 tiles on
    single CTAs give the oracle's product, ragged M included."""
    rng = np.random.default_rng(M + N + K + epi)
    A = rng.standard_normal((M, K)).astype(np.float16)
    B = (rng.standard_normal((N, K)) * 0.05).astype(np.float16)
    dA, dB = _h(A), _h(B)
    a, b = A.astype(np.float64), B.astype(np.float64)
    ctx.set_option("gemm_pair", pair)
    try:
        if epi == 0:
            out = torch.zeros((M, N), dtype=torch.float16, device="cuda")
            ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, 256, 0, out.data_ptr(), N)
            _close(_np64(out), a @ b.T, 2e-3, 2e-3 * np.sqrt(K) * 0.05, f"pair{pair} f16 M{M}")
        elif epi in (2, 5):
            R = rng.standard_normal((M, N)).astype(np.float32)
            dR = _h(R)
            ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, 256, epi, dR.data_ptr(), N)
            _close(_np64(dR), R.astype(np.float64) + a @ b.T, 1e-5, 2e-6 * np.sqrt(K), f"pair{pair} resid M{M}")
        else:
            f = N // 2
            g, u = b[:f], b[f:]
            inter = np.concatenate([np.concatenate([B[i:i + 128], B[f + i:f + i + 128]]) for i in range(0, f, 128)])
            dI = _h(inter)
            out = torch.zeros((M, f), dtype=torch.float16, device="cuda")
            ctx.op_gemm(dA.data_ptr(), K, dI.data_ptr(), K, M, N, K, 256, 3, out.data_ptr(), f)
            ref = tf.silu(a @ g.T) * (a @ u.T)
            _close(_np64(out), ref, 3e-3, 3e-3 * K * 0.0025, f"pair{pair} swiglu M{M}")
    finally:
        ctx.set_option("gemm_pair", 1)


def test_gemm_cta_pair_rope(ctx):
    rng = np.random.default_rng(99)
    hd, Hq, Hkv, M, K = 64, 32, 8, 1300, 512
    N = (Hq + 2 * Hkv) * hd
    A = rng.standard_normal((M, K)).astype(np.float16)
    B = (rng.standard_normal((N, K)) * 0.05).astype(np.float16)
    pos = rng.integers(0, 1100, M).astype(np.int32)
    cs = torch.zeros((1200, hd // 2), dtype=torch.float32, device="cuda")
    sn = torch.zeros_like(cs)
    ctx.op_rope_table(cs.data_ptr(), sn.data_ptr(), 1200, hd, 1.0e4)
    dA, dB, dP = _h(A), _h(B), _h(pos)
    out = torch.zeros((M, N), dtype=torch.float16, device="cuda")
    rope_cols = (Hq + Hkv) * hd
    ctx.op_gemm(dA.data_ptr(), K, dB.data_ptr(), K, M, N, K, 256, 1, out.data_ptr(), N, dP.data_ptr(),
                cs.data_ptr(), sn.data_ptr(), rope_cols, hd)
    y = A.astype(np.float64) @ B.astype(np.float64).T
    qk = y[:, :rope_cols].reshape(M, Hq + Hkv, hd)
    ref = np.concatenate([tf.rope(qk, pos, 1.0e4).reshape(M, rope_cols), y[:, rope_cols:]], axis=1)
    _close(_np64(out), ref, 2e-3, 2e-3 * np.sqrt(K) * 0.05, "pair rope")


def test_attention_tcgen05_matches_mma_sync_kernel(ctx):
    """The tcgen05 and the mma.sync attention kernels agree on a GQA batch with a
    shared prefix (both also match the oracle above)."""
    rng = np.random.default_rng(5)
    hd, Hq, Hkv, P = 64, 32, 8, 64
    lens = [3, 40, 64, 97, 200, 1]
    T = sum(lens)
    W = (Hq + 2 * Hkv) * hd
    pre = rng.standard_normal((P, W)).astype(np.float16)
    rows = rng.standard_normal((T, W)).astype(np.float16)
    pkv = np.ascontiguousarray(pre[:, Hq * hd:])
    starts = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    dq, ds, dp = _h(rows), _h(starts), _h(pkv)
    outs = []
    for tc in (1, 0):
        ctx.set_option("attention_tc", tc)
        out = torch.zeros((T, Hq * hd), dtype=torch.float16, device="cuda")
        ctx.op_attention(dq.data_ptr(), T, ds.data_ptr(), len(lens), Hq, Hkv, hd, out.data_ptr(), dp.data_ptr(), P)
        outs.append(_np64(out))
    ctx.set_option("attention_tc", 1)
    _close(outs[0], outs[1], 4e-3, 4e-3, "tcgen05 vs mma.sync attention")


@pytest.mark.parametrize("hd,growing", [(64, False), (64, True), (128, True)])
def test_attention_tcgen05_many_items_per_cta(ctx, hd, growing):
    """A batch large enough that every persistent CTA of the tcgen05 kernel runs
    hundreds of work items back to back (item boundaries, alternating output
    accumulators, read-outs after the next item's first block), against the
    mma.sync kernel on every element and the oracle on sampled rows.  With
    growing keys the scores rise along each row, so the running maximum grows
    by more than 2^8 inside items and the output is rescaled in place."""
    rng = np.random.default_rng(hd + 17 * growing)
    Hq, Hkv, P = 32, 8, 64
    n_rows = 2500 if hd == 64 else 1200          # about 300 work items per CTA either way
    lens = np.clip(np.round(np.exp(rng.normal(np.log(120.0), 0.5, n_rows))), 1, 512).astype(np.int64)
    T = int(lens.sum())
    W = (Hq + 2 * Hkv) * hd
    starts = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rows = rng.standard_normal((T, W), dtype=np.float32)
    pre = rng.standard_normal((P, W), dtype=np.float32)
    if growing:
        # keys scaled by 1 + position / 24 (prefix keys at their positions, row keys after them)
        pos = np.concatenate([np.arange(n) for n in lens]) + P
        rows[:, Hq * hd:(Hq + Hkv) * hd] *= (1.0 + pos / 24.0)[:, None] * 0.35
        pre[:, Hq * hd:(Hq + Hkv) * hd] *= (1.0 + np.arange(P) / 24.0)[:, None] * 0.35
    rows, pre = rows.astype(np.float16), pre.astype(np.float16)
    pkv = np.ascontiguousarray(pre[:, Hq * hd:])
    dq, ds, dp = _h(rows), _h(starts), _h(pkv)
    outs = []
    for tc in (1, 0):
        ctx.set_option("attention_tc", tc)
        out = torch.zeros((T, Hq * hd), dtype=torch.float16, device="cuda")
        ctx.op_attention(dq.data_ptr(), T, ds.data_ptr(), len(lens), Hq, Hkv, hd, out.data_ptr(), dp.data_ptr(), P)
        outs.append(_np64(out))
    ctx.set_option("attention_tc", 1)
    assert np.isfinite(outs[0]).all()
    _close(outs[0], outs[1], 4e-3, 4e-3, f"tcgen05 vs mma.sync attention, {T} tokens, hd {hd}")
    for i in rng.choice(len(lens), 4, replace=False):
        s, n = int(starts[i]), int(lens[i])
        seq = np.concatenate([pre, rows[s:s + n]]).astype(np.float64)
        m = P + n
        q = seq[:, :Hq * hd].reshape(m, Hq, hd)
        k = seq[:, Hq * hd:(Hq + Hkv) * hd].reshape(m, Hkv, hd)
        v = seq[:, (Hq + Hkv) * hd:].reshape(m, Hkv, hd)
        ref = tf.causal_attention(q, k, v).reshape(m, Hq * hd)[P:]
        _close(outs[0][s:s + n], ref, 4e-3, 4e-3, f"tcgen05 attention row {i} len {n}")
