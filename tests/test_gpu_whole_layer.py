"""The encoder layer on the device, launched as the encoder benchmark
launches it -- QKV -> attention -> output projection + residual ->
LayerNorm -> FFN1 + GELU -> FFN2 + residual -> LayerNorm, int8 between, all
on one stream with no host step -- and every stage checked against the
oracle on that stage's own device input (so a rounding-boundary difference
in one stage does not spread into the next):

  * the linears and the residual epilogues: bit for bit;
  * attention: within the bound derived in test_gpu_attention.py, int8
    exact away from rounding boundaries;
  * LayerNorm: int8 exact except within 1e-3 of a rounding boundary (as in
    test_gpu_layernorm.py).

This also checks the ordering between the attention kernel and the output
projection that reads its context (the linear is launched with
programmatic dependent launch and waits for the previous grid before it
reads activations).  Shapes: the cfg4 layer's weights at 80%, 2 sequences
x 384 tokens, 12 heads.  The QKV weight's scales are scaled down so that
the int8 q and k, dequantised with the calibrated QKV scale, give scores
of a few units (the synthetic weights otherwise make the softmax one-hot)."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

BATCH, SEQ, HEADS = 2, 384, 12


@pytest.fixture(scope="module")
def bsg():
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


# device helpers (one place to swap for a CPU dry run of the test's logic)
def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def alloc(shape, dtype):
    return torch.empty(shape, dtype={np.int8: torch.int8, np.float32: torch.float32}[dtype], device="cuda")


def attention_bound(qkv, scale, seq, heads):
    d = heads * 64
    x = qkv.astype(np.int64)
    smax = 0.0
    for b in range(qkv.shape[0] // seq):
        rows = slice(b * seq, (b + 1) * seq)
        for h in range(heads):
            qk = x[rows, h * 64:(h + 1) * 64] @ x[rows, d + h * 64:d + (h + 1) * 64].T
            smax = max(smax, float(np.abs(qk).max()) * scale * scale / 8.0)
    vmax = float(np.abs(x[:, 2 * d:]).max()) * scale
    return (3 * seq * 2.0 ** -24 + 2.0 ** -16 + 2.0 ** -21 * (smax + 1) + (2 * -(-seq // 64) + 4) * 2.0 ** -24) * vmax


def check_i8_near(got, want_f64, inv, band, what):
    t = want_f64 * np.float64(inv)
    ref = np.clip(np.rint(t), -128, 127).astype(np.int64)
    g = got.astype(np.int64)
    diff = g != ref
    near = np.abs(np.abs(t - np.floor(t)) - 0.5) <= band
    bad = diff & ~(near & (np.abs(g - ref) == 1))
    assert not bad.any(), f"{what}: {int(bad.sum())} int8 values differ away from a rounding boundary"
    assert int(diff.sum()) <= g.size // 100, f"{what}: {int(diff.sum())} boundary flips"


def scale_of(y) -> float:
    return float(np.float32(np.max(np.abs(y))) / np.float32(127.0))


def test_encoder_layer_on_device(bsg):
    m = BATCH * SEQ
    weights, _ = synth.encoder_layer()
    wq, wo, w1, w2 = weights
    wq.scales = (wq.scales * np.float32(5e-3)).astype(np.float32)  # scores: std ~4, max ~19
    dense = [oracle.weight_dense(w) for w in weights]
    x0 = synth.draw_x(synth.rng_for(synth.SEED_BASE + 90), m, 768, "u127")
    rng = synth.rng_for(synth.SEED_BASE + 91)
    g1, b1, g2, b2 = (rng.normal(mu, 0.1, 768).astype(np.float32) for mu in (1.0, 0.0, 1.0, 0.0))
    x_scale, ln_scale, eps = 0.02, 4.0 / 127.0, 1e-12

    # calibration on the oracle (frozen constants for the device pass)
    s_qkv = scale_of(oracle.linear(x0, dense[0], wq.scales, wq.bias, oracle.F32, threads=8))
    qkv_ref = oracle.linear(x0, dense[0], wq.scales, wq.bias, oracle.I8, s_qkv, threads=8)
    att_ref = oracle.attention_f64(qkv_ref, s_qkv, BATCH, SEQ, HEADS, threads=8)
    s_ctx = scale_of(att_ref)
    z1_ref = oracle.linear_resid(oracle.requant_f32(att_ref.astype(np.float32), s_ctx), dense[1], wo.scales, wo.bias,
                                 x0, x_scale, threads=8)
    h1_ref = oracle.requant_f32(oracle.layernorm(z1_ref, g1, b1, eps).astype(np.float32), ln_scale)
    s_f1 = scale_of(oracle.linear(h1_ref, dense[2], w1.scales, w1.bias, oracle.F32_GELU, threads=8))
    lins = [bsg.SparseInt8Linear(w.n_out, w.k_in, w.indptr, w.colidx, w.values, w.scales, w.bias) for w in weights]

    # one device pass, all on the current stream
    xd = dev(x0)
    gd = [dev(a) for a in (g1, b1, g2, b2)]
    qkv, ctx = alloc((m, 2304), np.int8), alloc((m, 768), np.int8)
    z1, f1, z2 = alloc((m, 768), np.float32), alloc((m, 3072), np.int8), alloc((m, 768), np.float32)
    lins[0].run(xd, qkv, bsg.OUT_I8, s_qkv)
    bsg.attention(qkv, BATCH, SEQ, HEADS, s_qkv, bsg.OUT_I8, s_ctx, out=ctx)
    lins[1].run(ctx, z1, bsg.OUT_F32_RESID, residual=xd, residual_scale=x_scale)
    h1 = bsg.layernorm(z1, gd[0], gd[1], eps, bsg.OUT_I8, ln_scale)
    lins[2].run(h1, f1, bsg.OUT_I8_GELU, s_f1)
    lins[3].run(f1, z2, bsg.OUT_F32_RESID, residual=h1, residual_scale=ln_scale)
    h2 = bsg.layernorm(z2, gd[2], gd[3], eps, bsg.OUT_I8, ln_scale)
    qkv_h, ctx_h, z1_h, h1_h, f1_h, z2_h, h2_h = (host(t) for t in (qkv, ctx, z1, h1, f1, z2, h2))

    # stage by stage, each on its own device input
    assert np.array_equal(qkv_h, qkv_ref), "QKV"
    att = oracle.attention_f64(qkv_h, s_qkv, BATCH, SEQ, HEADS, threads=8)
    inv_ctx = float(np.float32(1.0) / np.float32(s_ctx))
    check_i8_near(ctx_h, att, inv_ctx, attention_bound(qkv_h, s_qkv, SEQ, HEADS) * inv_ctx + 1e-6, "attention")
    assert np.array_equal(z1_h, oracle.linear_resid(ctx_h, dense[1], wo.scales, wo.bias, x0, x_scale, threads=8)), \
        "output projection + residual"
    inv_ln = float(np.float32(1.0) / np.float32(ln_scale))
    check_i8_near(h1_h, oracle.layernorm(z1_h, g1, b1, eps), inv_ln, 1e-3, "LayerNorm 1")
    assert np.array_equal(f1_h, oracle.linear(h1_h, dense[2], w1.scales, w1.bias, oracle.I8_GELU, s_f1, threads=8)), \
        "FFN1"
    assert np.array_equal(z2_h, oracle.linear_resid(f1_h, dense[3], w2.scales, w2.bias, h1_h, ln_scale, threads=8)), \
        "FFN2 + residual"
    check_i8_near(h2_h, oracle.layernorm(z2_h, g2, b2, eps), inv_ln, 1e-3, "LayerNorm 2")
    for lin in lins:
        lin.close()
