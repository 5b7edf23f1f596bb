"""Multi-head self-attention on device (bsgemm_attention) against the fp64
oracle (oracle.attention_f64).

Tolerance, derived from the kernel's arithmetic (fifth-generation tensor
cores, f16 operands, fp32 accumulators).  The scores are exact int32 dot
products (int8 values are exact in f16, products below 2^14, partial sums
of 64 below 2^24).  A weight is e_j = 2^t_j, t_j = fl(d_j c2 - M) (a fused
multiply-add; d_j the dot product, c2 = c log2(e) within 2^-23 of its exact
value, M = fl(m c2) for a reference maximum m that moves only when a block's
maximum passes it by more than 8).  The rounding of M scales every weight
taken against it, the context and the sum by one factor, so t_j is within
2^-22.4 |u_j| of the exact u_j = (d_j - m) c log2(e).  For u_j <= 0 that
bounds the weight's error by 2^-23.8 absolute (2^u |u| ln 2 <= 1/e), for 0
< u_j <= 8 by 2^-20 relative; ex2.approx.ftz.f32 adds at most 2 ulp
(2^-22) relative (2^-22.73 measured on GB300 over every fp32 input in
[-126, 0]; results below 2^-126 flush to 0).  When M moves, the context and
the sum are scaled by alpha = 2^(M_old - M_new), the difference taken
exactly as two floats and alpha as the product of their two powers: 2^-21
+ 2^-24 per move, at most R = ceil(seq / 64) - 1 of them.  P enters the P v
product as two f16 parts (hi + lo), which drops at most 2^-22 e + 2^-25 of
each weight; the products with the exact f16 v are exact.  The sums of e_j
(fp32, in four running parts per warp, then the two warps' parts) and of
e_j v_j (the tensor cores' fp32 accumulation, two products a key, counted
as truncating adds) add at most seq_pad 2^-24 and 2 seq_pad 2^-23 relative
to their sums of magnitudes (seq_pad = 64 (R + 1)); the final scale and
product add 2^-23.  A weight's error enters the numerator and the sum, so
it counts twice; the sum is at least 1 (the reference key's weight).  In
units of vmax = max |v| * qkv_scale that is at most
    ((6 + 4 R) 2^-22 + 2^-19 + 2 R 2^-24 + seq 2^-22.4 + 5 seq_pad 2^-24 + 2^-23) vmax
per element.  A dropped or repeated key (weight ~ 1 / seq), a wrong scale
or head offset moves an element by orders of magnitude more.  int8 outputs
must equal rne(exact * inv) saturated, except within that bound (times inv)
of a rounding boundary, where the neighbour is allowed."""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu

HD = 64


@pytest.fixture(scope="module")
def bsg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


def draw_qkv(rng, batch, seq, heads, pad=0, std=35.0):
    """int8 QKV rows like a calibrated QKV linear's output: rounded normals,
    clipped to [-127, 127]; `pad` extra bytes per row hold noise that the
    kernel must not read into the result."""
    d = heads * HD
    q = np.clip(np.rint(rng.normal(0.0, std, size=(batch * seq, 3 * d))), -127, 127).astype(np.int8)
    if pad:
        q = np.concatenate([q, rng.integers(-128, 128, size=(batch * seq, pad)).astype(np.int8)], axis=1)
    return np.ascontiguousarray(q)


def bound(qkv, scale, batch, seq, heads):
    d = heads * HD
    vmax = float(np.abs(qkv[:, 2 * d:3 * d].astype(np.int64)).max()) * scale
    r = -(-seq // 64) - 1
    seq_pad = 64 * (r + 1)
    return ((6 + 4 * r) * 2.0 ** -22 + 2.0 ** -19 + 2 * r * 2.0 ** -24 + seq * 2.0 ** -22.4
            + 5 * seq_pad * 2.0 ** -24 + 2.0 ** -23) * vmax


def run_device(bsg, qkv, batch, seq, heads, scale, kind=None, out_scale=1.0, guard_rows=0, stream=None):
    import torch
    kind = bsg.OUT_F32 if kind is None else kind
    d = heads * HD
    dt = torch.int8 if kind == bsg.OUT_I8 else torch.float32
    buf = torch.full((batch * seq + guard_rows, d), 90 if dt == torch.int8 else 1234.5, dtype=dt, device="cuda")
    out = buf[:batch * seq]
    bsg.attention(torch.from_numpy(qkv).cuda(), batch, seq, heads, scale, kind, out_scale, out=out, stream=stream)
    torch.cuda.synchronize()
    got = buf.cpu().numpy()
    if guard_rows:
        guard = got[batch * seq:]
        assert (guard == (90 if dt == torch.int8 else np.float32(1234.5))).all(), "bytes after out were written"
    return got[:batch * seq]


@pytest.mark.parametrize("batch,seq,heads,pad,scale", [
    (1, 1, 1, 0, 0.05), (2, 5, 2, 16, 0.05), (1, 64, 12, 0, 0.05), (3, 65, 4, 0, 0.08),
    (2, 130, 3, 48, 0.02), (1, 512, 2, 0, 0.05), (2, 384, 12, 0, 0.12), (1, 128, 2, 0, 0.05),
    (1, 129, 2, 0, 0.05), (2, 257, 1, 16, 0.05), (1, 383, 2, 0, 0.1), (1, 511, 1, 0, 0.05)])
def test_attention_f32_parity(bsg, batch, seq, heads, pad, scale):
    rng = np.random.default_rng(7000 + 7 * seq + heads)
    qkv = draw_qkv(rng, batch, seq, heads, pad)
    got = run_device(bsg, qkv, batch, seq, heads, scale, guard_rows=2)
    want = oracle.attention_f64(qkv, scale, batch, seq, heads=heads, head_dim=HD, threads=8)
    tol = bound(qkv, scale, batch, seq, heads)
    err = np.abs(got.astype(np.float64) - want)
    assert err.max() <= tol, f"max err {err.max():.3g} > bound {tol:.3g}"


def test_attention_i8_full_layer_shape(bsg):
    """The encoder layer's shape: 8 sequences x 384 tokens, 12 heads; int8
    context with the scale a calibration would pick (max |ctx| / 127)."""
    import torch
    batch, seq, heads, scale = 8, 384, 12, 0.05
    rng = np.random.default_rng(7100)
    qkv = draw_qkv(rng, batch, seq, heads)
    want = oracle.attention_f64(qkv, scale, batch, seq, heads=heads, head_dim=HD, threads=16)
    out_scale = float(np.float32(np.abs(want).max()) / np.float32(127.0))
    inv = float(np.float32(1.0) / np.float32(out_scale))
    got = run_device(bsg, qkv, batch, seq, heads, scale, bsg.OUT_I8, out_scale, guard_rows=1)
    tol = bound(qkv, scale, batch, seq, heads)
    t = want * inv
    ref = np.clip(np.rint(t), -128, 127).astype(np.int64)
    g = got.astype(np.int64)
    diff = g != ref
    near = np.abs(np.abs(t - np.floor(t)) - 0.5) <= tol * inv + 1e-6
    assert not (diff & ~(near & (np.abs(g - ref) == 1))).any(), \
        f"{int((diff & ~near).sum())} int8 values differ away from a rounding boundary"
    assert int(diff.sum()) <= g.size // 100
    # the fp32 path on the same input, from a side stream
    s = torch.cuda.Stream()
    got32 = run_device(bsg, qkv, batch, seq, heads, scale, stream=s)
    assert np.abs(got32.astype(np.float64) - want).max() <= tol


def test_attention_special_cases(bsg):
    rng = np.random.default_rng(7200)
    seq, heads = 100, 2
    d = heads * HD
    v = rng.integers(-127, 128, size=(seq, d))
    # one dominant key: every context row is that key's value times the scale (0.5), up to the
    # rounding of that key's weight (2^t with t the residual of fl(d c2): within an ulp of 1)
    k = np.full((seq, d), -127)
    k[37] = 127
    qkv = np.concatenate([np.full((seq, d), 127), k, v], axis=1).astype(np.int8)
    got = run_device(bsg, qkv, 1, seq, heads, 0.5)
    np.testing.assert_allclose(got, np.broadcast_to((v[37] * 0.5).astype(np.float32), (seq, d)), rtol=2.0 ** -21,
                               atol=0.0)
    # zero queries: every key weighs the same, the context is the mean value
    qkv = np.concatenate([np.zeros((seq, d)), rng.integers(-127, 128, size=(seq, d)), v], axis=1).astype(np.int8)
    got = run_device(bsg, qkv, 1, seq, heads, 0.05)
    want = oracle.attention_f64(qkv, 0.05, 1, seq, heads=heads, head_dim=HD)
    assert np.allclose(want, np.broadcast_to(v.mean(axis=0) * np.float64(np.float32(0.05)), (seq, d)), atol=1e-12)
    assert np.abs(got - want).max() <= bound(qkv, 0.05, 1, seq, heads)


def test_attention_checks_on_device(bsg):
    import torch
    qkv = torch.zeros((2 * 8, 3 * 64), dtype=torch.int8, device="cuda")
    with pytest.raises(ValueError):
        bsg.attention(qkv, 2, 9, 1, 0.05)                       # rows != batch * seq
    with pytest.raises(ValueError):
        bsg.attention(qkv[:, :100], 2, 8, 1, 0.05)              # rows too short for q | k | v
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.attention(qkv, 2, 8, 1, -1.0)
    assert e.value.code == bsg.ERR_INVALID
    out = bsg.attention(qkv, 2, 8, 1, 0.05)                    # all zero: the context is 0
    torch.cuda.synchronize()
    assert out.abs().max().item() == 0.0


@pytest.mark.parametrize("order", ["rising", "falling"])
def test_attention_running_maximum(bsg, order):
    """Scores that rise from key to key (by ~13 log2 units every 64 keys)
    move the reference maximum every block or two (the context and the sum
    are rescaled each time); falling scores never do.  Both against the
    oracle."""
    seq, heads, scale = 500, 2, 0.02
    d = heads * HD
    rng = np.random.default_rng(7300)
    ramp = np.rint(np.linspace(-127, 127, seq)).astype(np.int64)
    if order == "falling":
        ramp = ramp[::-1]
    k = np.repeat(ramp[:, None], d, axis=1)
    qkv = np.concatenate([np.full((seq, d), 90), k, rng.integers(-127, 128, size=(seq, d))], axis=1).astype(np.int8)
    got = run_device(bsg, qkv, 1, seq, heads, scale)
    want = oracle.attention_f64(qkv, scale, 1, seq, heads=heads, head_dim=HD)
    assert np.abs(got.astype(np.float64) - want).max() <= bound(qkv, scale, 1, seq, heads)


def test_attention_every_block_boundary(bsg):
    """Sequence lengths on both sides of every multiple of the 64-key block
    and of the 32 keys each warp of a pair takes (the padded tail of the
    keys and values, the last block's masked keys, a warp with no key, one
    to eight blocks), one head each."""
    rng = np.random.default_rng(7400)
    for seq in [1, 2, 31, 32, 33, 63, 64, 65, 95, 96, 97, 127, 128, 129, 159, 160, 161, 191, 192, 193, 255, 256,
                257, 319, 320, 321, 383, 384, 385, 447, 448, 449, 480, 500, 511, 512]:
        qkv = draw_qkv(rng, 1, seq, 1)
        got = run_device(bsg, qkv, 1, seq, 1, 0.05, guard_rows=1)
        want = oracle.attention_f64(qkv, 0.05, 1, seq, heads=1, head_dim=HD)
        assert np.abs(got.astype(np.float64) - want).max() <= bound(qkv, 0.05, 1, seq, 1), seq
    assert bsg.bsgemm_attention_status() == 0


def test_attention_act_ready_back_to_back(bsg):
    """Independent batches launched back to back on one stream with
    ACT_READY, as the bench times the kernel: each launch may read its qkv
    while the previous launch still runs (programmatic dependent launch) and
    writes its output only after it; every output matches the oracle."""
    import torch
    batch, seq, heads, scale = 2, 384, 12, 0.05
    rng = np.random.default_rng(7500)
    qkvs = [draw_qkv(rng, batch, seq, heads) for _ in range(4)]
    dev = [torch.from_numpy(q).cuda() for q in qkvs]
    outs = [torch.full((batch * seq, heads * HD), 1234.5, dtype=torch.float32, device="cuda") for _ in qkvs]
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    for rep in range(3):
        for q, o in zip(dev, outs):
            bsg.attention(q, batch, seq, heads, scale, bsg.OUT_F32, out=o, stream=s, flags=bsg.ACT_READY)
    torch.cuda.synchronize()
    for q, o in zip(qkvs, outs):
        want = oracle.attention_f64(q, scale, batch, seq, heads=heads, head_dim=HD, threads=8)
        assert np.abs(o.cpu().numpy().astype(np.float64) - want).max() <= bound(q, scale, batch, seq, heads)
    assert bsg.bsgemm_attention_status() == 0
