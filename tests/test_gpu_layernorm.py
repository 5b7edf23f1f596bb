"""Residual add in the linear's epilogue (BSGEMM_OUT_F32_RESID) and the
row-wise LayerNorm kernel (bsgemm_layernorm), against the oracle's
linear_resid (the same fp32 operations: exact) and layernorm (fp64: a
tolerance, and int8 decisions exact except next to a rounding boundary)."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def bsg():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


def make_linear(bsg, wt, n_out=None):
    w = oracle.weight_dense(wt)
    if n_out is not None:
        w = np.ascontiguousarray(w[:n_out])
        return bsg.SparseInt8Linear.from_dense(w, wt.scales[:n_out].copy(), wt.bias[:n_out].copy()), w
    return bsg.SparseInt8Linear(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias), w


def check_f32_close(got, want, what=""):
    err = np.abs(got.astype(np.float64) - want)
    bad = ~((err <= 1e-5) | (err <= 1e-6 * np.abs(want)))
    assert not bad.any(), f"{what}: {bad.sum()} values out of tolerance, max abs err {err.max():.3g}"


def check_i8_near(got, want_f64, inv, what=""):
    """q must equal rne(want * inv) saturated, except where want * inv lies
    within 1e-3 of a rounding boundary (the fp32 kernel and the fp64
    reference may then fall on either side), where a neighbour is allowed."""
    t = want_f64 * np.float64(inv)
    ref = np.clip(np.rint(t), -128, 127).astype(np.int64)
    g = got.astype(np.int64)
    diff = g != ref
    near = np.abs(np.abs(t - np.floor(t)) - 0.5) < 1e-3
    ok = ~diff | (near & (np.abs(g - ref) == 1))
    assert ok.all(), f"{what}: {int((~ok).sum())} int8 values differ away from a rounding boundary"
    return int(diff.sum())


@pytest.mark.parametrize("n_out,k_in,m,path", [(768, 768, 200, None), (768, 3072, 130, False), (96, 1001, 70, None),
                                               (6, 768, 65, None), (770, 512, 64, False)])
def test_residual_epilogue_is_exact(bsg, n_out, k_in, m, path):
    import torch
    rng = synth.rng_for(6400 + n_out + k_in)
    n4 = -(-n_out // 4) * 4
    wt = synth.draw_weight(rng, n4, k_in, 0.85)
    lin, w = make_linear(bsg, wt, n_out if n_out != n4 else None)
    x = synth.draw_x(rng, m, k_in, "u127")
    r = synth.draw_x(rng, m, n_out, "u127")
    want = oracle.linear_resid(x, w, wt.scales[:n_out], wt.bias[:n_out], r, 0.0375)
    out = torch.empty((m, n_out), dtype=torch.float32, device="cuda")
    lin.run(torch.from_numpy(x).cuda(), out, bsg.OUT_F32_RESID, workspace=path,
            residual=torch.from_numpy(r).cuda(), residual_scale=0.0375)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    assert np.array_equal(got, want), f"{int((got != want).sum())} of {got.size} differ"
    lin.close()


@pytest.mark.parametrize("m,n", [(300, 768), (7, 1), (33, 3), (64, 1000), (1, 3072)])
def test_layernorm_f32_and_i8(bsg, m, n):
    import torch
    rng = np.random.default_rng(6500 + m + n)
    z = (rng.normal(size=(m, n)) * rng.uniform(0.5, 20, size=(m, 1)) + rng.normal(size=(m, 1)) * 5).astype(np.float32)
    g = rng.normal(1.0, 0.3, size=n).astype(np.float32)
    b = rng.normal(0.0, 0.5, size=n).astype(np.float32)
    want = oracle.layernorm(z, g, b, 1e-5)
    zd, gd, bd = (torch.from_numpy(a).cuda() for a in (z, g, b))
    got = bsg.layernorm(zd, gd, bd, 1e-5).cpu().numpy()
    if n > 1:
        check_f32_close(got, want, "f32")
    else:  # one channel: the row normalises to 0, the output is beta
        assert np.array_equal(got[:, 0], np.full(m, b[0], np.float32))
    q = bsg.layernorm(zd, gd, bd, 1e-5, bsg.OUT_I8, 0.025).cpu().numpy()
    check_i8_near(q, want, np.float32(1.0) / np.float32(0.025), "i8")


def test_encoder_sublayer_output_projection(bsg):
    """The attention output projection of an encoder layer with its residual
    add and LayerNorm: int8 context in, int8 normalised hidden state out
    (M = 8 x 384 tokens, 768 -> 768 at 80%)."""
    import torch
    rng = synth.rng_for(6600)
    wt = synth.draw_weight(rng, 768, 768, 0.8)
    lin, w = make_linear(bsg, wt)
    m = 3072
    ctx = synth.draw_x(rng, m, 768, "u127")
    res = synth.draw_x(rng, m, 768, "u127")
    g = rng.normal(1.0, 0.1, size=768).astype(np.float32)
    b = rng.normal(0.0, 0.1, size=768).astype(np.float32)
    z = torch.empty((m, 768), dtype=torch.float32, device="cuda")
    lin.run(torch.from_numpy(ctx).cuda(), z, bsg.OUT_F32_RESID, residual=torch.from_numpy(res).cuda(),
            residual_scale=0.02)
    q = bsg.layernorm(z, torch.from_numpy(g).cuda(), torch.from_numpy(b).cuda(), 1e-12, bsg.OUT_I8, 0.03)
    torch.cuda.synchronize()
    z_ref = oracle.linear_resid(ctx, w, wt.scales, wt.bias, res, 0.02, threads=8)
    assert np.array_equal(z.cpu().numpy(), z_ref)
    want = oracle.layernorm(z_ref, g, b, 1e-12)
    flips = check_i8_near(q.cpu().numpy(), want, np.float32(1.0) / np.float32(0.03), "sublayer")
    assert flips <= m * 768 // 10000  # boundary cases are rare
    lin.close()


def test_argument_checks(bsg):
    import torch
    rng = synth.rng_for(6700)
    wt = synth.draw_weight(rng, 16, 64, 0.5)
    lin, _ = make_linear(bsg, wt)
    x = torch.zeros((8, 64), dtype=torch.int8, device="cuda")
    out = torch.empty((8, 16), dtype=torch.float32, device="cuda")
    with pytest.raises(bsg.BsgemmError) as e:  # no residual
        bsg.bsgemm_run(lin._h, x.data_ptr(), 8, out.data_ptr(), bsg.OUT_F32_RESID, 1.0, 0)
    assert e.value.code == bsg.ERR_INVALID
    r = torch.zeros((8 * 16 + 4,), dtype=torch.int8, device="cuda")
    with pytest.raises(bsg.BsgemmError):  # misaligned residual
        bsg.bsgemm_run(lin._h, x.data_ptr(), 8, out.data_ptr(), bsg.OUT_F32_RESID, 1.0, 0, 0, r.data_ptr() + 1)
    z = torch.zeros((8, 16), dtype=torch.float32, device="cuda")
    g = torch.ones(16, dtype=torch.float32, device="cuda")
    with pytest.raises(bsg.BsgemmError):  # int32 output
        bsg.bsgemm_layernorm(z.data_ptr(), 8, 16, g.data_ptr(), g.data_ptr(), 1e-5, out.data_ptr(), bsg.OUT_I32)
    with pytest.raises(bsg.BsgemmError):  # eps < 0
        bsg.bsgemm_layernorm(z.data_ptr(), 8, 16, g.data_ptr(), g.data_ptr(), -1.0, out.data_ptr(), bsg.OUT_F32)
    bsg.bsgemm_layernorm(0, 0, 16, 0, 0, 1e-5, 0, bsg.OUT_F32)  # M = 0: nothing to do
    lin.close()
