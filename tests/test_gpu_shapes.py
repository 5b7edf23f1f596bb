"""Other block shapes through the layer kernel, every element against the
oracle's linear on the oracle's own decompression of the same arrays
(integer outputs bit for bit, fp32 within 1e-4 abs or 1e-5 rel):
  * weights sparse in 1 x 4 blocks (one output row x 4 input columns), run
    natively by the kernel's 1 x 4 form (bsgemm_create_1x4): every kind but
    the residual, both staging paths, ragged K (relayout path), K = 4,
    N not a multiple of 4, rows without blocks, one token;
  * 2:4-sparse weights (bsgemm_create_2to4): N and K multiples of 128 on
    the sparse tensor cores (tcgen05.mma.sp, exact fp32 chunks of 2048
    columns added in int32), other shapes as the 4 x 1 blocks that hold
    them;
  * 4 x 1 block weights run dense over K on the tensor cores
    (bsgemm_create_tc: tcgen05.mma kind::f16, exact fp32 chunks of 1024
    columns added in int32)."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

KINDS = (synth.I32, synth.F32, synth.F32_GELU, synth.I8, synth.I8_GELU)


@pytest.fixture(scope="module")
def bsg():
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


def check(got: np.ndarray, want: np.ndarray, kind: int, what: str = ""):
    assert got.shape == want.shape, what
    if kind in (synth.F32, synth.F32_GELU):
        err = np.abs(got.astype(np.float64) - want)
        bad = ~((err <= 1e-4) | (err <= 1e-5 * np.abs(want)))
        assert not bad.any(), f"{what}: {bad.sum()} fp32 elements out of tolerance, max abs err {err.max():.3g}"
    else:
        diff = got != want
        assert not diff.any(), f"{what}: {diff.sum()} elements differ"


def gpu_run(lin, x: np.ndarray, kind: int, out_scale: float, workspace=None) -> np.ndarray:
    xd = torch.from_numpy(x).cuda()
    dtype = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
             synth.I8: torch.int8, synth.I8_GELU: torch.int8}[kind]
    out = torch.empty((x.shape[0], lin.n_out), dtype=dtype, device="cuda")
    lin.run(xd, out, kind, out_scale, workspace=workspace)
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("n_out,k_in,m,sparsity", [(96, 768, 130, 0.9), (30, 200, 70, 0.5), (768, 3072, 64, 0.9),
                                                    (7, 4, 65, 0.0), (130, 100, 1, 0.6), (64, 3072, 200, 0.97)])
def test_blocks_1x4_through_the_layer(bsg, n_out, k_in, m, sparsity):
    rng = synth.rng_for(8000 + n_out + k_in)
    wt = synth.draw_weight_1x4(rng, n_out, k_in, sparsity)
    w = oracle.bsr1x4_to_dense(n_out, k_in, wt.indptr, wt.colgrp, wt.values)
    lin = bsg.SparseInt8Linear.from_blocks_1x4(n_out, k_in, wt.indptr, wt.colgrp, wt.values, wt.scales, wt.bias)
    assert (lin.n_out, lin.k_in) == (n_out, k_in)
    x = synth.draw_x(rng, m, k_in, "u127")
    for kind in KINDS:
        want = oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05, threads=8)
        for path in (None, False):
            check(gpu_run(lin, x, kind, 0.05, workspace=path), want, kind, f"1x4 kind {kind} path {path}")
    lin.close()


@pytest.mark.parametrize("n_out,k_in,m", [(64, 768, 100), (30, 200, 70), (768, 3072, 64)])
def test_2to4_through_the_layer(bsg, n_out, k_in, m):
    rng = synth.rng_for(8100 + n_out + k_in)
    wt = synth.draw_weight_2to4(rng, n_out, k_in)
    w = oracle.sparse2to4_to_dense(wt.values, wt.idx)
    lin = bsg.SparseInt8Linear.from_2to4(wt.values, wt.idx, wt.scales, wt.bias)
    assert (lin.n_out, lin.k_in) == (n_out, k_in)
    x = synth.draw_x(rng, m, k_in, "n30")
    for kind in KINDS:
        want = oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05, threads=8)
        check(gpu_run(lin, x, kind, 0.05), want, kind, f"2:4 kind {kind}")
    lin.close()


@pytest.mark.parametrize("n_out,k_in,m", [(128, 128, 1), (256, 2048, 130), (768, 3072, 300), (128, 2176, 64),
                                          (384, 1024, 257)])
def test_2to4_on_the_sparse_tensor_cores(bsg, n_out, k_in, m):
    """Every kind, ragged token tiles, one and two exact accumulator chunks
    (a chunk holds 2048 columns), a chunk boundary at the last stage."""
    rng = synth.rng_for(8200 + n_out + k_in + m)
    wt = synth.draw_weight_2to4(rng, n_out, k_in)
    w = oracle.sparse2to4_to_dense(wt.values, wt.idx)
    lin = bsg.SparseInt8Linear.from_2to4(wt.values, wt.idx, wt.scales, wt.bias)
    x = synth.draw_x(rng, m, k_in, "u127")
    for kind in KINDS:
        want = oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05, threads=8)
        check(gpu_run(lin, x, kind, 0.05), want, kind, f"2:4 tensor cores kind {kind}")
    lin.close()


def test_2to4_tensor_cores_at_the_fp32_limit(bsg):
    """Every stored value -128 and every activation -128: each product is
    2^14 and a chunk's 1024 of them sum to exactly 2^24, the largest partial
    sum the exact fp32 accumulation has to hold; then mixed extremes."""
    n_out, k_in, m = 128, 3072, 70
    rng = synth.rng_for(8300)
    wt = synth.draw_weight_2to4(rng, n_out, k_in)
    values = np.full_like(wt.values, -128)
    w = oracle.sparse2to4_to_dense(values, wt.idx)
    lin = bsg.SparseInt8Linear.from_2to4(values, wt.idx, wt.scales, wt.bias)
    for x in (np.full((m, k_in), -128, dtype=np.int8),
              rng.choice(np.array([-128, 127], dtype=np.int8), size=(m, k_in))):
        want = oracle.linear(x, w, wt.scales, wt.bias, synth.I32, threads=8)
        check(gpu_run(lin, x, synth.I32, 1.0), want, synth.I32, "2:4 extremes")
    lin.close()


@pytest.mark.parametrize("n_out,k_in,m,sparsity", [(128, 128, 1, 0.0), (256, 2048, 130, 0.9), (768, 3072, 300, 0.9),
                                                    (384, 1152, 257, 0.5), (256, 2944, 64, 0.8), (128, 256, 70, 1.0)])
def test_dense_over_k_on_the_tensor_cores(bsg, n_out, k_in, m, sparsity):
    """bsgemm_create_tc: every kind, ragged token tiles, one to three exact
    accumulator chunks (a chunk holds 1024 columns; K = 1152 ends with a
    chunk of one stage, K = 2944 with one of seven), a weight without
    stored blocks; then an act
    pointer off the 16-byte boundary, which the block-sparse kernel takes."""
    rng = synth.rng_for(8400 + n_out + k_in + m)
    wt = synth.draw_weight(rng, n_out, k_in, sparsity)
    w = oracle.bsr_to_dense(n_out, k_in, wt.indptr, wt.colidx, wt.values)
    lin = bsg.SparseInt8Linear(n_out, k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias, tensor_cores=True)
    assert lin.info["nnzb"] == wt.nnzb
    assert lin.info["device_bytes"] >= 2 * n_out * k_in  # the f16 image of the dense form
    x = synth.draw_x(rng, m, k_in, "u127")
    for kind in KINDS:
        want = oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05, threads=8)
        check(gpu_run(lin, x, kind, 0.05), want, kind, f"dense tensor cores kind {kind}")
    buf = torch.empty(m * k_in + 4, dtype=torch.int8, device="cuda")
    xd = buf[4:].view(m, k_in)
    xd.copy_(torch.from_numpy(x))
    out = torch.empty((m, n_out), dtype=torch.int32, device="cuda")
    lin.run(xd, out, synth.I32, 1.0)
    torch.cuda.synchronize()
    check(out.cpu().numpy(), oracle.linear(x, w, wt.scales, wt.bias, synth.I32, threads=8), synth.I32, "offset act")
    lin.close()


def test_dense_tensor_cores_at_the_fp32_limit(bsg):
    """Every weight -128 and every activation -128: each product is 2^14 and
    a chunk's 1024 of them sum to exactly 2^24, the largest partial sum the
    exact fp32 accumulation has to hold (three chunks); then mixed
    extremes."""
    n_out, k_in, m = 128, 3072, 70
    rng = synth.rng_for(8500)
    wt = synth.draw_weight(rng, n_out, k_in, 0.0)
    values = np.full_like(wt.values, -128)
    w = oracle.bsr_to_dense(n_out, k_in, wt.indptr, wt.colidx, values)
    lin = bsg.SparseInt8Linear(n_out, k_in, wt.indptr, wt.colidx, values, wt.scales, wt.bias, tensor_cores=True)
    for x in (np.full((m, k_in), -128, dtype=np.int8),
              rng.choice(np.array([-128, 127], dtype=np.int8), size=(m, k_in))):
        want = oracle.linear(x, w, wt.scales, wt.bias, synth.I32, threads=8)
        check(gpu_run(lin, x, synth.I32, 1.0), want, synth.I32, "dense extremes")
    lin.close()


def test_blocks_1x4_empty_rows_and_residual_rejected(bsg):
    rng = synth.rng_for(8050)
    n_out, k_in = 40, 256
    wt = synth.draw_weight_1x4(rng, n_out, k_in, 0.8)
    # rows 0, 5 and 39 without blocks
    keep = np.ones(wt.indptr[-1], bool)
    for r in (0, 5, 39):
        keep[wt.indptr[r]:wt.indptr[r + 1]] = False
    counts = np.diff(wt.indptr).copy()
    for r in (0, 5, 39):
        counts[r] = 0
    indptr = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    colgrp, values = wt.colgrp[keep], wt.values[keep]
    w = oracle.bsr1x4_to_dense(n_out, k_in, indptr, colgrp, values)
    lin = bsg.SparseInt8Linear.from_blocks_1x4(n_out, k_in, indptr, colgrp, values, wt.scales, wt.bias)
    assert lin.info["nnzb"] == int(indptr[-1])
    x = synth.draw_x(rng, 99, k_in, "u127")
    for kind in (synth.I32, synth.F32, synth.I8):
        check(gpu_run(lin, x, kind, 0.05), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05), kind)
    out = torch.empty((99, n_out), dtype=torch.float32, device="cuda")
    r8 = torch.zeros((99, n_out), dtype=torch.int8, device="cuda")
    with pytest.raises(bsg.BsgemmError) as e:
        lin.run(torch.from_numpy(x).cuda(), out, bsg.OUT_F32_RESID, residual=r8, residual_scale=0.1)
    assert e.value.code == bsg.ERR_UNSUPPORTED
    lin.close()
