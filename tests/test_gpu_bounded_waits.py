"""Failure detection without a GPU fault: every wait in device code is
bounded, and a wait that gives up leaves an error the host reads.

The test hooks (bsgemm_set_test_hooks) make the waits run out on purpose:
the layer kernel issues no tile copy (so no copy is in flight when its CTAs
leave) and polls its copy barriers 64 times; the pruning kernel's CTA 0
leaves before the first grid barrier, which the other CTAs give up after
4096 polls; the attention kernel issues no tensor-core MMA and polls the
mbarriers its MMAs would complete 64 times.  Each call must return, report the failure, and leave the
context usable: a normal run right after matches the oracle.
"""
import os

import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def bsg():
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


@pytest.fixture
def hooks(bsg):
    """Clears the hooks after the test, whatever happens."""
    yield bsg.bsgemm_set_test_hooks
    bsg.bsgemm_set_test_hooks(0)


def _linear(bsg, n, k, sparsity, seed):
    rng = synth.rng_for(seed)
    wt = synth.draw_weight(rng, n, k, sparsity)
    lin = bsg.SparseInt8Linear(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias)
    return lin, wt, rng


@pytest.mark.parametrize("workspace", [None, False], ids=["ws", "nows"])
def test_tile_copy_wait_gives_up_and_reports_timeout(bsg, hooks, workspace):
    # K = 3072 with aligned x: the one-kernel path whose CTAs wait for the
    # tensor copies of their token tile
    lin, wt, rng = _linear(bsg, 768, 3072, 0.90, 6400)
    x = synth.draw_x(rng, 300, 3072, "u0_127")
    xd = torch.from_numpy(x).cuda()
    out = torch.zeros((300, 768), dtype=torch.int8, device="cuda")
    assert bsg.bsgemm_device_status(lin._h) == 0
    assert hooks(bsg.TEST_SKIP_TILE_COPY) == 0
    lin.run(xd, out, synth.I8, 0.05, workspace=workspace)  # returns: the waits are bounded
    torch.cuda.synchronize()
    assert hooks(0) == bsg.TEST_SKIP_TILE_COPY
    assert bsg.bsgemm_device_status(lin._h, clear=True) == bsg.STATUS_TIMEOUT
    assert bsg.bsgemm_device_status(lin._h) == 0
    # the context is fine: the same run without the hook is exact
    lin.run(xd, out, synth.I8, 0.05, workspace=workspace)
    torch.cuda.synchronize()
    want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, synth.I8, 0.05,
                         threads=os.cpu_count() or 8)
    assert np.array_equal(out.cpu().numpy(), want)
    assert bsg.bsgemm_device_status(lin._h) == 0
    lin.close()


def test_relaid_tile_copy_wait_gives_up(bsg, hooks):
    # K = 1000: relayout kernel + one bulk copy of each tile, whose wait runs out
    lin, wt, rng = _linear(bsg, 256, 1000, 0.80, 6401)
    x = synth.draw_x(rng, 200, 1000, "u127")
    xd = torch.from_numpy(x).cuda()
    out = torch.zeros((200, 256), dtype=torch.int32, device="cuda")
    hooks(bsg.TEST_SKIP_TILE_COPY)
    lin.run(xd, out, synth.I32, 1.0)
    torch.cuda.synchronize()
    hooks(0)
    assert bsg.bsgemm_device_status(lin._h, clear=True) == bsg.STATUS_TIMEOUT
    lin.run(xd, out, synth.I32, 1.0)
    torch.cuda.synchronize()
    want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, synth.I32, threads=os.cpu_count() or 8)
    assert np.array_equal(out.cpu().numpy(), want)
    lin.close()


def test_prune_grid_barrier_gives_up_and_the_call_fails(bsg, hooks):
    rng = synth.rng_for(6402)
    w = rng.normal(0.0, 0.02, size=(768, 3072)).astype(np.float32)
    wd = torch.from_numpy(w).cuda()
    hooks(bsg.TEST_STALL_PRUNE_CTA)
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.block_prune(wd, 0.9)
    hooks(0)
    assert e.value.code == bsg.ERR_CUDA
    # every CTA left: the next call on the same device works and is exact
    keep = bsg.block_prune(wd, 0.9)
    torch.cuda.synchronize()
    assert np.array_equal(keep.cpu().numpy().astype(bool), oracle.block_prune(w, 0.9))


def test_attention_mma_wait_gives_up_and_reports_timeout(bsg, hooks):
    from test_gpu_attention import HD, bound, draw_qkv
    batch, seq, heads, scale = 2, 300, 3, 0.05
    qkv = draw_qkv(np.random.default_rng(6403), batch, seq, heads)
    qd = torch.from_numpy(qkv).cuda()
    out = torch.zeros((batch * seq, heads * HD), dtype=torch.float32, device="cuda")
    assert bsg.bsgemm_attention_status(clear=True) in (0, bsg.STATUS_TIMEOUT)
    hooks(bsg.TEST_ATTN_SKIP_MMA)
    bsg.attention(qd, batch, seq, heads, scale, out=out)  # returns: the waits are bounded
    torch.cuda.synchronize()
    hooks(0)
    assert bsg.bsgemm_attention_status(clear=True) == bsg.STATUS_TIMEOUT
    assert bsg.bsgemm_attention_status() == 0
    bsg.attention(qd, batch, seq, heads, scale, out=out)
    torch.cuda.synchronize()
    want = oracle.attention_f64(qkv, scale, batch, seq, heads=heads, head_dim=HD, threads=2)
    assert np.abs(out.cpu().numpy().astype(np.float64) - want).max() <= bound(qkv, scale, batch, seq, heads)
    assert bsg.bsgemm_attention_status() == 0
