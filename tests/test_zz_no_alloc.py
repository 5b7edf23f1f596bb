"""bsgemm_run_static, the entry point that allocates nothing (its token
tiles go to a fixed device array held by the library), against
bsgemm_run_ws on the same inputs: two calls in a row, with different token
counts, kinds and weights, so that the second call cannot lean on what the
first left in the scratch.  Named to run last; it also passes alone."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

DTYPES = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
          synth.I8: torch.int8, synth.I8_GELU: torch.int8}


@pytest.fixture(scope="module")
def bsg():
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


def _layer(bsg, n, k, sparsity, seed):
    rng = synth.rng_for(seed)
    wt = synth.draw_weight(rng, n, k, sparsity)
    return bsg.SparseInt8Linear(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias), rng


def _both(bsg, lin, x, kind, out_scale):
    """(bsgemm_run_static output, bsgemm_run_ws output) on one stream."""
    s = torch.cuda.current_stream().cuda_stream
    m = x.shape[0]
    got = torch.full((m, lin.n_out), 7, dtype=DTYPES[kind], device="cuda")
    want = torch.full((m, lin.n_out), -7, dtype=DTYPES[kind], device="cuda")
    bsg.bsgemm_run_static(lin._h, x.data_ptr(), m, got.data_ptr(), kind, out_scale, s)
    ws_bytes = lin.workspace_bytes(m)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, want.data_ptr(), kind, out_scale, ws.data_ptr(), ws_bytes, s)
    torch.cuda.synchronize()
    return got.cpu().numpy(), want.cpu().numpy()


def test_two_calls_in_a_row_match_run_ws(bsg):
    # 1st: FFN2-shaped (K = 3072, 64-token tiles), ragged M; 2nd: a 768-wide
    # layer (128-token tiles) with fewer tokens, another kind and weight.
    calls = [(768, 3072, 0.90, 1000, "u0_127", synth.I8, 0.05),
             (768, 768, 0.80, 333, "u127", synth.F32_GELU, 1.0)]
    for i, (n, k, sp, m, dist, kind, out_scale) in enumerate(calls):
        lin, rng = _layer(bsg, n, k, sp, 4200 + i)
        x = torch.from_numpy(synth.draw_x(rng, m, k, dist)).cuda()
        got, want = _both(bsg, lin, x, kind, out_scale)
        assert np.array_equal(got, want), f"call {i + 1}: {np.sum(got != want)} elements differ"
        assert bsg.bsgemm_device_status(lin._h) == 0
        lin.close()


def test_largest_m_fits_and_one_tile_more_is_rejected(bsg):
    lin, rng = _layer(bsg, 64, 3072, 0.90, 4300)
    tile = lin.info["tile_m"]
    per_tile = lin.workspace_bytes(tile)
    m_max = bsg.STATIC_SCRATCH_BYTES // per_tile * tile
    assert lin.workspace_bytes(m_max) <= bsg.STATIC_SCRATCH_BYTES < lin.workspace_bytes(m_max + 1)
    x = torch.from_numpy(synth.draw_x(rng, m_max, 3072, "u127")).cuda()
    got, want = _both(bsg, lin, x, synth.I32, 1.0)
    assert np.array_equal(got, want)
    out = torch.empty((m_max + 1, 64), dtype=torch.int32, device="cuda")
    xl = torch.zeros((m_max + 1, 3072), dtype=torch.int8, device="cuda")
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.bsgemm_run_static(lin._h, xl.data_ptr(), m_max + 1, out.data_ptr(), synth.I32, 1.0,
                              torch.cuda.current_stream().cuda_stream)
    assert e.value.code == bsg.ERR_INVALID and "static scratch" in str(e.value)
    lin.close()
