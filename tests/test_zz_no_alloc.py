"""bsgemm_run_static, the entry point that allocates nothing.

Some callers cannot allocate device memory while they run: a serving loop
whose memory is fixed once at start-up, code that runs inside a host
callback or another runtime's allocator, or a caller with no CUDA allocator
of its own to hand.  For them bsgemm_run_static keeps the token tiles it
needs in a fixed device array the library holds.

Every call here takes the scratch path (K not a multiple of 16, or an
activation pointer that is not 16-byte aligned), so the tiles really go
through that array, and every element is checked against the CPU oracle
(and against bsgemm_run_ws on the same inputs).  The calls come back to
back with different shapes, the larger one first, so that stale tiles left
by one call would show in the next.  Named to run last; it also passes
alone in a fresh process.
"""
import os

import numpy as np
import pytest

import oracle
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
    return bsg.SparseInt8Linear(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias), wt, rng


def _device_act(x: np.ndarray, offset: int):
    """x on the device at `offset` bytes past a 256-byte aligned base: (keep-alive
    buffer, pointer)."""
    buf = torch.zeros(x.size + 256, dtype=torch.int8, device="cuda")
    buf[offset:offset + x.size] = torch.from_numpy(x.reshape(-1)).cuda()
    return buf, buf.data_ptr() + offset


def _run_both(bsg, lin, ptr, m, kind, out_scale):
    """(bsgemm_run_static output, bsgemm_run_ws output) on one stream."""
    s = torch.cuda.current_stream().cuda_stream
    got = torch.full((m, lin.n_out), 7, dtype=DTYPES[kind], device="cuda")
    ref = torch.full((m, lin.n_out), -7, dtype=DTYPES[kind], device="cuda")
    bsg.bsgemm_run_static(lin._h, ptr, m, got.data_ptr(), kind, out_scale, s)
    ws_bytes = lin.workspace_bytes(m)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    bsg.bsgemm_run_ws(lin._h, ptr, m, ref.data_ptr(), kind, out_scale, ws.data_ptr(), ws_bytes, s)
    torch.cuda.synchronize()
    return got.cpu().numpy(), ref.cpu().numpy()


def _check(got, want, kind, what):
    if kind in (synth.F32, synth.F32_GELU):
        err = np.abs(got.astype(np.float64) - want)
        bad = ~((err <= 1e-4) | (err <= 1e-5 * np.abs(want)))
        assert not bad.any(), f"{what}: {bad.sum()} fp32 elements out of tolerance (max abs err {err.max():.3g})"
    else:
        diff = got != want
        assert not diff.any(), f"{what}: {diff.sum()} elements differ"


def test_calls_in_a_row_through_the_scratch_match_the_oracle(bsg):
    # (n_out, k_in, sparsity, M, x_dist, kind, out_scale, act offset):
    # K = 1001 (not a multiple of 16), then K = 3072 from an act pointer
    # 4 bytes past alignment, then K = 1001 again with fewer tokens.
    calls = [(768, 1001, 0.90, 1500, "u127", synth.I8, 0.05, 0),
             (256, 3072, 0.90, 333, "u0_127", synth.F32_GELU, 1.0, 4),
             (768, 1001, 0.90, 130, "n30", synth.I32, 1.0, 0)]
    lins = {}
    for i, (n, k, sp, m, dist, kind, out_scale, offset) in enumerate(calls):
        key = (n, k, sp)
        if key not in lins:
            lins[key] = _layer(bsg, n, k, sp, 4200 + i)
        lin, wt, rng = lins[key]
        x = synth.draw_x(rng, m, k, dist)
        _, ptr = keep = _device_act(x, offset)
        got, ref = _run_both(bsg, lin, ptr, m, kind, out_scale)
        want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, kind, out_scale=out_scale,
                             threads=os.cpu_count() or 8)
        _check(got, want, kind, f"call {i + 1} against the oracle")
        _check(ref, want, kind, f"call {i + 1}, bsgemm_run_ws against the oracle")
        assert np.array_equal(got, ref), f"call {i + 1}: bsgemm_run_static and bsgemm_run_ws differ"
        assert bsg.bsgemm_device_status(lin._h) == 0
        del keep
    for lin, _, _ in lins.values():
        lin.close()


def test_largest_m_fits_and_one_tile_more_is_rejected(bsg):
    # K = 3072 from a misaligned act takes the scratch: M <= 5440 tokens.
    k = 3072
    lin, wt, rng = _layer(bsg, 64, k, 0.90, 4300)
    tile = lin.info["tile_m"]
    m_max = bsg.STATIC_SCRATCH_BYTES // lin.workspace_bytes(tile) * tile
    assert m_max == 5440
    assert lin.workspace_bytes(m_max) <= bsg.STATIC_SCRATCH_BYTES < lin.workspace_bytes(m_max + 1)
    x = synth.draw_x(rng, m_max + 1, k, "u127")
    _, ptr = keep = _device_act(x, 4)
    got, ref = _run_both(bsg, lin, ptr, m_max, synth.I32, 1.0)
    want = oracle.linear(x[:m_max], oracle.weight_dense(wt), wt.scales, wt.bias, synth.I32,
                         threads=os.cpu_count() or 8)
    _check(got, want, synth.I32, "M = 5440 through the scratch")
    out = torch.empty((m_max + 1, 64), dtype=torch.int32, device="cuda")
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.bsgemm_run_static(lin._h, ptr, m_max + 1, out.data_ptr(), synth.I32, 1.0,
                              torch.cuda.current_stream().cuda_stream)
    assert e.value.code == bsg.ERR_INVALID and "static scratch" in str(e.value)
    # the same M from an aligned act takes the one-kernel path, which uses
    # no scratch: accepted
    _, aptr = keep2 = _device_act(x, 0)
    bsg.bsgemm_run_static(lin._h, aptr, m_max + 1, out.data_ptr(), synth.I32, 1.0,
                          torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy()[:m_max], want)
    del keep, keep2
    lin.close()
