"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Integer outputs (int32 accumulators, requantised int8) must match bit for
bit; fp32 outputs within |d| <= 1e-4 or |d| <= 1e-5 |oracle| per element,
where the oracle gives the exact value in fp64.
"""
import os

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
        assert not bad.any(), (f"{what}: {bad.sum()} fp32 elements out of tolerance, max abs err "
                               f"{err.max():.3g}, first at {np.argwhere(bad)[0].tolist()}")
    else:
        diff = got != want
        assert not diff.any(), f"{what}: {diff.sum()} elements differ, first at {np.argwhere(diff)[0].tolist()}"


def make_linear(bsg, wt):
    return bsg.SparseInt8Linear(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values, wt.scales, wt.bias)


def gpu_run(lin, x: np.ndarray, kind: int, out_scale: float, workspace=None) -> np.ndarray:
    """workspace=None: bsgemm_run_ws (with K % 16 == 0 the one kernel that
    stages tiles by tensor copies, else relayout + bulk copies);
    workspace=False: bsgemm_run (tensor copies, else per-thread gathers)."""
    xd = torch.from_numpy(x).cuda()
    dtype = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
             synth.I8: torch.int8, synth.I8_GELU: torch.int8}[kind]
    out = torch.empty((x.shape[0], lin.n_out), dtype=dtype, device="cuda")
    lin.run(xd, out, kind, out_scale, workspace=workspace)
    torch.cuda.synchronize()
    return out.cpu().numpy()


PATHS = {"ws": None, "nows": False}


# -------------------------------------------------- small, every element --

SMALL = [  # (n_out, k_in, m, sparsity, x_dist)
    (768, 768, 300, 0.90, "u127"),    # 128-token tiles, 3 tiles + ragged tail
    (256, 768, 129, 0.80, "n30"),
    (64, 3072, 200, 0.90, "u0_127"),  # 64-token tiles (K > 1536)
    (3072, 96, 70, 0.70, "u127"),
]


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("shape", SMALL, ids=lambda s: "x".join(map(str, s[:3])))
@pytest.mark.parametrize("kind", KINDS, ids=lambda k: synth.KIND_NAMES[k])
def test_small_all_elements(bsg, shape, kind, path):
    n, k, m, sp, dist = shape
    rng = synth.rng_for(1000 + n + k + m)
    wt = synth.draw_weight(rng, n, k, sp)
    x = synth.draw_x(rng, m, k, dist)
    lin = make_linear(bsg, wt)
    got = gpu_run(lin, x, kind, 0.05, PATHS[path])
    want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, kind, out_scale=0.05, threads=8)
    check(got, want, kind, f"{shape}")


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("m", [1, 3, 63, 64, 65, 127, 128, 129, 257])
def test_token_counts_span_tiles(bsg, m, path):
    for k in (768, 3072):
        rng = synth.rng_for(2000 + m + k)
        wt = synth.draw_weight(rng, 32, k, 0.85)
        x = synth.draw_x(rng, m, k, "u127")
        lin = make_linear(bsg, wt)
        want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, synth.I32)
        check(gpu_run(lin, x, synth.I32, 1.0, PATHS[path]), want, synth.I32, f"m={m} k={k}")


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("k", [1, 3, 5, 17, 37, 100, 1001, 1536, 1537, 2049])
def test_ragged_k(bsg, k, path):
    """K not a multiple of 4/16/32 takes the byte-wise load paths."""
    rng = synth.rng_for(3000 + k)
    wt = synth.draw_weight(rng, 48, k, 0.5)
    x = synth.draw_x(rng, 77, k, "u127")
    lin = make_linear(bsg, wt)
    w = oracle.weight_dense(wt)
    for kind in (synth.I32, synth.I8_GELU):
        check(gpu_run(lin, x, kind, 0.07, PATHS[path]), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.07),
              kind, f"k={k}")


@pytest.mark.parametrize("k", [512, 1024, 2048, 2560, 3072])
def test_k_multiple_of_64_tile_copies(bsg, k):
    """K a multiple of 64: the one-kernel path copies the token tile in
    boxes of 64 columns, one 3-D copy of K / 512 boxes per warp where that
    is more than one box (K = 1024, 2048, 2560, 3072), 2-D boxes otherwise
    (K = 512); tokens span three tiles and a ragged tail."""
    rng = synth.rng_for(3100 + k)
    wt = synth.draw_weight(rng, 80, k, 0.7)
    x = synth.draw_x(rng, 150, k, "u127")
    lin = make_linear(bsg, wt)
    w = oracle.weight_dense(wt)
    for kind in (synth.I32, synth.I8):
        check(gpu_run(lin, x, kind, 0.07, False), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.07),
              kind, f"k={k}")


def test_max_k_and_int32_extremes(bsg):
    """Largest supported K with the largest-magnitude values."""
    k = bsg.bsgemm_max_k()
    rng = synth.rng_for(4000)
    wt = synth.draw_weight(rng, 16, k, 0.0, value_lo=-128, value_hi=127)
    wt.values[:] = np.where(wt.values < 0, -128, 127).astype(np.int8)
    x = synth.draw_x(rng, 40, k, "extreme")
    x[0] = -128
    wt.values[: k] = -128  # block-row 0 all -128: acc = 16384 * K on row 0
    lin = make_linear(bsg, wt)
    w = oracle.weight_dense(wt)
    want = oracle.linear(x, w, wt.scales, wt.bias, synth.I32)
    assert want[0, 0] == 16384 * k
    check(gpu_run(lin, x, synth.I32, 1.0), want, synth.I32, "extremes i32")
    for kind in (synth.I8, synth.F32):
        check(gpu_run(lin, x, kind, 0.5), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.5), kind)


def test_empty_and_dense_block_rows(bsg):
    """Block-rows with no stored block, fully dense block-rows, and stored
    blocks whose values are all zero."""
    n, k = 40, 300
    rng = synth.rng_for(5000)
    dense = rng.integers(-127, 128, size=(n, k)).astype(np.int8)
    mask = rng.random((n // 4, k)) < 0.2
    mask[0] = False          # empty
    mask[3] = False          # empty
    mask[9] = False          # empty (last)
    mask[1] = True           # fully dense
    mask[5] = True
    dense[8:12, :] = 0       # block-row 2: stored blocks of zeros
    mask[2, ::3] = True
    indptr, colidx, values = oracle.dense_to_bsr(dense, mask)
    scales = rng.uniform(1e-3, 1e-2, n).astype(np.float32)
    bias = rng.normal(0, 0.02, n).astype(np.float32)
    lin = bsg.SparseInt8Linear(n, k, indptr, colidx, values, scales, bias)
    w = oracle.bsr_to_dense(n, k, indptr, colidx, values)
    x = synth.draw_x(rng, 150, k, "u127")
    for kind in KINDS:
        check(gpu_run(lin, x, kind, 0.05), oracle.linear(x, w, scales, bias, kind, out_scale=0.05), kind,
              synth.KIND_NAMES[kind])


def test_all_blocks_pruned_gives_bias(bsg):
    rng = synth.rng_for(5100)
    wt = synth.draw_weight(rng, 64, 768, 1.0)
    assert wt.nnzb == 0
    x = synth.draw_x(rng, 200, 768, "u127")
    lin = make_linear(bsg, wt)
    assert not gpu_run(lin, x, synth.I32, 1.0).any()
    y = gpu_run(lin, x, synth.F32, 1.0)
    assert np.array_equal(y, np.broadcast_to(wt.bias, y.shape))


def test_null_bias_and_zero_m(bsg):
    rng = synth.rng_for(5200)
    wt = synth.draw_weight(rng, 16, 64, 0.5)
    lin = bsg.SparseInt8Linear(16, 64, wt.indptr, wt.colidx, wt.values, wt.scales, None)
    x = synth.draw_x(rng, 9, 64, "u127")
    want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, None, synth.F32)
    check(gpu_run(lin, x, synth.F32, 1.0), want, synth.F32)
    empty = torch.empty((0, 64), dtype=torch.int8, device="cuda")
    assert lin(empty, synth.F32).shape == (0, 16)


def test_run_argument_errors(bsg):
    rng = synth.rng_for(5300)
    wt = synth.draw_weight(rng, 16, 64, 0.5)
    lin = make_linear(bsg, wt)
    x = torch.zeros((4, 64), dtype=torch.int8, device="cuda")
    out = torch.empty((4, 16), dtype=torch.int8, device="cuda")
    for bad_scale in (0.0, -1.0, float("inf"), float("nan")):
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_run(lin._h, x.data_ptr(), 4, out.data_ptr(), bsg.OUT_I8, bad_scale)
        assert e.value.code == bsg.ERR_INVALID
    with pytest.raises(bsg.BsgemmError):
        bsg.bsgemm_run(lin._h, x.data_ptr(), 4, out.data_ptr(), 7, 1.0)
    with pytest.raises(bsg.BsgemmError):
        bsg.bsgemm_run(lin._h, x.data_ptr(), -1, out.data_ptr(), bsg.OUT_I32, 1.0)
    raw = torch.empty(4 * 16 * 4 + 16, dtype=torch.uint8, device="cuda")
    with pytest.raises(bsg.BsgemmError):  # misaligned output
        bsg.bsgemm_run(lin._h, x.data_ptr(), 4, raw.data_ptr() + 4, bsg.OUT_I32, 1.0)


@pytest.mark.parametrize("offset", [1, 3, 4, 8])
def test_misaligned_activations(bsg, offset):
    """An activation pointer that is not 16-byte aligned is still exact, on
    both paths."""
    rng = synth.rng_for(5400 + offset)
    wt = synth.draw_weight(rng, 32, 768, 0.9)
    x = synth.draw_x(rng, 100, 768, "u127")
    buf = torch.zeros(100 * 768 + 16, dtype=torch.int8, device="cuda")
    buf[offset:offset + 100 * 768] = torch.from_numpy(x.reshape(-1)).cuda()
    lin = make_linear(bsg, wt)
    want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, synth.I32)
    stream = torch.cuda.current_stream().cuda_stream
    out = torch.empty((100, 32), dtype=torch.int32, device="cuda")
    bsg.bsgemm_run(lin._h, buf.data_ptr() + offset, 100, out.data_ptr(), bsg.OUT_I32, 1.0, stream)
    torch.cuda.synchronize()
    check(out.cpu().numpy(), want, synth.I32, "no workspace")
    ws = torch.empty(lin.workspace_bytes(100), dtype=torch.uint8, device="cuda")
    out.zero_()
    bsg.bsgemm_run_ws(lin._h, buf.data_ptr() + offset, 100, out.data_ptr(), bsg.OUT_I32, 1.0, ws.data_ptr(),
                      ws.numel(), stream)
    torch.cuda.synchronize()
    check(out.cpu().numpy(), want, synth.I32, "workspace")


def test_workspace_validation_and_status(bsg):
    rng = synth.rng_for(5450)
    wt = synth.draw_weight(rng, 64, 3072, 0.9)
    lin = make_linear(bsg, wt)
    m = 70
    need = lin.workspace_bytes(m)
    assert need == -(-m // lin.info["tile_m"]) * 3072 * lin.info["tile_m"]
    x = torch.zeros((m, 3072), dtype=torch.int8, device="cuda")
    out = torch.empty((m, 64), dtype=torch.int8, device="cuda")
    ws = torch.empty(need + 16, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    with pytest.raises(bsg.BsgemmError):  # too small
        bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, out.data_ptr(), bsg.OUT_I8, 0.05, ws.data_ptr(), need - 16, stream)
    with pytest.raises(bsg.BsgemmError):  # misaligned
        bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, out.data_ptr(), bsg.OUT_I8, 0.05, ws.data_ptr() + 8, need, stream)
    with pytest.raises(bsg.BsgemmError):  # NULL
        bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, out.data_ptr(), bsg.OUT_I8, 0.05, None, need, stream)
    bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, out.data_ptr(), bsg.OUT_I8, 0.05, ws.data_ptr(), need, stream)
    torch.cuda.synchronize()
    assert bsg.bsgemm_device_status(lin._h) == 0


@pytest.mark.parametrize("path", sorted(PATHS))
def test_guard_bands_and_determinism(bsg, path):
    """Nothing is written outside out[M][N] (nor outside the workspace); two
    runs are bit-identical."""
    rng = synth.rng_for(5500)
    wt = synth.draw_weight(rng, 96, 3072, 0.9)
    m = 131
    x = torch.from_numpy(synth.draw_x(rng, m, 3072, "u0_127")).cuda()
    lin = make_linear(bsg, wt)
    stream = torch.cuda.current_stream().cuda_stream
    guard = 4096
    need = lin.workspace_bytes(m)
    wsraw = torch.full((guard * 2 + need,), 0x3C, dtype=torch.uint8, device="cuda")

    def run(kind, ptr):
        if path == "ws":
            bsg.bsgemm_run_ws(lin._h, x.data_ptr(), m, ptr, kind, 0.05, wsraw.data_ptr() + guard, need, stream)
        else:
            bsg.bsgemm_run(lin._h, x.data_ptr(), m, ptr, kind, 0.05, stream)

    for kind, elem in ((synth.I8, 1), (synth.F32, 4)):
        raw = torch.full((guard * 2 + m * 96 * elem,), 0x5A, dtype=torch.uint8, device="cuda")
        run(kind, raw.data_ptr() + guard)
        first = raw.clone()
        run(kind, raw.data_ptr() + guard)
        torch.cuda.synchronize()
        assert torch.equal(first, raw)
        assert bool((raw[:guard] == 0x5A).all()) and bool((raw[-guard:] == 0x5A).all())
        assert bool((wsraw[:guard] == 0x3C).all()) and bool((wsraw[-guard:] == 0x3C).all())
    assert bsg.bsgemm_device_status(lin._h) == 0


def test_one_handle_many_streams(bsg):
    """The handle is immutable: concurrent runs on several streams (weight
    sharing across parallel instances) all give the oracle's result."""
    rng = synth.rng_for(5600)
    wt = synth.draw_weight(rng, 768, 768, 0.9)
    lin = make_linear(bsg, wt)
    w = oracle.weight_dense(wt)
    xs = [synth.draw_x(rng, 64 * (i + 1), 768, "u127") for i in range(4)]
    streams = [torch.cuda.Stream() for _ in xs]
    outs = []
    for x, s in zip(xs, streams):
        with torch.cuda.stream(s):
            xd = torch.from_numpy(x).cuda(non_blocking=False)
            out = torch.empty((x.shape[0], 768), dtype=torch.int8, device="cuda")
            lin.run(xd, out, synth.I8, 0.05, stream=s)
            outs.append(out)
    torch.cuda.synchronize()
    for x, out in zip(xs, outs):
        check(out.cpu().numpy(), oracle.linear(x, w, wt.scales, wt.bias, synth.I8, out_scale=0.05), synth.I8)


def test_host_tensors_round_trip(bsg):
    """The end-to-end call: CPU input in, CPU result out."""
    rng = synth.rng_for(5700)
    wt = synth.draw_weight(rng, 64, 768, 0.9)
    x = synth.draw_x(rng, 50, 768, "u127")
    lin = make_linear(bsg, wt)
    got = lin(torch.from_numpy(x), synth.I8, 0.05)
    assert not got.is_cuda
    check(got.numpy(), oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, synth.I8, out_scale=0.05),
          synth.I8)


def test_host_tensors_pipelined_on_two_streams(bsg):
    """The asynchronous end-to-end call: pinned batches in, pinned results
    out, steps alternating between two streams, read after a synchronize."""
    import torch
    rng = synth.rng_for(5710)
    wt = synth.draw_weight(rng, 96, 1024, 0.9)
    w = oracle.weight_dense(wt)
    lin = make_linear(bsg, wt)
    streams = [torch.cuda.Stream() for _ in range(2)]
    xs = [synth.draw_x(rng, m, 1024, "u127") for m in (130, 64, 1, 257)]
    hx = [torch.from_numpy(x).pin_memory() for x in xs]
    hout = [torch.empty((x.shape[0], 96), dtype=torch.int8, pin_memory=True) for x in xs]
    for i in range(len(xs)):
        got = lin(hx[i], synth.I8_GELU, 0.03, stream=streams[i % 2], out=hout[i], sync=False)
        assert got is hout[i]
    for st in streams:
        st.synchronize()
    for x, out in zip(xs, hout):
        check(out.numpy(), oracle.linear(x, w, wt.scales, wt.bias, synth.I8_GELU, out_scale=0.03), synth.I8_GELU)
    with pytest.raises(ValueError):
        lin(torch.from_numpy(xs[0]), synth.I8, 1.0, out=hout[0], sync=False)
    with pytest.raises(ValueError):
        lin(hx[0], synth.F32, 1.0, out=hout[0])


def test_run_host_through_the_c_abi(bsg):
    """bsgemm_run_host with raw pointers: pageable buffers (the copies block),
    every epilogue kind, and its argument checks."""
    import torch
    rng = synth.rng_for(5720)
    wt = synth.draw_weight(rng, 64, 520, 0.8)
    w = oracle.weight_dense(wt)
    lin = make_linear(bsg, wt)
    x = synth.draw_x(rng, 77, 520, "u127")
    for kind in KINDS:
        need = bsg.bsgemm_host_workspace_bytes(lin._h, 77, kind)
        elem = 1 if kind in (synth.I8, synth.I8_GELU) else 4
        assert need >= 77 * 520 + bsg.bsgemm_workspace_bytes(lin._h, 77) + 77 * 64 * elem
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        out = np.zeros((77, 64), dtype={synth.I32: np.int32, synth.I8: np.int8, synth.I8_GELU: np.int8}.get(kind, np.float32))
        bsg.bsgemm_run_host(lin._h, x.ctypes.data, 77, out.ctypes.data, kind, 0.04, ws.data_ptr(), need, 0)
        torch.cuda.synchronize()
        check(out, oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.04), kind)
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_run_host(lin._h, x.ctypes.data, 77, out.ctypes.data, kind, 0.04, ws.data_ptr(), need - 1, 0)
        assert e.value.code == bsg.ERR_INVALID
    assert bsg.bsgemm_host_workspace_bytes(lin._h, 77, 7) == 0
    bsg.bsgemm_run_host(lin._h, 0, 0, 0, synth.I8, 1.0, 0, 0, 0)  # M = 0: nothing to do
    with pytest.raises(bsg.BsgemmError):
        bsg.bsgemm_run_host(lin._h, 0, 77, 0, synth.I8, 1.0, ws.data_ptr(), need, 0)


@pytest.mark.parametrize("k", [768, 1001, 3072])
def test_relayout_then_tiled_kernel(bsg, k):
    """The two-kernel path: the relayout kernel writes the token tiles
    (bsgemm_tile_activations) and the layer kernel copies them in
    (bsgemm_run_tiled); the fast call stages tiles from x itself instead."""
    import torch
    rng = synth.rng_for(5900 + k)
    wt = synth.draw_weight(rng, 96, k, 0.85)
    w = oracle.weight_dense(wt)
    lin = make_linear(bsg, wt)
    m = 150
    x = synth.draw_x(rng, m, k, "u127")
    xd = torch.from_numpy(x).cuda()
    need = lin.workspace_bytes(m)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    for kind in KINDS:
        dt = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
              synth.I8: torch.int8, synth.I8_GELU: torch.int8}[kind]
        out = torch.empty((m, 96), dtype=dt, device="cuda")
        torch.cuda.synchronize()
        bsg.bsgemm_tile_activations(lin._h, xd.data_ptr(), m, ws.data_ptr(), need, 0)
        bsg.bsgemm_run_tiled(lin._h, ws.data_ptr(), need, m, out.data_ptr(), kind, 0.05, 0)
        torch.cuda.synchronize()
        check(out.cpu().numpy(), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05), kind)
    assert bsg.bsgemm_device_status(lin._h) == 0


@pytest.mark.parametrize("n_out,k_in,m,pad", [(96, 768, 200, 0), (64, 3072, 130, 16), (48, 1001, 64, 0),
                                              (32, 40, 1, 16), (16, 3072, 4096, 0), (16, 3136, 70, 0)])
def test_kmajor_input(bsg, n_out, k_in, m, pad):
    """bsgemm_run_kmajor: X^T [K][M] (row stride a multiple of 16, padded or
    not) copied straight into the tile layout; every element, every kind."""
    import torch
    rng = synth.rng_for(6000 + n_out + k_in + m)
    wt = synth.draw_weight(rng, n_out, k_in, 0.85)
    w = oracle.weight_dense(wt)
    lin = make_linear(bsg, wt)
    x = synth.draw_x(rng, m, k_in, "u127")
    ld = -(-m // 16) * 16 + pad
    xt_full = torch.full((k_in, ld), 99, dtype=torch.int8, device="cuda")  # padding columns hold junk
    xt_full[:, :m] = torch.from_numpy(np.ascontiguousarray(x.T)).cuda()
    xt = xt_full[:, :m]
    for kind in KINDS:
        dt = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
              synth.I8: torch.int8, synth.I8_GELU: torch.int8}[kind]
        out = torch.empty((m, n_out), dtype=dt, device="cuda")
        lin.run_kmajor(xt, out, kind, 0.05)
        torch.cuda.synchronize()
        check(out.cpu().numpy(), oracle.linear(x, w, wt.scales, wt.bias, kind, out_scale=0.05), kind)
    assert bsg.bsgemm_device_status(lin._h) == 0
    lin.close()


def test_kmajor_argument_checks(bsg):
    import torch
    rng = synth.rng_for(6050)
    wt = synth.draw_weight(rng, 16, 64, 0.5)
    lin = make_linear(bsg, wt)
    xt = torch.zeros((64, 48), dtype=torch.int8, device="cuda")
    out = torch.empty((40, 16), dtype=torch.int8, device="cuda")
    with pytest.raises(bsg.BsgemmError) as e:  # ld not a multiple of 16
        bsg.bsgemm_run_kmajor(lin._h, xt.data_ptr(), 40, 40, out.data_ptr(), synth.I8, 1.0, 0)
    assert e.value.code == bsg.ERR_INVALID
    with pytest.raises(bsg.BsgemmError):  # ld < M
        bsg.bsgemm_run_kmajor(lin._h, xt.data_ptr(), 40, 32, out.data_ptr(), synth.I8, 1.0, 0)
    with pytest.raises(bsg.BsgemmError):  # misaligned act
        bsg.bsgemm_run_kmajor(lin._h, xt.data_ptr() + 4, 40, 48, out.data_ptr(), synth.I8, 1.0, 0)
    lin.close()


@pytest.mark.parametrize("n_out,k_in,m", [(6, 768, 130), (1, 64, 70), (18, 1001, 65), (770, 768, 200),
                                          (3, 3072, 64)])
def test_n_not_a_multiple_of_4(bsg, n_out, k_in, m):
    """The last block-row holds N % 4 rows: zero-padded at create time, only
    channels < N stored (rows of out are then not 16-byte aligned).  Every
    staging path, every kind, every element."""
    import torch
    rng = synth.rng_for(6200 + n_out + k_in)
    n4 = -(-n_out // 4) * 4
    wt = synth.draw_weight(rng, n4, k_in, 0.8)
    w = np.ascontiguousarray(oracle.weight_dense(wt)[:n_out])
    scales, bias = wt.scales[:n_out].copy(), wt.bias[:n_out].copy()
    lin = bsg.SparseInt8Linear.from_dense(w, scales, bias)
    assert lin.n_out == n_out
    x = synth.draw_x(rng, m, k_in, "u127")
    for kind in KINDS:
        want = oracle.linear(x, w, scales, bias, kind, out_scale=0.05)
        for path in (None, False):
            check(gpu_run(lin, x, kind, 0.05, workspace=path), want, kind, f"path {path}")
        if m % 16 == 0:
            dt = {synth.I32: torch.int32, synth.F32: torch.float32, synth.F32_GELU: torch.float32,
                  synth.I8: torch.int8, synth.I8_GELU: torch.int8}[kind]
            out = torch.empty((m, n_out), dtype=dt, device="cuda")
            lin.run_kmajor(torch.from_numpy(np.ascontiguousarray(x.T)).cuda(), out, kind, 0.05)
            torch.cuda.synchronize()
            check(out.cpu().numpy(), want, kind, "kmajor")
    # a guard after the last row of out stays untouched
    xd = torch.from_numpy(x).cuda()
    buf = torch.full((m * n_out + 64,), 77, dtype=torch.int8, device="cuda")
    lin.run(xd, buf[: m * n_out].view(m, n_out), synth.I8, 0.05)
    torch.cuda.synchronize()
    assert (buf[m * n_out:].cpu().numpy() == 77).all()
    lin.close()


def test_act_ready_back_to_back(bsg):
    """BSGEMM_ACT_READY on independent batches launched back to back (the
    tile copies may start while the previous launch ends): every result
    equals the oracle's; an unknown flag bit is rejected."""
    import torch
    rng = synth.rng_for(6300)
    wt = synth.draw_weight(rng, 128, 1024, 0.85)
    w = oracle.weight_dense(wt)
    lin = make_linear(bsg, wt)
    xs = [synth.draw_x(rng, m, 1024, "u127") for m in (300, 64, 513, 129)]
    xds = [torch.from_numpy(x).cuda() for x in xs]
    outs = [torch.empty((x.shape[0], 128), dtype=torch.int8, device="cuda") for x in xs]
    torch.cuda.synchronize()
    for _ in range(3):
        for xd, out in zip(xds, outs):
            lin.run(xd, out, synth.I8_GELU, 0.04, act_ready=True)
    torch.cuda.synchronize()
    for x, out in zip(xs, outs):
        check(out.cpu().numpy(), oracle.linear(x, w, wt.scales, wt.bias, synth.I8_GELU, out_scale=0.04), synth.I8_GELU)
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.bsgemm_run(lin._h, xds[0].data_ptr(), 300, outs[0].data_ptr(), synth.I8, 1.0, 0, 2)
    assert e.value.code == bsg.ERR_INVALID
    lin.close()


def test_from_dense(bsg):
    rng = synth.rng_for(5800)
    wt = synth.draw_weight(rng, 128, 768, 0.8)
    w = oracle.weight_dense(wt)
    lin = bsg.SparseInt8Linear.from_dense(w, wt.scales, wt.bias)
    x = synth.draw_x(rng, 33, 768, "u127")
    check(gpu_run(lin, x, synth.F32_GELU, 1.0), oracle.linear(x, w, wt.scales, wt.bias, synth.F32_GELU),
          synth.F32_GELU)


# ------------------------------------------ full-size workloads, every element --

_ORACLE_CACHE = {}


def oracle_full(case, kind, out_scale):
    """The oracle's whole output for a full-size case (every row), computed
    once per (case, kind) and shared by the staging paths."""
    key = (case.name, kind, out_scale)
    if key not in _ORACLE_CACHE:
        wt = case.weight
        _ORACLE_CACHE[key] = oracle.linear(case.x, oracle.weight_dense(wt), wt.scales, wt.bias, kind,
                                           out_scale=out_scale, threads=os.cpu_count() or 8)
    return _ORACLE_CACHE[key]


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("case_fn", [synth.single_768, synth.ffn1, synth.ffn2], ids=lambda f: f.__name__)
def test_full_size_workloads(bsg, case_fn, path):
    case = case_fn()
    lin = make_linear(bsg, case.weight)
    got = gpu_run(lin, case.x, case.kind, case.out_scale, PATHS[path])
    check(got, oracle_full(case, case.kind, case.out_scale), case.kind, case.name)
    if case.kind in (synth.I8, synth.I8_GELU):
        # also the int32 accumulators, every element
        acc = gpu_run(lin, case.x, synth.I32, 1.0, PATHS[path])
        check(acc, oracle_full(case, synth.I32, 1.0), synth.I32, case.name + " acc")
    lin.close()


def test_encoder_layer_linears_full_size(bsg):
    """The four linears of one encoder layer at M = 8 x 384, int8 between,
    every element."""
    ws, x0 = synth.encoder_layer()
    x = x0
    for (name, n, k, kind), wt in zip(synth.LAYER_LINEARS, ws):
        if x.shape[1] != k:  # FFN2 consumes FFN1's width: use a seeded input
            x = synth.draw_x(synth.rng_for(6000), x0.shape[0], k, "u0_127")
        lin = make_linear(bsg, wt)
        got = gpu_run(lin, x, kind, 0.05)
        want = oracle.linear(x, oracle.weight_dense(wt), wt.scales, wt.bias, kind, out_scale=0.05,
                             threads=os.cpu_count() or 8)
        check(got, want, kind, name)
        lin.close()
