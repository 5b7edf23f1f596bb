"""Create-side block pruning on the GPU (App. A.1) against the oracle's
average-magnitude pruning: the keep-masks must be identical, ties included."""
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


def gpu_prune(bsg, w: np.ndarray, sparsity: float) -> np.ndarray:
    import torch
    keep = bsg.block_prune(torch.from_numpy(np.ascontiguousarray(w, np.float32)).cuda(), sparsity)
    torch.cuda.synchronize()
    return keep.cpu().numpy().astype(bool)


def check(bsg, w: np.ndarray, sparsity: float):
    got = gpu_prune(bsg, w, sparsity)
    want = oracle.block_prune(w, sparsity)
    assert got.shape == want.shape
    bad = np.argwhere(got != want)
    assert bad.size == 0, f"{len(bad)} blocks differ, first at {bad[0].tolist()}"
    return got


@pytest.mark.parametrize("sparsity", [0.0, 1 / 3, 0.5, 0.8, 0.9, 0.97, 1.0])
def test_prune_random_weights(bsg, sparsity):
    rng = synth.rng_for(6100)
    w = rng.normal(0.0, 0.02, size=(96, 333)).astype(np.float32)
    keep = check(bsg, w, sparsity)
    total = keep.size
    assert keep.sum() == total - int(np.floor(sparsity * total + 0.5))


def test_prune_ties_broken_by_lower_index(bsg):
    """Integer-valued weights give many equal scores; an all-equal weight
    makes every block a tie, so the lowest indices are pruned."""
    rng = synth.rng_for(6110)
    w = rng.integers(-3, 4, size=(64, 250)).astype(np.float32)
    for s in (0.1, 0.5, 0.77):
        check(bsg, w, s)
    flat = np.full((8, 50), 0.25, np.float32)
    keep = check(bsg, flat, 0.3)
    assert not keep.reshape(-1)[:30].any() and keep.reshape(-1)[30:].all()


def test_prune_zeros_signs_and_wide_exponents(bsg):
    """Signed zeros score 0; magnitudes far apart make the double sum round."""
    rng = synth.rng_for(6120)
    w = rng.normal(0.0, 1.0, size=(40, 77)).astype(np.float32)
    w *= np.float32(2.0) ** rng.integers(-60, 60, size=w.shape).astype(np.float32)
    w[::3, ::5] = 0.0
    w[1::3, ::7] = -0.0
    for s in (0.25, 0.6, 0.9):
        check(bsg, w, s)


@pytest.mark.parametrize("n_out,k_in", [(4, 1), (4, 7), (8, 1), (12, 3)])
def test_prune_tiny_shapes(bsg, n_out, k_in):
    rng = synth.rng_for(6130 + n_out + k_in)
    w = rng.normal(size=(n_out, k_in)).astype(np.float32)
    for s in (0.0, 0.2, 0.5, 0.99, 1.0):
        check(bsg, w, s)


def test_prune_ffn_weights_full_size(bsg):
    """The FFN2 (3072 -> 768) and FFN1 (768 -> 3072) weight shapes."""
    rng = synth.rng_for(6140)
    check(bsg, rng.normal(0.0, 0.02, size=(768, 3072)).astype(np.float32), 0.9)
    check(bsg, rng.normal(0.0, 0.02, size=(3072, 768)).astype(np.float32), 0.8)


def test_prune_rejects_non_finite_weights(bsg):
    import torch
    w = torch.zeros((8, 16), dtype=torch.float32, device="cuda")
    w[5, 3] = float("nan")
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.block_prune(w, 0.5)
    assert e.value.code == bsg.ERR_INVALID
    w[5, 3] = float("inf")
    with pytest.raises(bsg.BsgemmError):
        bsg.block_prune(w, 0.5)


def test_pruned_weight_through_the_layer(bsg):
    """Prune, quantise symmetric per output channel, pack with the mask, run:
    the layer equals the oracle's linear on the masked dense weight."""
    import torch
    rng = synth.rng_for(6150)
    n_out, k_in, m = 128, 640, 200
    wf = rng.normal(0.0, 0.05, size=(n_out, k_in)).astype(np.float32)
    keep = gpu_prune(bsg, wf, 0.85)
    mask = np.repeat(keep, 4, axis=0)
    amax = np.abs(wf * mask).max(axis=1, keepdims=True)
    amax[amax == 0] = 1.0
    wq = np.clip(np.rint(wf / amax * 127.0), -127, 127).astype(np.int8) * mask.astype(np.int8)
    scales = (amax[:, 0] / 127.0 * 0.02).astype(np.float32)
    bias = rng.normal(0.0, 0.02, size=n_out).astype(np.float32)
    lin = bsg.SparseInt8Linear.from_dense(wq, scales, bias, keep=keep)
    assert lin.info["nnzb"] == int(keep.sum())
    x = synth.draw_x(rng, m, k_in, "u127")
    out = lin(torch.from_numpy(x).cuda(), synth.I8, 0.05).cpu().numpy()
    want = oracle.linear(x, wq, scales, bias, synth.I8, out_scale=0.05)
    assert np.array_equal(out, want)
    lin.close()
