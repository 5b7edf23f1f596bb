"""The C-ABI library builds, loads, exports every symbol include/bsgemm.h
declares, and rejects bad arguments before touching a GPU; the binding's
create-time helpers agree with the oracle.  CPU only."""
import ctypes
import os
import re
import shutil

import numpy as np
import pytest

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bsgemm.h")


@pytest.fixture(scope="module")
def bsg():
    if not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bsgemm_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("bsgemm_create", "bsgemm_run", "bsgemm_destroy", "bsgemm_last_error"):
        assert required in names


def test_library_exports_every_declared_symbol(bsg):
    lib = ctypes.CDLL(bsg.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(bsg.EXPORTED)


def test_max_k(bsg):
    k = bsg.bsgemm_max_k()
    assert 3072 <= k < 131072  # covers the DistilBERT FFN2 (K = 3072)


@pytest.fixture(params=["bsgemm_create", "bsgemm_create_tc"])
def create_fn(request):
    return request.param


def test_create_rejects_bad_arrays(bsg, create_fn):
    """bsgemm_create and bsgemm_create_tc (the same weight, also laid out
    for the tensor cores) validate the same way, before any device call."""
    def _create(bsg, *args):
        with pytest.raises(bsg.BsgemmError) as e:
            getattr(bsg, create_fn)(*args)
        return e.value.code

    ones = [1.0] * 8
    assert _create(bsg, 6, 8, 4, [0, 1, 1, 8], [[1] * 4], [1.0] * 6) == bsg.ERR_INVALID  # N = 6 (2 block-rows): column = K
    assert _create(bsg, 8, 8, 2, [0, 0, 0], [], ones) == bsg.ERR_UNSUPPORTED         # block != 4
    assert _create(bsg, 8, 10**6, 4, [0, 0, 0], [], ones) == bsg.ERR_UNSUPPORTED     # K too large
    assert _create(bsg, 8, 8, 4, [1, 1, 1], [], ones) == bsg.ERR_INVALID             # indptr[0] != 0
    assert _create(bsg, 8, 8, 4, [0, 2, 1, 9, 3], [[1] * 4] * 2, ones) == bsg.ERR_INVALID  # decreasing
    assert _create(bsg, 8, 8, 4, [0, 1, 1, 8], [[1] * 4], ones) == bsg.ERR_INVALID   # column = K
    assert _create(bsg, 8, 8, 4, [0, 2, 2, 3, 3], [[1] * 4] * 2, ones) == bsg.ERR_INVALID  # repeated column
    assert _create(bsg, 8, 8, 4, [0, 2, 2, 5, 3], [[1] * 4] * 2, ones) == bsg.ERR_INVALID  # unsorted
    assert _create(bsg, 8, 8, 4, [0, 0, 0], [], [1.0] * 7 + [np.inf]) == bsg.ERR_INVALID  # scale inf
    assert _create(bsg, 4, 8, 4, [0, 0], [], [1.0] * 4, [0, 0, np.nan, 0]) == bsg.ERR_INVALID  # bias nan
    assert _create(bsg, 0, 8, 4, [0], [], []) == bsg.ERR_INVALID


def test_run_rejects_bad_arguments_without_a_gpu(bsg):
    # a NULL handle is rejected before any CUDA call
    with pytest.raises(bsg.BsgemmError) as e:
        bsg.bsgemm_run(None, 0, 1, 0, bsg.OUT_I32)
    assert e.value.code == bsg.ERR_INVALID
    assert "handle" in bsg.bsgemm_last_error()


def test_dense_to_blocks(bsg):
    rng = np.random.default_rng(3)
    w = rng.integers(-3, 4, size=(12, 7)).astype(np.int8)
    w[rng.random(w.shape) < 0.6] = 0
    indptr, colidx, values = bsg.dense_to_blocks(w)
    back = np.zeros_like(w)
    for r in range(3):
        for j in range(indptr[r], indptr[r + 1]):
            back[4 * r:4 * r + 4, colidx[j]] = values[j]
    assert np.array_equal(back, w)
    assert all((values[j] != 0).any() for j in range(len(colidx)))


def test_block_prune_rejects_bad_arguments(bsg):
    """Shape, pointer and sparsity checks come before any CUDA call."""
    def code(*args):
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_block_prune(*args)
        return e.value.code
    assert code(6, 8, 16, 0.5, 16) == bsg.ERR_INVALID      # N % 4
    assert code(0, 8, 16, 0.5, 16) == bsg.ERR_INVALID      # N = 0
    assert code(8, 0, 16, 0.5, 16) == bsg.ERR_INVALID      # K = 0
    assert code(8, 8, 0, 0.5, 16) == bsg.ERR_INVALID       # W NULL
    assert code(8, 8, 16, 0.5, 0) == bsg.ERR_INVALID       # keep NULL
    assert code(8, 8, 16, 1.5, 16) == bsg.ERR_INVALID      # sparsity > 1
    assert code(8, 8, 16, -0.1, 16) == bsg.ERR_INVALID     # sparsity < 0
    assert code(8, 8, 16, float("nan"), 16) == bsg.ERR_INVALID


def test_attention_rejects_bad_arguments(bsg):
    """Shape, stride, scale, kind and pointer checks come before any CUDA
    call; batch = 0 is a no-op."""
    def code(batch=2, seq=8, heads=12, head_dim=64, ld=2304, scale=0.05, qkv=16, out=16, kind=None, out_scale=1.0,
             flags=0):
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_attention(qkv, batch, seq, heads, head_dim, ld, scale, out,
                                 bsg.OUT_F32 if kind is None else kind, out_scale, 0, flags)
        return e.value.code
    assert code(head_dim=32) == bsg.ERR_UNSUPPORTED
    assert code(seq=bsg.ATTN_MAX_SEQ + 1) == bsg.ERR_UNSUPPORTED
    assert code(batch=-1) == bsg.ERR_INVALID
    assert code(batch=65536) == bsg.ERR_INVALID
    assert code(heads=0) == bsg.ERR_INVALID
    assert code(seq=-1) == bsg.ERR_INVALID
    assert code(seq=0) == bsg.ERR_INVALID
    assert code(ld=2304 - 16) == bsg.ERR_INVALID            # ld < 3d
    assert code(ld=2304 + 8) == bsg.ERR_INVALID             # ld % 16
    assert code(scale=0.0) == bsg.ERR_INVALID
    assert code(scale=float("nan")) == bsg.ERR_INVALID
    assert code(scale=1e-20) == bsg.ERR_INVALID             # scale^2 / 8 not a normal fp32
    assert code(scale=1e30) == bsg.ERR_INVALID              # scores would overflow
    assert code(kind=bsg.OUT_I32) == bsg.ERR_INVALID
    assert code(kind=bsg.OUT_F32_GELU) == bsg.ERR_INVALID
    assert code(kind=bsg.OUT_I8, out_scale=0.0) == bsg.ERR_INVALID
    assert code(flags=2) == bsg.ERR_INVALID                 # only BSGEMM_ACT_READY is defined
    assert code(qkv=0) == bsg.ERR_INVALID
    assert code(out=0) == bsg.ERR_INVALID
    assert code(qkv=24) == bsg.ERR_INVALID                  # not 16-byte aligned
    assert code(out=8) == bsg.ERR_INVALID
    assert "aligned" in bsg.bsgemm_last_error()
    bsg.bsgemm_attention(0, 0, 8, 12, 64, 2304, 0.05, 0, bsg.OUT_F32)  # batch = 0: nothing to do


@pytest.mark.parametrize("n_out,k_in,sparsity", [(10, 24, 0.6), (30, 200, 0.5), (7, 8, 0.0), (5, 16, 1.0)])
def test_variant_shapes_decompress_like_the_oracle(bsg, n_out, k_in, sparsity):
    """The binding's 1 x 4 and 2:4 decompressions (create-time helpers)
    give the oracle's dense weight; the regrouped 4 x 1 blocks hold it."""
    rng = np.random.default_rng(90 + n_out)
    w1 = synth.draw_weight_1x4(rng, n_out, k_in, sparsity)
    a = bsg.dense_from_blocks_1x4(n_out, k_in, w1.indptr, w1.colgrp, w1.values)
    assert np.array_equal(a, oracle.bsr1x4_to_dense(n_out, k_in, w1.indptr, w1.colgrp, w1.values))
    indptr, colidx, values = bsg.dense_to_blocks(a)
    assert np.array_equal(oracle.bsr_to_dense(-(-n_out // 4) * 4, k_in, indptr, colidx, values)[:n_out], a)
    t = synth.draw_weight_2to4(rng, n_out, k_in)
    b = bsg.dense_from_2to4(t.values, t.idx)
    assert np.array_equal(b, oracle.sparse2to4_to_dense(t.values, t.idx))


def test_variant_shapes_reject_bad_arrays(bsg):
    ones = np.ones((2, 4), np.int8)
    for n, k, ip, cg in ((2, 6, [0, 1, 2], [0, 0]),       # K % 4
                         (2, 8, [1, 1, 2], [0, 1]),       # indptr[0] != 0
                         (2, 8, [0, 2, 1], [0, 1]),       # decreasing
                         (2, 8, [0, 1, 2], [0, 2]),       # group = K / 4
                         (2, 8, [0, 2, 2], [1, 1]),       # repeated group in a row
                         (2, 8, [0, 2, 2], [1, 0]),       # unsorted
                         (2, 8, [0, 1, 3], [0, 1])):      # indptr[N] != number of blocks
        with pytest.raises(ValueError):
            bsg.dense_from_blocks_1x4(n, k, ip, cg, ones)
    v = np.ones((1, 4), np.int8)
    for bad in ([[1, 1, 0, 1]], [[2, 1, 0, 1]], [[0, 4, 0, 1]]):
        with pytest.raises(ValueError):
            bsg.dense_from_2to4(v, np.array(bad, np.uint8))
    with pytest.raises(ValueError):
        bsg.dense_from_2to4(np.ones((1, 3), np.int8), np.zeros((1, 3), np.uint8))   # K not a multiple of 4


def test_create_1x4_and_2to4_reject_bad_arrays_before_the_device(bsg):
    """bsgemm_create_1x4 / bsgemm_create_2to4 check their host arrays before
    any device call (so this runs without a GPU)."""
    ones = np.ones((2, 4), np.int8)
    sc = np.ones(2, np.float32)
    for n, k, ip, cg in ((2, 6, [0, 1, 2], [0, 0]),       # K % 4
                         (2, 8, [1, 1, 2], [0, 1]),       # indptr[0] != 0
                         (2, 8, [0, 2, 1], [0, 1]),       # decreasing
                         (2, 8, [0, 1, 2], [0, 2]),       # group = K / 4
                         (2, 8, [0, 2, 2], [1, 1]),       # repeated group in a row
                         (2, 8, [0, 2, 2], [1, 0]),       # unsorted
                         (0, 8, [0], [])):                # N = 0
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_create_1x4(n, k, np.array(ip + cg, np.int32), ones, sc)
        assert e.value.code == bsg.ERR_INVALID
    with pytest.raises(bsg.BsgemmError) as e:  # a NaN scale
        bsg.bsgemm_create_1x4(2, 8, np.array([0, 1, 2, 0, 1], np.int32), ones, np.array([1, np.nan], np.float32))
    assert e.value.code == bsg.ERR_INVALID
    with pytest.raises(bsg.BsgemmError) as e:  # K beyond the tile
        bsg.bsgemm_create_1x4(1, 4 * (bsg.bsgemm_max_k() // 4 + 1), np.array([0, 0], np.int32), ones, sc[:1])
    assert e.value.code == bsg.ERR_UNSUPPORTED
    v = np.ones((1, 2), np.int8)
    for bad in ([[1, 1]], [[2, 1]], [[0, 4]]):  # positions must strictly increase within [0, 4)
        with pytest.raises(bsg.BsgemmError) as e:
            bsg.bsgemm_create_2to4(1, 4, v, np.array(bad, np.uint8), sc[:1])
        assert e.value.code == bsg.ERR_INVALID
