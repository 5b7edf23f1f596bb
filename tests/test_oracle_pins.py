"""Pins for the CPU oracle: checks against values and identities that do not
come from the oracle itself (hand-worked cases, closed forms, a library
matmul, brute force, invariants).  CPU only.

A mistake anywhere in the oracle (a dropped term, a wrong sign or index, a
transposed operand, a wrong rounding mode or coefficient) fails one of them.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _hand_cases():
    with open(os.path.join(GOLDEN, "hand_small.json")) as f:
        return json.load(f)["cases"]


# ---------------------------------------------------------------- format --

@pytest.mark.parametrize("case", _hand_cases(), ids=lambda c: c["name"])
def test_hand_cases_acc(case):
    """Hand-worked accumulators (App. A.1 block layout, Algorithm 1 dot)."""
    w = oracle.bsr_to_dense(case["N"], case["K"], case["indptr"], case["colidx"], case["values"])
    a = oracle.acc(np.array(case["X"], dtype=np.int8), w)
    assert a.tolist() == case["acc"]


def test_hand_case_epilogue():
    """Hand-worked dequantisation and tie-heavy requantisation."""
    case = [c for c in _hand_cases() if "q" in c][0]
    w = oracle.bsr_to_dense(case["N"], case["K"], case["indptr"], case["colidx"], case["values"])
    x = np.array(case["X"], dtype=np.int8)
    s = np.full(case["N"], case["scale"], np.float32)
    b = np.full(case["N"], case["bias"], np.float32)
    y = oracle.linear(x, w, s, b, oracle.F32)
    assert y.tolist() == case["y"]
    q = oracle.linear(x, w, s, b, oracle.I8, out_scale=case["out_scale"])
    assert q.tolist() == case["q"]


def test_block_orientation_is_output_rows():
    """A block covers 4 consecutive OUTPUT rows of one column (App. A.1)."""
    w = oracle.bsr_to_dense(8, 5, [0, 0, 1], [3], [[1, 2, 3, 4]])
    expect = np.zeros((8, 5), np.int8)
    expect[4:8, 3] = [1, 2, 3, 4]
    assert np.array_equal(w, expect)


def test_bsr_rejects_bad_arrays():
    with pytest.raises(ValueError):
        oracle.bsr_to_dense(4, 3, [0, 2], [2, 1], [[1] * 4, [1] * 4])  # unsorted
    with pytest.raises(ValueError):
        oracle.bsr_to_dense(4, 3, [0, 1], [3], [[1] * 4])  # column out of range
    with pytest.raises(ValueError):
        oracle.bsr_to_dense(6, 3, [0, 0], [], np.zeros((0, 4)))  # N not a multiple of 4


def test_dense_bsr_roundtrip_keeps_zero_valued_blocks():
    rng = np.random.default_rng(1)
    w = rng.integers(-127, 128, size=(12, 9)).astype(np.int8)
    mask = rng.random((3, 9)) < 0.4
    w[0:4, 2] = 0
    mask[0, 2] = True  # a stored block whose values are all zero
    indptr, colidx, values = oracle.dense_to_bsr(w, mask)
    assert indptr[-1] == mask.sum()
    back = oracle.bsr_to_dense(12, 9, indptr, colidx, values)
    expect = np.where(np.repeat(mask, 4, axis=0), w, 0).astype(np.int8)
    assert np.array_equal(back, expect)


def test_generator_matches_requested_sparsity():
    """Stored-block count = total - round(s * total); positions unique."""
    for (n, k, s) in [(768, 768, 0.9), (3072, 768, 0.8), (768, 3072, 0.9), (20, 7, 0.5)]:
        wt = synth.draw_weight(synth.rng_for(5), n, k, s)
        total = n // 4 * k
        assert wt.nnzb == total - int(math.floor(s * total + 0.5))
        w = oracle.weight_dense(wt)  # validates sortedness and range
        assert w.shape == (n, k)


# ---------------------------------------------------------- accumulation --

def test_fully_dense_equals_library_matmul():
    """0% block sparsity: the oracle equals numpy's int64 matmul."""
    rng = synth.rng_for(11)
    wt = synth.draw_weight(rng, 16, 37, 0.0)
    x = synth.draw_x(rng, 9, 37, "u127")
    # independent construction of the dense weight from the block values
    w_indep = wt.values.reshape(4, 37, 4).transpose(0, 2, 1).reshape(16, 37)
    expect = x.astype(np.int64) @ w_indep.astype(np.int64).T
    assert np.array_equal(oracle.acc(x, oracle.weight_dense(wt)), expect)


def test_random_sparse_equals_library_matmul():
    rng = synth.rng_for(12)
    wt = synth.draw_weight(rng, 64, 200, 0.9)
    x = synth.draw_x(rng, 33, 200, "n30")
    w = np.zeros((64, 200), np.int64)
    for r in range(16):
        for j in range(wt.indptr[r], wt.indptr[r + 1]):
            w[4 * r:4 * r + 4, wt.colidx[j]] = wt.values[j]
    assert np.array_equal(oracle.acc(x, oracle.weight_dense(wt)), x.astype(np.int64) @ w.T)


def test_all_blocks_zero_gives_bias():
    rng = synth.rng_for(13)
    wt = synth.draw_weight(rng, 32, 50, 1.0)
    assert wt.nnzb == 0
    x = synth.draw_x(rng, 7, 50, "u127")
    w = oracle.weight_dense(wt)
    assert not oracle.acc(x, w).any()
    y = oracle.linear(x, w, wt.scales, wt.bias, oracle.F32)
    assert np.array_equal(y, np.broadcast_to(wt.bias.astype(np.float64), y.shape))
    y32 = oracle.linear(x, w, wt.scales, None, oracle.F32)
    assert not y32.any()


def test_one_hot_block():
    rng = synth.rng_for(14)
    x = synth.draw_x(rng, 5, 11, "u127")
    v = [7, -128, 0, 127]
    w = oracle.bsr_to_dense(12, 11, [0, 0, 1, 1], [6], [v])
    a = oracle.acc(x, w)
    expect = np.zeros((5, 12), np.int64)
    for i in range(4):
        expect[:, 4 + i] = x[:, 6].astype(np.int64) * v[i]
    assert np.array_equal(a, expect)


def test_k_permutation_invariance_and_linearity():
    rng = synth.rng_for(15)
    wt = synth.draw_weight(rng, 24, 40, 0.7)
    w = oracle.weight_dense(wt)
    x1 = rng.integers(-63, 64, size=(6, 40)).astype(np.int8)
    x2 = rng.integers(-63, 64, size=(6, 40)).astype(np.int8)
    a1 = oracle.acc(x1, w)
    perm = rng.permutation(40)
    assert np.array_equal(oracle.acc(x1[:, perm], w[:, perm]), a1)
    assert np.array_equal(oracle.acc((x1 + x2).astype(np.int8), w), a1 + oracle.acc(x2, w))
    # negating the input negates the accumulator
    assert np.array_equal(oracle.acc((-x1).astype(np.int8), w), -a1)


def test_int32_extreme_and_overflow():
    """K = 131071 of (-128)*(-128) is the largest sum that fits int32."""
    k = 131071
    x = np.full((1, k), -128, np.int8)
    w = np.full((4, k), -128, np.int8)
    assert oracle.acc(x, w).tolist() == [[16384 * k] * 4]
    assert 16384 * k <= 2**31 - 1 < 16384 * (k + 1)
    with pytest.raises(OverflowError):
        oracle.acc(np.full((1, k + 1), -128, np.int8), np.full((4, k + 1), -128, np.int8))


# -------------------------------------------------------------- epilogue --

def _nearest_f32(q: Fraction) -> np.float32:
    """Round an exact rational to the nearest fp32, ties to even."""
    f = np.float32(float(q))
    best = None
    for c in (np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))):
        d = abs(Fraction(float(c)) - q)
        if best is None or d < best[0] or (d == best[0] and (c.view(np.int32) & 1) == 0):
            best = (d, c)
    return best[1]


def test_dequant_f32_is_single_rounding_of_exact_value():
    rng = np.random.default_rng(21)
    for _ in range(2000):
        a = int(rng.integers(-5_000_000, 5_000_000))
        s = np.float32(rng.uniform(1e-3, 1e-2))
        b = np.float32(rng.normal(0, 0.02))
        exact = Fraction(a) * Fraction(float(s)) + Fraction(float(b))  # |a| < 2^24: (float)a exact
        assert oracle.dequant_f32(a, s, b) == _nearest_f32(exact)
        assert oracle.dequant_f64(a, s, b) == pytest.approx(float(exact), rel=1e-15, abs=1e-300)


def test_requant_ties_and_saturation():
    """Round half to even, saturate to [-128, 127]."""
    cases = {2.5: 2, 3.5: 4, -2.5: -2, -3.5: -4, 0.5: 0, -0.5: 0, 1.4999999: 1,
             126.5: 126, 127.4: 127, 127.5: 127, 1e6: 127, -127.5: -128, -128.5: -128,
             -128.6: -128, -1e6: -128, 0.0: 0}
    for t, q in cases.items():
        assert oracle.requant(t, 1.0) == q, t
    # the multiply happens in fp32: 0.05 -> inv = 1/0.05f
    inv = np.float32(1.0) / np.float32(0.05)
    assert oracle.requant(np.float32(1.275), inv) == int(np.rint(np.float32(1.275) * inv))


def test_gelu_f64_closed_forms():
    """GELU(y) = y * Phi(y); standard normal CDF values from tables."""
    assert oracle.gelu_f64(0.0) == 0.0
    assert oracle.gelu_f64(1.0) == pytest.approx(0.8413447460685429, abs=1e-15)
    assert oracle.gelu_f64(-1.0) == pytest.approx(-0.15865525393145707, abs=1e-15)
    assert oracle.gelu_f64(2.0) == pytest.approx(2 * 0.9772498680518208, abs=1e-14)
    for y in (-3.0, -0.3, 0.7, 4.0):  # GELU(y) - GELU(-y) = y
        assert oracle.gelu_f64(y) - oracle.gelu_f64(-y) == pytest.approx(y, abs=1e-14)


def test_gelu_f32_within_derived_bound():
    """A&S 7.1.28 error <= 3e-7 on erf; fp32 evaluation of p^16 adds at
    most ~31 half-ulps relative; together |err| <= 1.2e-6 |y| + 1e-12."""
    ys = np.concatenate([np.linspace(-12, 12, 4801), np.linspace(-0.05, 0.05, 401),
                         np.linspace(-400, 400, 801)]).astype(np.float32)
    for y in ys:
        exact = 0.5 * float(y) * (1.0 + math.erf(float(y) / math.sqrt(2.0)))
        assert abs(float(oracle.gelu_f32(y)) - exact) <= 1.2e-6 * abs(float(y)) + 1e-12, y


def test_recip_f32_within_an_ulp_of_the_quotient():
    """Newton's method for 1/b (three steps from the 1/17 straight line)
    lands within one ulp of the exact reciprocal over [1, 2^25)."""
    rng = np.random.default_rng(7)
    bs = np.concatenate([rng.uniform(1.0, 2.0, 20000), np.exp2(rng.uniform(0.0, 25.0, 20000)),
                         [1.0, np.nextafter(np.float32(1), np.float32(2)), np.nextafter(np.float32(2), np.float32(1)),
                          3.0, 7.5, 2.0 ** 24 + 2.0, np.nextafter(np.float32(2.0 ** 25), np.float32(0))]]).astype(np.float32)
    for b in bs:
        r = float(oracle.recip_f32(b))
        exact = 1.0 / float(b)
        ulp = float(np.spacing(np.float32(exact)))
        assert abs(r - exact) <= ulp, (b, r, exact)


def test_recip_f32_powers_of_two_exact():
    for k in range(25):
        assert float(oracle.recip_f32(np.float32(2.0 ** k))) == 2.0 ** -k


def test_gelu_f32_special_values():
    assert float(oracle.gelu_f32(0.0)) == 0.0
    assert float(oracle.gelu_f32(1.0)) == pytest.approx(0.8413447460685429, abs=2e-7)
    for y in (5.7, 6.0, 50.0, 1e30):
        assert float(oracle.gelu_f32(y)) == np.float32(y)  # erf term rounds to exactly 1
    for y in (-5.7, -6.0, -50.0, -1e30):
        assert float(oracle.gelu_f32(y)) == 0.0


def test_i8_gelu_path_uses_fp32_sequence():
    """The int8 GELU output is requant(gelu_f32(fp32 dequant))."""
    rng = synth.rng_for(31)
    wt = synth.draw_weight(rng, 16, 64, 0.5)
    x = synth.draw_x(rng, 8, 64, "n30")
    w = oracle.weight_dense(wt)
    a = oracle.acc(x, w)
    q = oracle.linear(x, w, wt.scales, wt.bias, oracle.I8_GELU, out_scale=0.03)
    inv = np.float32(1.0) / np.float32(0.03)
    for m in range(8):
        for n in range(16):
            y = oracle.dequant_f32(a[m, n], wt.scales[n], wt.bias[n])
            assert q[m, n] == oracle.requant(oracle.gelu_f32(y), inv)


def test_row_sampling_and_threads_agree():
    rng = synth.rng_for(41)
    wt = synth.draw_weight(rng, 40, 96, 0.8)
    x = synth.draw_x(rng, 50, 96, "u127")
    w = oracle.weight_dense(wt)
    full = oracle.linear(x, w, wt.scales, wt.bias, oracle.I8, out_scale=0.05)
    par = oracle.linear(x, w, wt.scales, wt.bias, oracle.I8, out_scale=0.05, threads=4)
    rows = [0, 7, 49, 23]
    part = oracle.linear(x, w, wt.scales, wt.bias, oracle.I8, out_scale=0.05, rows=rows)
    assert np.array_equal(full, par)
    assert np.array_equal(full[rows], part)


# --------------------------------------------------------------- pruning --

def test_block_prune_hand_case():
    """Average-magnitude block score (App. A.1); lowest scores pruned."""
    w = np.array([[1, -8, 0.5],
                  [1, 8, 0.5],
                  [-1, 0, 0.5],
                  [1, 0, 0.5]], np.float32)  # scores: col0 1.0, col1 4.0, col2 0.5
    assert oracle.block_prune(w, 1 / 3).tolist() == [[True, True, False]]
    assert oracle.block_prune(w, 2 / 3).tolist() == [[False, True, False]]
    assert oracle.block_prune(w, 0.0).tolist() == [[True, True, True]]
    assert oracle.block_prune(w, 1.0).tolist() == [[False, False, False]]
    tie = np.ones((4, 3), np.float32)  # equal scores: lower index pruned first
    assert oracle.block_prune(tie, 1 / 3).tolist() == [[False, True, True]]


def test_block_prune_brute_force():
    rng = np.random.default_rng(51)
    for trial in range(20):
        n, k = 4 * int(rng.integers(1, 5)), int(rng.integers(1, 9))
        w = rng.normal(size=(n, k)).astype(np.float32)
        if trial % 3 == 0:
            w = np.round(w).astype(np.float32)  # many ties
        s = float(rng.uniform())
        keep = oracle.block_prune(w, s)
        total = (n // 4) * k
        npruned = int(math.floor(s * total + 0.5))
        assert keep.sum() == total - npruned
        # brute force: mean |w| of each block, stable order by (score, id)
        scores = []
        for r in range(n // 4):
            for c in range(k):
                scores.append((float(np.mean(np.abs(w[4 * r:4 * r + 4, c].astype(np.float64)))), r * k + c))
        pruned = {i for (_, i) in sorted(scores)[:npruned]}
        for r in range(n // 4):
            for c in range(k):
                assert keep[r, c] == ((r * k + c) not in pruned)


# ------------------------------------------------- residual add + LayerNorm --

def test_layernorm_hand_case():
    """z = [1, 2, 3, 4]: mean 2.5, variance 1.25, so the normalised row is
    (z - 2.5) / sqrt(1.25) = [-3, -1, 1, 3] / sqrt(5)."""
    z = np.array([[1, 2, 3, 4]], np.float32)
    got = oracle.layernorm(z, np.ones(4, np.float32), np.zeros(4, np.float32), 0.0)
    want = np.array([[-3, -1, 1, 3]]) / math.sqrt(5.0)
    assert np.allclose(got, want, rtol=0, atol=1e-15)
    # gamma and beta act per channel: 2 * norm + 3
    got2 = oracle.layernorm(z, np.full(4, 2, np.float32), np.full(4, 3, np.float32), 0.0)
    assert np.allclose(got2, 2 * want + 3, rtol=0, atol=1e-14)
    # eps enters under the root: var + eps = 1.25 + 3.75 = 5 -> (z - 2.5) / sqrt(5)
    got3 = oracle.layernorm(z, np.ones(4, np.float32), np.zeros(4, np.float32), 3.75)
    assert np.allclose(got3, (z.astype(np.float64) - 2.5) / math.sqrt(5.0), rtol=0, atol=1e-15)


def test_layernorm_invariants():
    rng = np.random.default_rng(61)
    # multiples of 2^-10 below 2^7: shifting by 64 and doubling stay exact in fp32
    z = (np.round((rng.normal(size=(5, 768)) * 7 + 3) * 1024) / 1024).astype(np.float32)
    g = rng.normal(size=768).astype(np.float32)
    b = rng.normal(size=768).astype(np.float32)
    ones, zeros = np.ones(768, np.float32), np.zeros(768, np.float32)
    norm = oracle.layernorm(z, ones, zeros, 0.0)
    assert np.allclose(norm.mean(axis=1), 0.0, atol=1e-12)             # zero mean
    assert np.allclose((norm ** 2).mean(axis=1), 1.0, atol=1e-12)      # unit variance
    # a constant row normalises to 0: the output is beta
    const = np.full((1, 768), 4.25, np.float32)
    assert np.array_equal(oracle.layernorm(const, g, b, 1e-5)[0], b.astype(np.float64))
    # shifting a row (exactly representable shift) changes nothing
    shifted = (z + np.float32(64.0)).astype(np.float32)
    assert np.allclose(oracle.layernorm(shifted, g, b, 1e-5), oracle.layernorm(z, g, b, 1e-5), atol=1e-9)
    # scaling a row by 2 (exact in fp32) changes nothing when eps = 0
    assert np.allclose(oracle.layernorm(z * np.float32(2), g, b, 0.0), oracle.layernorm(z, g, b, 0.0), atol=1e-12)


def test_linear_resid_hand_case_and_special_cases():
    """The residual add: z = fmaf((float)acc, s, b) + res_scale * (float)r,
    two fp32 operations."""
    # W 4x2 holding one block [1, -2, 3, 127] in column 0; x = [[-127, 5]]:
    # acc = [-127, 254, -381, -16129]
    w = np.zeros((4, 2), np.int8)
    w[:, 0] = [1, -2, 3, 127]
    x = np.array([[-127, 5]], np.int8)
    s = np.array([0.5, 0.25, 1.0, 0.125], np.float32)
    b = np.array([1, -1, 0.5, 2], np.float32)
    r = np.array([[4, -8, 0, 127]], np.int8)
    z = oracle.linear_resid(x, w, s, b, r, 0.25)
    # y = [-62.5, 62.5, -380.5, -2014.125]; 0.25 r = [1, -2, 0, 31.75]
    assert z.tolist() == [[-61.5, 60.5, -380.5, -1982.375]]
    rng = np.random.default_rng(62)
    wt = synth.draw_weight(rng, 64, 200, 0.8)
    wd = oracle.weight_dense(wt)
    xx = synth.draw_x(rng, 30, 200, "u127")
    zero = np.zeros((30, 64), np.int8)
    y = oracle.linear(xx, wd, wt.scales, wt.bias, oracle.F32)
    # r = 0: z is the fp32 dequantised value itself
    assert np.array_equal(oracle.linear_resid(xx, wd, wt.scales, wt.bias, zero, 0.5), y.astype(np.float32))
    # res_scale = 0: the same
    rr = synth.draw_x(rng, 30, 64, "u127")
    assert np.array_equal(oracle.linear_resid(xx, wd, wt.scales, wt.bias, rr, 0.0), y.astype(np.float32))
    # otherwise the exact sum rounded once more (both terms are fp32)
    z = oracle.linear_resid(xx, wd, wt.scales, wt.bias, rr, 0.03)
    rs = (np.float32(0.03) * rr.astype(np.float32)).astype(np.float32)
    assert np.array_equal(z, (y.astype(np.float32) + rs).astype(np.float32))


# ------------------------------------------------------- multi-head attention --

def _qkv_rows(q, k, v):
    """Token rows q | k | v (int8) from per-token lists."""
    return np.concatenate([np.asarray(q), np.asarray(k), np.asarray(v)], axis=1).astype(np.int8)


def test_attention_closed_form_two_keys():
    """One head of width 4, two tokens.  Token 0's query (1,1,1,1) meets keys
    0 and (1,1,1,1): scores 0 and 4 s^2 / sqrt(4) = 2 s^2.  With s^2 =
    ln(3) / 2 the weights are 1/4 and 3/4, so its context is
    s (v0 + 3 v1) / 4 (this fixes the 1/sqrt(hd) factor, the sign of the
    softmax and which values get mixed).  Token 1's query is 0: equal
    scores, the context is the mean s (v0 + v1) / 2."""
    s = np.float32(math.sqrt(math.log(3.0) / 2.0))
    v0, v1 = np.array([10, 0, -5, 3]), np.array([2, 8, 1, -7])
    qkv = _qkv_rows([[1, 1, 1, 1], [0, 0, 0, 0]], [[0, 0, 0, 0], [1, 1, 1, 1]], [v0, v1])
    got = oracle.attention_f64(qkv, s, 1, 2, heads=1)
    want0 = float(s) * (v0 + 3 * v1) / 4.0
    want1 = float(s) * (v0 + v1) / 2.0
    # the float rounding of s moves the weight 3 by ~1e-7 relative
    assert np.allclose(got[0], want0, rtol=0, atol=1e-6)
    assert np.allclose(got[1], want1, rtol=0, atol=1e-15)


def test_attention_max_subtraction_and_dominant_key():
    """hd = 64, scale 1: all queries and keys 127 give scores of 127^2 * 64
    / 8 = 129032 (exp overflows unless the row maximum is subtracted): equal
    scores, the context is the mean of the values.  A single key of +127
    among keys of -127 wins by 258064: the context is that key's value
    exactly (the other weights underflow to 0)."""
    rng = np.random.default_rng(63)
    seq = 5
    v = rng.integers(-127, 128, size=(seq, 64))
    qkv = _qkv_rows(np.full((seq, 64), 127), np.full((seq, 64), 127), v)
    got = oracle.attention_f64(qkv, 1.0, 1, seq, heads=1)
    assert np.all(np.isfinite(got))
    assert np.allclose(got, np.broadcast_to(v.mean(axis=0), (seq, 64)), rtol=0, atol=1e-12)
    k = np.full((seq, 64), -127)
    k[3] = 127
    qkv = _qkv_rows(np.full((seq, 64), 127), k, v)
    got = oracle.attention_f64(qkv, 1.0, 1, seq, heads=1)
    assert np.array_equal(got, np.broadcast_to(v[3].astype(np.float64), (seq, 64)))


def test_attention_single_token_is_its_value():
    rng = np.random.default_rng(64)
    qkv = rng.integers(-127, 128, size=(3, 3 * 2 * 64)).astype(np.int8)  # 3 sequences of 1 token, 2 heads
    got = oracle.attention_f64(qkv, 0.125, 3, 1, heads=2)
    assert np.array_equal(got, qkv[:, 2 * 128:].astype(np.float64) * 0.125)


def test_attention_permutation_equivariance_and_independence():
    """Permuting the tokens of a sequence permutes its context rows the same
    way; a head's context depends only on that head's columns of its own
    sequence."""
    rng = np.random.default_rng(65)
    batch, seq, heads, hd = 2, 7, 3, 8
    d = heads * hd
    qkv = rng.integers(-127, 128, size=(batch * seq, 3 * d)).astype(np.int8)
    base = oracle.attention_f64(qkv, 0.02, batch, seq, heads=heads)
    perm = rng.permutation(seq)
    pq = qkv.copy()
    pq[:seq] = qkv[perm]
    got = oracle.attention_f64(pq, 0.02, batch, seq, heads=heads)
    assert np.allclose(got[:seq], base[perm], rtol=1e-12, atol=1e-14)
    assert np.array_equal(got[seq:], base[seq:])
    # change head 1's queries, keys or values in sequence 0 only
    for part in range(3):
        cq = qkv.copy()
        cq[:seq, part * d + hd:part * d + 2 * hd] = rng.integers(-127, 128, size=(seq, hd))
        got = oracle.attention_f64(cq, 0.02, batch, seq, heads=heads)
        changed = np.abs(got - base) > 0
        assert changed[:seq, hd:2 * hd].any(), part
        changed[:seq, hd:2 * hd] = False
        assert not changed.any(), part


def test_attention_agrees_with_fp32_numpy_fixture():
    """The fp32 numpy attention (matmul + exp through numpy/BLAS, another
    implementation) lies within fp32 rounding of the fp64 oracle."""
    rng = np.random.default_rng(66)
    batch, seq = 2, 40
    qkv = rng.integers(-127, 128, size=(batch * seq, 3 * 768)).astype(np.int8)
    a = oracle.attention_f64(qkv, 0.01, batch, seq)
    b = oracle.attention_f32(qkv, 0.01, batch, seq)
    assert np.abs(a - b).max() <= 1e-5 * 127 * 0.01
    c = oracle.attention_f64(qkv, 0.01, batch, seq, threads=2)
    assert np.array_equal(a, c)


# ------------------------------------------------------------- 1 x 4 blocks --

def test_bsr1x4_hand_case_and_rejects():
    w = oracle.bsr1x4_to_dense(2, 8, [0, 1, 2], [1, 0], [[1, 2, 3, 4], [5, 6, 7, -8]])
    assert w.tolist() == [[0, 0, 0, 0, 1, 2, 3, 4], [5, 6, 7, -8, 0, 0, 0, 0]]
    ones = [[1, 1, 1, 1]] * 2
    for args in (([1, 1, 2], [0, 1]),       # indptr[0] != 0
                 ([0, 2, 1], [0, 1]),       # decreasing
                 ([0, 1, 2], [0, 2]),       # group = K / 4
                 ([0, 2, 2], [1, 1]),       # repeated group
                 ([0, 2, 2], [1, 0])):      # unsorted
        with pytest.raises(ValueError):
            oracle.bsr1x4_to_dense(2, 8, args[0], args[1], ones)
    with pytest.raises(ValueError):                       # K not a multiple of 4
        oracle.bsr1x4_to_dense(2, 6, [0, 0, 0], [], np.zeros((0, 4)))


def test_bsr1x4_is_the_transpose_of_4x1_blocks():
    """A 1 x 4 block of W (row n, columns 4j .. 4j+3) is a 4 x 1 block of
    W^T (rows 4j .. 4j+3, column n): re-indexed by group, the same arrays
    through the 4 x 1 decompression give W^T."""
    rng = np.random.default_rng(67)
    n, k = 10, 24
    keep = rng.random((n, k // 4)) < 0.4
    rows, grps = np.nonzero(keep)                          # row-major: by n, then j
    vals = rng.integers(-127, 128, size=(len(rows), 4)).astype(np.int8)
    indptr = np.concatenate([[0], np.cumsum(keep.sum(axis=1))]).astype(np.int32)
    w = oracle.bsr1x4_to_dense(n, k, indptr, grps.astype(np.int32), vals)
    order = np.lexsort((rows, grps))                       # by j, then n
    indptr_t = np.concatenate([[0], np.cumsum(np.bincount(grps, minlength=k // 4))]).astype(np.int32)
    wt = oracle.bsr_to_dense(k, n, indptr_t, rows[order].astype(np.int32), vals[order])
    assert np.array_equal(w, wt.T)
    # and the linear through it is the library's integer matmul
    x = rng.integers(-127, 128, size=(7, k)).astype(np.int8)
    acc = oracle.linear(x, w, np.ones(n, np.float32), np.zeros(n, np.float32), oracle.I32)
    assert np.array_equal(acc, x.astype(np.int64) @ w.astype(np.int64).T)


# ------------------------------------------------------------ 2:4 sparsity --

def test_2to4_hand_case_and_rejects():
    vals = np.array([[3, -4, 5, 6]], np.int8)
    idx = np.array([[0, 3, 1, 2]], np.uint8)
    w = oracle.sparse2to4_to_dense(vals, idx)
    assert w.tolist() == [[3, 0, 0, -4, 0, 5, 6, 0]]
    for bad in ([[1, 1, 0, 1]], [[2, 1, 0, 1]], [[0, 4, 0, 1]]):   # repeated, decreasing, out of range
        with pytest.raises(ValueError):
            oracle.sparse2to4_to_dense(vals, np.array(bad, np.uint8))


def test_2to4_structure_and_linear():
    """Every group of 4 columns holds at most 2 nonzeros and exactly the
    stored values; the linear through it is the library's integer matmul."""
    rng = np.random.default_rng(68)
    n, k = 12, 40
    pos = np.sort(np.stack([rng.choice(4, 2, replace=False) for _ in range(n * k // 4)]), axis=1)
    idx = pos.reshape(n, k // 2).astype(np.uint8)
    vals = rng.integers(-127, 128, size=(n, k // 2)).astype(np.int8)
    w = oracle.sparse2to4_to_dense(vals, idx)
    groups = w.reshape(n, k // 4, 4)
    assert ((groups != 0).sum(axis=2) <= 2).all()
    # the stored values sit at their positions
    got = np.take_along_axis(groups, idx.reshape(n, k // 4, 2).astype(np.int64), axis=2)
    assert np.array_equal(got.reshape(n, k // 2), vals)
    # the other two positions of each group are zero
    assert int(np.abs(groups.astype(np.int64)).sum()) == int(np.abs(vals.astype(np.int64)).sum())
    x = rng.integers(-127, 128, size=(9, k)).astype(np.int8)
    acc = oracle.linear(x, w, np.ones(n, np.float32), np.zeros(n, np.float32), oracle.I32)
    assert np.array_equal(acc, x.astype(np.int64) @ w.astype(np.int64).T)
