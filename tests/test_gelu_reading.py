"""The cost of the int8-GELU reading, counted on CPU with the oracle alone.

The paper fixes no GELU evaluation (App. A.3.3 names the fused
post-operators, not how they are computed).  For int8 outputs both sides
evaluate erf by Abramowitz & Stegun 7.1.28 as one fixed fp32 operation
sequence (bit-exact between them), so an int8 output can differ from the
ideal rne(GELU(y) / out_scale) of the exact erf.  These tests count such
outputs on the FFN1 configuration's seeded inputs and check that each one
is explained by the approximation: |q_spec - q_exact| = 1 and the exact
value t = GELU(y) * inv lies within the error bound of the rounding
boundary between the two codes.

Bound on |t_spec - t| (before rounding to an integer): the fp32 GELU is
within 1.2e-6 |y| + 1e-12 of GELU(y) (pinned in test_oracle_pins.py), and
the fp32 multiply by inv adds at most half an ulp of the product, 2^-24 |t|.
"""
import os

import numpy as np
import pytest

import oracle
import synth

scipy_special = pytest.importorskip("scipy.special")


def _y32(acc: np.ndarray, scales: np.ndarray, bias: np.ndarray) -> np.ndarray:
    """fmaf((float)acc, s, b) for every element, exactly: the product of two
    fp32 values is exact in fp64, the sum is split into hi + lo by TwoSum,
    and hi rounds to the same fp32 as hi + lo unless hi is itself a midpoint
    of the fp32 grid (those few elements go through the oracle's own
    dequantisation)."""
    p = acc.astype(np.float32).astype(np.float64) * scales.astype(np.float64)[None, :]
    b = np.broadcast_to(bias.astype(np.float64)[None, :], p.shape)
    hi = p + b
    bb = hi - p
    lo = (p - (hi - bb)) + (b - bb)
    y = hi.astype(np.float32)
    yd = y.astype(np.float64)
    other = np.where(yd < hi, np.nextafter(y, np.float32(np.inf)), np.nextafter(y, np.float32(-np.inf)))
    mid = (lo != 0) & (np.abs(hi - yd) == np.abs(other.astype(np.float64) - hi))
    for m, n in zip(*np.nonzero(mid)):
        y[m, n] = oracle.dequant_f32(int(acc[m, n]), float(scales[n]), float(bias[n]))
    return y


def _count_against_exact_erf(y: np.ndarray, q_spec: np.ndarray, out_scale: float):
    inv = np.float32(1.0) / np.float32(out_scale)
    yd = y.astype(np.float64)
    t = 0.5 * yd * (1.0 + scipy_special.erf(yd / np.sqrt(2.0))) * np.float64(inv)
    q_exact = np.clip(np.rint(t), -128, 127).astype(np.int64)
    differ = q_spec.astype(np.int64) != q_exact
    idx = np.nonzero(differ)
    if idx[0].size:
        qs, qe, td = q_spec[idx].astype(np.int64), q_exact[idx], t[idx]
        assert np.all(np.abs(qs - qe) == 1), "an int8 GELU output is more than one code away from the exact one"
        boundary = (qs + qe) / 2.0
        bound = (1.2e-6 * np.abs(yd[idx]) + 1e-12) * float(inv) + 2.0 ** -24 * np.abs(td) + 1e-12
        assert np.all(np.abs(td - boundary) <= bound), "a differing output lies farther from the boundary than the bound"
    return int(differ.sum()), int(differ.size)


def test_ffn1_int8_gelu_differs_from_exact_erf_only_at_rounding_boundaries():
    """FFN1 (768 -> 3072, 80%, M = 4096, its seeded N(0, 30) activations),
    requantised after GELU with the post-training scale max |GELU(y)| / 127
    (the calibration the chain uses) and with a finer scale (a quarter of
    it, saturating the largest outputs), so that more codes are decided."""
    case = synth.ffn1()
    wt = case.weight
    w = oracle.weight_dense(wt)
    threads = os.cpu_count() or 8
    acc = oracle.linear(case.x, w, wt.scales, wt.bias, synth.I32, threads=threads)
    sc, bi = np.asarray(wt.scales, np.float32), np.asarray(wt.bias, np.float32)
    y = _y32(acc, sc, bi)
    rng = np.random.default_rng(5)
    for m, n in zip(rng.integers(0, y.shape[0], 2000), rng.integers(0, y.shape[1], 2000)):
        assert y[m, n] == oracle.dequant_f32(int(acc[m, n]), float(sc[n]), float(bi[n]))
    g = oracle.linear(case.x, w, wt.scales, wt.bias, synth.F32_GELU, threads=threads)
    calib = float(np.float32(np.max(np.abs(g))) / np.float32(127.0))
    counts = {}
    for name, s in (("calibrated", calib), ("quarter", calib / 4)):
        q_spec = oracle.linear(case.x, w, wt.scales, wt.bias, synth.I8_GELU, out_scale=s, threads=threads)
        counts[name] = _count_against_exact_erf(y, q_spec, s)
    print("int8 GELU outputs that differ from rne(GELU_exact(y) / out_scale):", counts)
    for n_diff, total in counts.values():
        # the A&S error is ~1e-6 |y| against code steps of 1: a few per million
        assert n_diff <= total * 1e-4
