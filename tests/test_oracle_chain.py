"""Pins of the encoder-layer chain's host pieces: the attention reference
step and the chain's calibration.  CPU only."""
import json
import os

import numpy as np
import pytest

import oracle
import synth

HERE = os.path.dirname(os.path.abspath(__file__))


def qkv_int8(rng, m, d=768):
    return rng.integers(-127, 128, size=(m, 3 * d)).astype(np.int8)


def test_attention_uniform_keys_average_the_values():
    # identical keys for every token -> equal weights -> each head's context
    # is the mean of its values over the sequence
    rng = np.random.default_rng(1)
    batch, seq, d = 2, 16, 768
    qkv = qkv_int8(rng, batch * seq)
    qkv[:, d:2 * d] = qkv[0, d:2 * d]
    ctx = oracle.attention_f32(qkv, 0.01, batch, seq)
    v = qkv[:, 2 * d:].astype(np.float64) * np.float32(0.01)
    want = v.reshape(batch, seq, d).mean(axis=1, keepdims=True).repeat(seq, axis=1).reshape(batch * seq, d)
    np.testing.assert_allclose(ctx, want, rtol=1e-5, atol=1e-6)


def test_attention_dominant_key_picks_its_value():
    # one key aligned with every query, the others orthogonal to it with a
    # gap of 100 in the scaled score: the softmax weight of the rest is e^-100
    batch, seq, d, hd = 1, 8, 768, 64
    qkv = np.zeros((seq, 3 * d), np.int8)
    qkv[:, :d] = 100                     # all queries
    qkv[3, d:2 * d] = 100                # token 3's key
    rng = np.random.default_rng(2)
    qkv[:, 2 * d:] = rng.integers(-127, 128, size=(seq, d)).astype(np.int8)
    scale = np.float32(np.sqrt(100.0 / (hd * 100 * 100 / 8.0)))  # score of token 3: 100
    ctx = oracle.attention_f32(qkv, scale, batch, seq)
    want = np.repeat(qkv[3:4, 2 * d:].astype(np.float32) * scale, seq, axis=0)
    np.testing.assert_allclose(ctx, want, rtol=1e-5, atol=1e-6)


def test_attention_sequences_are_independent():
    rng = np.random.default_rng(3)
    batch, seq = 3, 8
    qkv = qkv_int8(rng, batch * seq)
    a = oracle.attention_f32(qkv, 0.02, batch, seq)
    qkv2 = qkv.copy()
    qkv2[seq:2 * seq] = qkv_int8(rng, seq)  # change sequence 1 only
    b = oracle.attention_f32(qkv2, 0.02, batch, seq)
    assert np.array_equal(a[:seq], b[:seq]) and np.array_equal(a[2 * seq:], b[2 * seq:])
    assert not np.array_equal(a[seq:2 * seq], b[seq:2 * seq])


def test_attention_equals_float64_definition():
    rng = np.random.default_rng(4)
    batch, seq, heads, d = 2, 12, 12, 768
    hd = d // heads
    qkv = qkv_int8(rng, batch * seq)
    ctx = oracle.attention_f32(qkv, 0.003, batch, seq)
    x = qkv.astype(np.float64) * np.float64(np.float32(0.003))
    want = np.empty((batch * seq, d))
    for b in range(batch):
        rows = slice(b * seq, (b + 1) * seq)
        for h in range(heads):
            cols = slice(h * hd, (h + 1) * hd)
            q, k, v = x[rows, cols], x[rows, d:][:, cols], x[rows, 2 * d:][:, cols]
            s = q @ k.T / np.sqrt(hd)
            p = np.exp(s - s.max(axis=1, keepdims=True))
            want[rows, cols] = (p / p.sum(axis=1, keepdims=True)) @ v
    np.testing.assert_allclose(ctx, want, rtol=2e-5, atol=2e-6 * np.abs(want).max())


def test_requant_f32_rounds_half_to_even_and_saturates():
    y = np.array([2.5, 3.5, -2.5, -3.5, 1e6, -1e6, 0.49], np.float32)
    assert oracle.requant_f32(y, 1.0).tolist() == [2, 4, -2, -4, 127, -128, 0]


def test_calibrated_chain_reaches_full_int8_range():
    # small chain: calibration makes every stage's largest |value| 127
    weights, x0 = synth.encoder_layer(m=64)
    scales = oracle.calibrate_chain(x0, weights, 2, 32, threads=4)
    out = oracle.layer_chain(x0, weights, scales, 2, 32, threads=4)
    for stage in oracle.CHAIN_STAGES:
        assert np.abs(out[stage].astype(np.int32)).max() == 127, stage


def test_frozen_layer_scales_file():
    with open(os.path.join(HERE, "golden", "layer_scales.json")) as f:
        doc = json.load(f)
    assert set(doc["scales"]) == set(oracle.CHAIN_STAGES)
    assert all(np.float32(v) == v and v > 0 for v in doc["scales"].values())
    assert doc["batch"] * doc["seq"] == 3072
