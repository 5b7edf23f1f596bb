"""Host-side arithmetic of bench.py's measurement objects (CPU only): the
attention kernel's floors and the DRAM traffic read from the committed ncu
summaries, which must follow the kernel source they were taken on."""
import os

import bench


def test_attention_floors_follow_their_definitions():
    """8 x 384 tokens, 12 heads of 64: 905,969,664 multiply-adds per
    product.  Tensor floor = 6 x that many flops at the given bf16 rate,
    exp floor = one exponential per score at 32 per SM per clock, HBM floor
    = the int8 QKV rows once; the largest one is the bound."""
    r = bench.attention_roofline(8, 384, 12, 0.0155, 152, 2070.0, 6783.5, 1903.9)
    macs = 8 * 12 * 384 * 384 * 64
    assert macs == 905_969_664
    assert r["ops"] == 4 * macs
    assert abs(r["floors_us"]["tensor"] - 6 * macs / 1903.9e12 * 1e6) < 1e-3
    assert abs(r["floors_us"]["exp"] - 8 * 12 * 384 * 384 / (152 * 32 * 2070e6) * 1e6) < 1e-3
    assert abs(r["floors_us"]["hbm"] - 8 * 384 * 2304 / 6783.5e9 * 1e6) < 1e-3
    assert r["bound"] == "tensor" and r["floor"] == "tensor"
    assert abs(r["frac"] - r["floors_us"]["tensor"] / 15.5) < 1e-3
    assert "mma_sync_floor_us" not in r  # the kernel runs on tcgen05, whose rate is the measured one
    # a slow exponential unit makes exp the bound
    r = bench.attention_roofline(8, 384, 12, 0.0155, 1, 2070.0, 6783.5, 1903.9)
    assert r["bound"] == "alu" and r["floor"] == "exp"


def test_profile_traffic_follows_the_kernel_source(tmp_path, monkeypatch):
    """The committed FFN2 summary gives its bytes while the sources hash to
    the recorded value; a summary taken on other sources gives None."""
    got = bench.profile_traffic("ffn2")
    text = open(os.path.join(bench.ROOT, "profiles", "ffn2_ncu.md")).read()
    if f"kernel_source_sha256: {bench.kernel_sha()}" in text:
        assert isinstance(got, int) and got > 0
    else:
        assert got is None
    sha = bench.kernel_sha()
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "x_ncu.md").write_text("kernel_source_sha256: 0000000000000000\ndram_bytes_per_launch: 5\n")
    (tmp_path / "profiles" / "y_ncu.md").write_text(f"kernel_source_sha256: {sha}\ndram_bytes_per_launch: 7\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_sha", lambda: sha)
    assert bench.profile_traffic("x") is None
    assert bench.profile_traffic("y") == 7
    assert bench.profile_traffic("missing") is None


def test_encoder_cpu_baseline_runs_the_oracle_layer():
    """One sequence through the oracle's whole layer: the value counts the
    four linears' effective ops over the measured time."""
    import json

    import numpy as np

    import synth
    with open(bench.LAYER_SCALES) as f:
        scales = json.load(f)["scales"]
    weights, x0 = synth.encoder_layer()
    g = np.ones(768, np.float32)
    z = np.zeros(768, np.float32)
    r = bench.encoder_cpu_baseline(weights, x0, scales, 384, g, z, g, z, 0.02, 4.0 / 127.0, 1e-12, threads=4, nseq=1)
    assert r["kind"] == "oracle" and r["cores"] == 4 and r["unit"] == bench.UNIT
    ops = sum(2.0 * 384 * w.nnzb * 4 for w in weights)
    dt = 384 / r["tokens_per_s"]
    assert abs(r["value"] - ops / dt / 1e12) <= 1e-3 * r["value"] + 1e-6
