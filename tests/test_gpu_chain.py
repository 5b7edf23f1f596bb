"""One encoder layer's four linears chained on the GPU (QKV -> attention
reference step on the host -> attention output -> FFN1 + GELU -> FFN2,
int8 between, frozen calibrated scales) against the oracle's chain: every
stage bit-exact."""
import json
import os

import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

HERE = os.path.dirname(os.path.abspath(__file__))
KINDS = {"qkv": synth.I8, "attn_out": synth.I8, "ffn1": synth.I8_GELU, "ffn2": synth.I8}


@pytest.fixture(scope="module")
def bsg():
    import paper_2211_07715_gb300
    return paper_2211_07715_gb300


@pytest.fixture(scope="module")
def scales():
    with open(os.path.join(HERE, "golden", "layer_scales.json")) as f:
        return json.load(f)["scales"]


def gpu_chain(bsg, weights, x0: np.ndarray, s: dict, batch: int, seq: int) -> dict:
    """The chain with every linear on the device through the Python binding;
    only the attention step runs on the host."""
    lins = [bsg.SparseInt8Linear(w.n_out, w.k_in, w.indptr, w.colidx, w.values, w.scales, w.bias) for w in weights]
    out = {}
    x = torch.from_numpy(x0).cuda()
    qkv = lins[0](x, synth.I8, s["qkv"])
    out["qkv"] = qkv.cpu().numpy()
    ctx = oracle.attention(out["qkv"], s["qkv"], batch, seq, s["ctx"])
    out["ctx"] = ctx
    o = lins[1](torch.from_numpy(ctx).cuda(), synth.I8, s["attn_out"])
    f1 = lins[2](o, synth.I8_GELU, s["ffn1"])
    f2 = lins[3](f1, synth.I8, s["ffn2"])
    out["attn_out"], out["ffn1"], out["ffn2"] = o.cpu().numpy(), f1.cpu().numpy(), f2.cpu().numpy()
    for lin in lins:
        lin.close()
    return out


def compare(got: dict, want: dict, rows=slice(None)):
    for stage in oracle.CHAIN_STAGES:
        g, w = got[stage][rows], want[stage]
        diff = g != w
        assert not diff.any(), f"{stage}: {diff.sum()} of {diff.size} int8 values differ"


def test_chain_small_every_element(bsg, scales):
    # batch 2 x seq 64: the whole chain compared
    weights, x0 = synth.encoder_layer(m=128, seed=synth.SEED_BASE + 31)
    got = gpu_chain(bsg, weights, x0, scales, 2, 64)
    compare(got, oracle.layer_chain(x0, weights, scales, 2, 64))


def test_chain_full_size_every_sequence(bsg, scales):
    # the configuration's 8 x 384 tokens, every stage of every sequence
    batch, seq = 8, 384
    weights, x0 = synth.encoder_layer()
    got = gpu_chain(bsg, weights, x0, scales, batch, seq)
    compare(got, oracle.layer_chain(x0, weights, scales, batch, seq, threads=os.cpu_count() or 8))
