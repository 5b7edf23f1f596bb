"""Seeded synthetic inputs with the shapes of the DistilBERT linears.

This module only draws random numbers.  It holds none of the method's
arithmetic: it emits the block-compressed weight arrays (indptr, colidx,
values), the int8 activations and the per-channel scales/bias exactly as
sampled.  Both the CUDA path and the CPU oracle consume these arrays; the
oracle decompresses them itself.

The paper measures on SQuADv1.1 through a pruned, quantised DistilBERT
(Sec. 4).  Neither the dataset nor the trained weights are available, so
seeded tensors of the same shapes stand in for them:
  * weights: blocks of 4 output rows x 1 input column (App. A.1); a fraction
    `sparsity` of all blocks is zero, the zero blocks chosen uniformly
    without replacement; stored block values uniform integers in [-127, 127];
  * activations: uniform in [-127, 127], clip(rint(N(0, 30))), or uniform in
    [0, 127], per workload;
  * scales uniform in [1e-3, 1e-2] (fp32), bias ~ N(0, 0.02) (fp32).

RNG: numpy Generator(PCG64(seed)); draw order per linear layer: block
positions, block values, scales, bias; activations are drawn after all
layers' weights.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

BLOCK = 4
SEED_BASE = 2211077150

# output kinds (same numbering as the library's public header)
I32, F32, F32_GELU, I8, I8_GELU = 0, 1, 2, 3, 4
KIND_NAMES = {I32: "i32", F32: "f32", F32_GELU: "f32_gelu", I8: "i8", I8_GELU: "i8_gelu"}


def rng_for(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def n_nonzero_blocks(n_out: int, k_in: int, sparsity: float) -> int:
    """Number of stored blocks: total - round(sparsity * total), halves up."""
    total = (n_out // BLOCK) * k_in
    pruned = int(np.floor(sparsity * total + 0.5))
    return total - min(max(pruned, 0), total)


@dataclass
class BsrWeight:
    n_out: int
    k_in: int
    indptr: np.ndarray  # int32 [N/4 + 1]
    colidx: np.ndarray  # int32 [nnzb]
    values: np.ndarray  # int8  [nnzb, 4]
    scales: np.ndarray  # float32 [N]
    bias: np.ndarray    # float32 [N]

    @property
    def nnzb(self) -> int:
        return int(self.colidx.shape[0])

    def indices(self) -> np.ndarray:
        """indptr followed by colidx, the layout the C entry point takes."""
        return np.concatenate([self.indptr, self.colidx]).astype(np.int32)


def draw_weight(rng: np.random.Generator, n_out: int, k_in: int, sparsity: float,
                value_lo: int = -127, value_hi: int = 127) -> BsrWeight:
    if n_out % BLOCK:
        raise ValueError("n_out must be a multiple of 4")
    nbr = n_out // BLOCK
    total = nbr * k_in
    nnzb = n_nonzero_blocks(n_out, k_in, sparsity)
    if nnzb == total:
        ids = np.arange(total, dtype=np.int64)
    else:
        ids = np.sort(rng.choice(total, size=nnzb, replace=False))
    rows = ids // k_in
    colidx = (ids % k_in).astype(np.int32)
    indptr = np.zeros(nbr + 1, dtype=np.int32)
    np.cumsum(np.bincount(rows, minlength=nbr), out=indptr[1:])
    values = rng.integers(value_lo, value_hi + 1, size=(nnzb, BLOCK), dtype=np.int64).astype(np.int8)
    scales = rng.uniform(1e-3, 1e-2, size=n_out).astype(np.float32)
    bias = rng.normal(0.0, 0.02, size=n_out).astype(np.float32)
    return BsrWeight(n_out, k_in, indptr, colidx, values, scales, bias)


def draw_x(rng: np.random.Generator, m: int, k_in: int, dist: str) -> np.ndarray:
    if dist == "u127":      # uniform integers in [-127, 127]
        x = rng.integers(-127, 128, size=(m, k_in), dtype=np.int64)
    elif dist == "n30":     # clip(rint(N(0, 30)), -127, 127)
        x = np.clip(np.rint(rng.normal(0.0, 30.0, size=(m, k_in))), -127, 127)
    elif dist == "u0_127":  # uniform integers in [0, 127]
        x = rng.integers(0, 128, size=(m, k_in), dtype=np.int64)
    elif dist == "extreme":  # only -128 and 127, the largest magnitudes
        x = np.where(rng.integers(0, 2, size=(m, k_in)) == 0, -128, 127)
    else:
        raise ValueError(dist)
    return np.ascontiguousarray(x.astype(np.int8))


@dataclass
class LinearCase:
    """One linear layer workload: weights, activations and the epilogue."""
    name: str
    weight: BsrWeight
    x: np.ndarray
    kind: int
    out_scale: float = 1.0
    meta: dict = field(default_factory=dict)

    @property
    def m(self) -> int:
        return int(self.x.shape[0])


def linear_case(name: str, n_out: int, k_in: int, m: int, sparsity: float, x_dist: str,
                kind: int, out_scale: float = 1.0, seed: int = SEED_BASE) -> LinearCase:
    rng = rng_for(seed)
    w = draw_weight(rng, n_out, k_in, sparsity)
    x = draw_x(rng, m, k_in, x_dist)
    return LinearCase(name, w, x, kind, out_scale,
                      {"sparsity": sparsity, "x_dist": x_dist, "seed": seed})


# The five DistilBERT-shaped workloads (hidden 768, FFN 3072, 12 heads).
def single_768(m: int = 128) -> LinearCase:
    """768x768 at 90% block sparsity, batch 1 x seq 128, fp32 dequantised."""
    return linear_case("single_768x768_s90_m128", 768, 768, m, 0.90, "u127", F32, seed=SEED_BASE + 0)


def ffn1(m: int = 4096) -> LinearCase:
    """FFN1 768->3072 at 80%, 32 x 128 tokens, bias + GELU, fp32 output."""
    return linear_case("ffn1_768to3072_s80_m4096", 3072, 768, m, 0.80, "n30", F32_GELU, seed=SEED_BASE + 1)


def ffn2(m: int = 4096) -> LinearCase:
    """FFN2 3072->768 at 90%, 32 x 128 tokens, bias + requantise (scale 0.05)."""
    return linear_case("ffn2_3072to768_s90_m4096", 768, 3072, m, 0.90, "u0_127", I8, out_scale=0.05,
                       seed=SEED_BASE + 2)


# Encoder-layer chain: QKV, attention output, FFN1 (+GELU), FFN2, int8 between.
LAYER_LINEARS = (("qkv", 2304, 768, I8), ("attn_out", 768, 768, I8),
                 ("ffn1", 3072, 768, I8_GELU), ("ffn2", 768, 3072, I8))


def layer_weights(rng: np.random.Generator, sparsity: float) -> list[BsrWeight]:
    return [draw_weight(rng, n, k, sparsity) for (_, n, k, _) in LAYER_LINEARS]


def encoder_layer(m: int = 3072, sparsity: float = 0.80, seed: int = SEED_BASE + 3):
    """Weights of one encoder layer's four linears and the layer input."""
    rng = rng_for(seed)
    ws = layer_weights(rng, sparsity)
    x0 = draw_x(rng, m, 768, "u127")
    return ws, x0


def stack_point(batch: int, seq: int, sparsity: float, point: int, n_layers: int = 6):
    """Six encoder layers' weights, the stack input and a seeded int8 context
    buffer that stands in for the attention output in the timed stack."""
    rng = rng_for(SEED_BASE + 4 + 100 * point)
    layers = [layer_weights(rng, sparsity) for _ in range(n_layers)]
    m = batch * seq
    x0 = draw_x(rng, m, 768, "u127")
    ctx = draw_x(rng, m, 768, "u127")
    return layers, x0, ctx


STACK_POINTS = [(b, s, sp) for b in (1, 8, 32, 128) for s in (128, 384) for sp in (0.70, 0.80, 0.90)]


# ----------------------------------------------------- variant block shapes --

@dataclass
class Blocks1x4:
    """A weight sparse in 1 x 4 blocks (one output row x 4 consecutive input
    columns): row n holds blocks indptr[n] .. indptr[n+1]-1, block e covers
    columns 4 colgrp[e] .. 4 colgrp[e] + 3 with values[e][0..3]."""
    n_out: int
    k_in: int
    indptr: np.ndarray  # int32 [N + 1]
    colgrp: np.ndarray  # int32 [nnz]
    values: np.ndarray  # int8  [nnz, 4]
    scales: np.ndarray  # float32 [N]
    bias: np.ndarray    # float32 [N]


def draw_weight_1x4(rng: np.random.Generator, n_out: int, k_in: int, sparsity: float) -> Blocks1x4:
    """round(sparsity * total) of the N x K/4 blocks zero, chosen uniformly
    without replacement; values uniform in [-127, 127]; scales and bias as
    draw_weight's.  Draw order: positions, values, scales, bias."""
    if k_in % 4:
        raise ValueError("k_in must be a multiple of 4")
    total = n_out * (k_in // 4)
    pruned = min(max(int(np.floor(sparsity * total + 0.5)), 0), total)
    nnz = total - pruned
    ids = np.arange(total, dtype=np.int64) if nnz == total else np.sort(rng.choice(total, size=nnz, replace=False))
    rows = ids // (k_in // 4)
    indptr = np.zeros(n_out + 1, dtype=np.int32)
    np.cumsum(np.bincount(rows, minlength=n_out), out=indptr[1:])
    colgrp = (ids % (k_in // 4)).astype(np.int32)
    values = rng.integers(-127, 128, size=(nnz, 4)).astype(np.int8)
    scales = rng.uniform(1e-3, 1e-2, size=n_out).astype(np.float32)
    bias = rng.normal(0.0, 0.02, size=n_out).astype(np.float32)
    return Blocks1x4(n_out, k_in, indptr, colgrp, values, scales, bias)


@dataclass
class Sparse2to4:
    """A 2:4-sparse weight: per output row and group of 4 input columns, two
    values at in-group positions idx (ascending)."""
    n_out: int
    k_in: int
    values: np.ndarray  # int8  [N, K/2]
    idx: np.ndarray     # uint8 [N, K/2]
    scales: np.ndarray  # float32 [N]
    bias: np.ndarray    # float32 [N]


def draw_weight_2to4(rng: np.random.Generator, n_out: int, k_in: int) -> Sparse2to4:
    """Each group's two positions uniform among the 6 pairs, values uniform
    in [-127, 127]; scales and bias as draw_weight's.  Draw order:
    positions, values, scales, bias."""
    if k_in % 4:
        raise ValueError("k_in must be a multiple of 4")
    pairs = np.array([(a, b) for a in range(4) for b in range(a + 1, 4)], dtype=np.uint8)
    pick = rng.integers(0, len(pairs), size=(n_out, k_in // 4))
    idx = pairs[pick].reshape(n_out, k_in // 2)
    values = rng.integers(-127, 128, size=(n_out, k_in // 2)).astype(np.int8)
    scales = rng.uniform(1e-3, 1e-2, size=n_out).astype(np.float32)
    bias = rng.normal(0.0, 0.02, size=n_out).astype(np.float32)
    return Sparse2to4(n_out, k_in, values, idx, scales, bias)
