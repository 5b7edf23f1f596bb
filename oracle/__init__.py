"""CPU oracle for the block-sparse INT8 linear layer (ctypes front end).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the
benchmark's CPU-baseline leg may import this package; the library and its
Python binding never do.  The arithmetic lives in ``bsgemm_oracle.c``, a
plain triple loop over the decompressed weights followed by the epilogue;
every function there cites the passage of arXiv 2211.07715 it follows.

ctypes releases the GIL during a foreign call, so ``linear(...,
threads=n)`` runs row ranges on n host threads.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bsgemm_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

I32, F32, F32_GELU, I8, I8_GELU = 0, 1, 2, 3, 4
BLOCK = 4


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (IEEE fp32: no contraction, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                               "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            i8p = ctypes.POINTER(ctypes.c_int8)
            i32p = ctypes.POINTER(ctypes.c_int32)
            u8p = ctypes.POINTER(ctypes.c_uint8)
            f32p = ctypes.POINTER(ctypes.c_float)
            c_int, c_float, c_double = ctypes.c_int, ctypes.c_float, ctypes.c_double
            lib.oracle_bsr_to_dense.argtypes = [c_int, c_int, i32p, i32p, i8p, i8p]
            lib.oracle_bsr_to_dense.restype = c_int
            lib.oracle_dense_to_bsr.argtypes = [c_int, c_int, i8p, u8p, i32p, i32p, i8p]
            lib.oracle_dense_to_bsr.restype = c_int
            lib.oracle_acc.argtypes = [c_int, c_int, c_int, i8p, i8p, i32p, c_int, c_int]
            lib.oracle_acc.restype = c_int
            lib.oracle_dequant_f32.argtypes = [ctypes.c_int32, c_float, c_float]
            lib.oracle_dequant_f32.restype = c_float
            lib.oracle_dequant_f64.argtypes = [ctypes.c_int32, c_float, c_float]
            lib.oracle_dequant_f64.restype = c_double
            lib.oracle_gelu_f64.argtypes = [c_double]
            lib.oracle_gelu_f64.restype = c_double
            lib.oracle_gelu_f32.argtypes = [c_float]
            lib.oracle_gelu_f32.restype = c_float
            lib.oracle_recip_f32.argtypes = [c_float]
            lib.oracle_recip_f32.restype = c_float
            lib.oracle_requant.argtypes = [c_float, c_float]
            lib.oracle_requant.restype = ctypes.c_int8
            lib.oracle_linear.argtypes = [c_int, c_int, c_int, i8p, i8p, f32p, f32p, c_int, c_float,
                                          ctypes.c_void_p, c_int, c_int]
            lib.oracle_linear.restype = c_int
            lib.oracle_block_prune.argtypes = [c_int, c_int, f32p, c_double, u8p]
            lib.oracle_linear_resid.argtypes = [c_int, c_int, c_int, i8p, i8p, f32p, f32p, i8p, c_float, f32p,
                                                c_int, c_int]
            lib.oracle_linear_resid.restype = c_int
            lib.oracle_layernorm.argtypes = [c_int, c_int, f32p, f32p, f32p, c_double,
                                             ctypes.POINTER(c_double)]
            lib.oracle_layernorm.restype = None
            lib.oracle_block_prune.restype = ctypes.c_int64
            lib.oracle_attention.argtypes = [c_int, c_int, c_int, c_int, i8p, c_int, c_float,
                                             ctypes.POINTER(c_double)]
            lib.oracle_attention.restype = c_int
            lib.oracle_bsr1x4_to_dense.argtypes = [c_int, c_int, i32p, i32p, i8p, i8p]
            lib.oracle_bsr1x4_to_dense.restype = c_int
            lib.oracle_2to4_to_dense.argtypes = [c_int, c_int, i8p, u8p, i8p]
            lib.oracle_2to4_to_dense.restype = c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# --- block-compressed format (App. A.1, App. A.3.4) ----------------------

def bsr_to_dense(n_out: int, k_in: int, indptr, colidx, values) -> np.ndarray:
    lib = _load()
    indptr, colidx = _c(indptr, np.int32), _c(colidx, np.int32)
    values = _c(values, np.int8).reshape(-1)
    w = np.empty((n_out, k_in), dtype=np.int8)
    rc = lib.oracle_bsr_to_dense(n_out, k_in, _ptr(indptr, ctypes.c_int32), _ptr(colidx, ctypes.c_int32),
                                 _ptr(values, ctypes.c_int8), _ptr(w, ctypes.c_int8))
    if rc:
        raise ValueError("invalid block-compressed arrays")
    return w


def bsr1x4_to_dense(n_out: int, k_in: int, indptr, colgrp, values) -> np.ndarray:
    """Dense int8 W [N][K] of a weight sparse in 1 x 4 blocks (one output
    row x 4 consecutive input columns; block e of row n covers columns
    4 colgrp[e] .. 4 colgrp[e] + 3)."""
    lib = _load()
    indptr, colgrp = _c(indptr, np.int32), _c(colgrp, np.int32)
    values = _c(values, np.int8).reshape(-1)
    w = np.empty((n_out, k_in), dtype=np.int8)
    rc = lib.oracle_bsr1x4_to_dense(n_out, k_in, _ptr(indptr, ctypes.c_int32), _ptr(colgrp, ctypes.c_int32),
                                    _ptr(values, ctypes.c_int8), _ptr(w, ctypes.c_int8))
    if rc:
        raise ValueError("invalid 1x4 block arrays")
    return w


def sparse2to4_to_dense(values, idx) -> np.ndarray:
    """Dense int8 W [N][K] of a 2:4-sparse weight: values and idx [N][K/2],
    two values per group of 4 input columns at in-group positions idx
    (strictly increasing per group)."""
    lib = _load()
    values, idx = _c(values, np.int8), _c(idx, np.uint8)
    n_out, half = values.shape
    if idx.shape != values.shape:
        raise ValueError("values and idx must have the same shape")
    w = np.empty((n_out, 2 * half), dtype=np.int8)
    if lib.oracle_2to4_to_dense(n_out, 2 * half, _ptr(values, ctypes.c_int8), _ptr(idx, ctypes.c_uint8),
                                _ptr(w, ctypes.c_int8)):
        raise ValueError("invalid 2:4 arrays")
    return w


def dense_to_bsr(w: np.ndarray, mask: np.ndarray):
    lib = _load()
    w = _c(w, np.int8)
    n_out, k_in = w.shape
    mask = _c(mask != 0, np.uint8)
    indptr = np.empty(n_out // BLOCK + 1, dtype=np.int32)
    nnzb = lib.oracle_dense_to_bsr(n_out, k_in, _ptr(w, ctypes.c_int8), _ptr(mask, ctypes.c_uint8),
                                   _ptr(indptr, ctypes.c_int32), None, None)
    colidx = np.empty(nnzb, dtype=np.int32)
    values = np.empty((nnzb, BLOCK), dtype=np.int8)
    lib.oracle_dense_to_bsr(n_out, k_in, _ptr(w, ctypes.c_int8), _ptr(mask, ctypes.c_uint8),
                            _ptr(indptr, ctypes.c_int32), _ptr(colidx, ctypes.c_int32),
                            _ptr(values, ctypes.c_int8))
    return indptr, colidx, values


def weight_dense(wt) -> np.ndarray:
    """Decompress a synth.BsrWeight."""
    return bsr_to_dense(wt.n_out, wt.k_in, wt.indptr, wt.colidx, wt.values)


# --- accumulation and epilogue (Sec. 3, Algorithm 1, App. A.3.3) ---------

def acc(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    lib = _load()
    x, w = _c(x, np.int8), _c(w, np.int8)
    m, k_in = x.shape
    n_out = w.shape[0]
    out = np.empty((m, n_out), dtype=np.int32)
    rc = lib.oracle_acc(m, n_out, k_in, _ptr(x, ctypes.c_int8), _ptr(w, ctypes.c_int8),
                        _ptr(out, ctypes.c_int32), 0, m)
    if rc:
        raise OverflowError("accumulator leaves the int32 range")
    return out


def dequant_f32(a: int, scale: float, bias: float) -> np.float32:
    return np.float32(_load().oracle_dequant_f32(int(a), float(scale), float(bias)))


def dequant_f64(a: int, scale: float, bias: float) -> float:
    return _load().oracle_dequant_f64(int(a), float(scale), float(bias))


def gelu_f32(y: float) -> np.float32:
    return np.float32(_load().oracle_gelu_f32(float(np.float32(y))))


def recip_f32(b: float) -> np.float32:
    """1/b (1 <= b < 2^25) by the fixed Newton-Raphson fp32 sequence that
    the int8 GELU uses."""
    return np.float32(_load().oracle_recip_f32(float(np.float32(b))))


def gelu_f64(y: float) -> float:
    return _load().oracle_gelu_f64(float(y))


def requant(v: float, inv_out_scale: float) -> int:
    return int(_load().oracle_requant(float(np.float32(v)), float(np.float32(inv_out_scale))))


def out_dtype(kind: int):
    return {I32: np.int32, F32: np.float64, F32_GELU: np.float64, I8: np.int8, I8_GELU: np.int8}[kind]


def linear(x: np.ndarray, w: np.ndarray, scales, bias, kind: int, out_scale: float = 1.0,
           rows=None, threads: int = 1) -> np.ndarray:
    """The whole layer on rows `rows` of x (all rows if None).

    Output dtype by kind: I32 -> int32, F32/F32_GELU -> float64 (exact-valued
    reference), I8/I8_GELU -> int8 decided in fp32.
    """
    lib = _load()
    w = _c(w, np.int8)
    n_out, k_in = w.shape
    x = _c(x, np.int8)
    if rows is not None:
        x = np.ascontiguousarray(x[np.asarray(rows, dtype=np.int64)])
    m = x.shape[0]
    scales = _c(scales, np.float32)
    bias_arr = None if bias is None else _c(bias, np.float32)
    out = np.empty((m, n_out), dtype=out_dtype(kind))

    def run(r0, r1):
        return lib.oracle_linear(m, n_out, k_in, _ptr(x, ctypes.c_int8), _ptr(w, ctypes.c_int8),
                                 _ptr(scales, ctypes.c_float),
                                 None if bias_arr is None else _ptr(bias_arr, ctypes.c_float),
                                 kind, float(out_scale), out.ctypes.data_as(ctypes.c_void_p), r0, r1)

    threads = max(1, min(int(threads), m))
    if threads == 1:
        rcs = [run(0, m)]
    else:
        bounds = [m * i // threads for i in range(threads + 1)]
        with ThreadPoolExecutor(threads) as ex:
            rcs = list(ex.map(lambda i: run(bounds[i], bounds[i + 1]), range(threads)))
    for rc in rcs:
        if rc == -1:
            raise ValueError("bad kind or out_scale")
        if rc == -2:
            raise OverflowError("accumulator leaves the int32 range")
        if rc:
            raise RuntimeError(f"oracle_linear failed ({rc})")
    return out


def linear_resid(x: np.ndarray, w: np.ndarray, scales, bias, residual: np.ndarray, res_scale: float,
                 threads: int = 1) -> np.ndarray:
    """z = fmaf((float)acc, scale, bias) + res_scale * (float)residual, in
    fp32 op by op (the residual add before LayerNorm); float32 [M][N]."""
    lib = _load()
    w = _c(w, np.int8)
    n_out, k_in = w.shape
    x = _c(x, np.int8)
    m = x.shape[0]
    residual = _c(residual, np.int8)
    if residual.shape != (m, n_out):
        raise ValueError("residual must be [M][N]")
    scales = _c(scales, np.float32)
    bias_arr = None if bias is None else _c(bias, np.float32)
    out = np.empty((m, n_out), dtype=np.float32)

    def run(r0, r1):
        return lib.oracle_linear_resid(m, n_out, k_in, _ptr(x, ctypes.c_int8), _ptr(w, ctypes.c_int8),
                                       _ptr(scales, ctypes.c_float),
                                       None if bias_arr is None else _ptr(bias_arr, ctypes.c_float),
                                       _ptr(residual, ctypes.c_int8), float(np.float32(res_scale)),
                                       _ptr(out, ctypes.c_float), r0, r1)

    threads = max(1, min(int(threads), m))
    bounds = [m * i // threads for i in range(threads + 1)]
    if threads == 1:
        rcs = [run(0, m)]
    else:
        with ThreadPoolExecutor(threads) as ex:
            rcs = list(ex.map(lambda i: run(bounds[i], bounds[i + 1]), range(threads)))
    for rc in rcs:
        if rc == -2:
            raise OverflowError("accumulator leaves the int32 range")
        if rc:
            raise RuntimeError(f"oracle_linear_resid failed ({rc})")
    return out


def layernorm(z: np.ndarray, gamma, beta, eps: float) -> np.ndarray:
    """LayerNorm of each row of the fp32 z [M][N] in fp64 (float64 [M][N])."""
    lib = _load()
    z = _c(z, np.float32)
    m, n = z.shape
    gamma = _c(gamma, np.float32)
    beta = _c(beta, np.float32)
    out = np.empty((m, n), dtype=np.float64)
    lib.oracle_layernorm(m, n, _ptr(z, ctypes.c_float), _ptr(gamma, ctypes.c_float), _ptr(beta, ctypes.c_float),
                         float(eps), out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return out


def block_prune(w: np.ndarray, sparsity: float) -> np.ndarray:
    """Keep-mask [N/4][K] of the average-magnitude block pruning (App. A.1)."""
    lib = _load()
    w = _c(w, np.float32)
    n_out, k_in = w.shape
    keep = np.empty((n_out // BLOCK, k_in), dtype=np.uint8)
    lib.oracle_block_prune(n_out, k_in, _ptr(w, ctypes.c_float), float(sparsity), _ptr(keep, ctypes.c_uint8))
    return keep.astype(bool)


# ------------------------------------------------------------------ encoder layer chain --
# The layer chain of the DistilBERT encoder: QKV, attention, output
# projection, FFN1 (+GELU), FFN2, int8 between the linears (Sec. 3; the
# paper's engine quantises every linear, Sec. 2).  Attention itself is not
# part of the sparse linear; it is the plain reference step below, run on
# the host between the QKV and output linears of both chains.  Residual
# connections and LayerNorm are omitted.

HEADS = 12


def requant_f32(y: np.ndarray, out_scale) -> np.ndarray:
    """fp32 -> int8: multiply by the fp32 reciprocal of the scale, round half
    to even, saturate -- the same requantisation as the linears' epilogue."""
    inv = np.float32(1.0) / np.float32(out_scale)
    t = (np.asarray(y, dtype=np.float32) * inv).astype(np.float32)
    return np.clip(np.rint(t), -128, 127).astype(np.int8)


def attention_f32(qkv: np.ndarray, qkv_scale, batch: int, seq: int, heads: int = HEADS) -> np.ndarray:
    """Multi-head self-attention in fp32 on an int8 QKV output [M][3d],
    M = batch x seq: q, k, v are its dequantised thirds (int8 x qkv_scale);
    per sequence and head (d / heads wide) P = softmax(q k^T / sqrt(d /
    heads)) with the row maximum subtracted, context = P v.  Returns the
    context [M][d] in fp32."""
    m, d3 = qkv.shape
    assert m == batch * seq and d3 % 3 == 0
    d = d3 // 3
    hd = d // heads
    x = qkv.astype(np.float32) * np.float32(qkv_scale)

    def split(part):  # [M][d] -> [batch][heads][seq][hd]
        return np.ascontiguousarray(part.reshape(batch, seq, heads, hd).transpose(0, 2, 1, 3))

    q, k, v = split(x[:, :d]), split(x[:, d:2 * d]), split(x[:, 2 * d:])
    s = np.matmul(q, k.transpose(0, 1, 3, 2)) * np.float32(1.0 / np.sqrt(hd))
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s, dtype=np.float32)
    p = p / p.sum(axis=-1, keepdims=True, dtype=np.float32)
    ctx = np.matmul(p, v)  # [batch][heads][seq][hd]
    return np.ascontiguousarray(ctx.transpose(0, 2, 1, 3).reshape(m, d)).astype(np.float32)


def attention_f64(qkv: np.ndarray, qkv_scale, batch: int, seq: int, heads: int = HEADS, head_dim: int = None,
                  threads: int = 1) -> np.ndarray:
    """Multi-head self-attention in fp64 (the C oracle's oracle_attention):
    the context [batch * seq][heads * head_dim] of the int8 QKV rows
    [batch * seq][>= 3 * heads * head_dim] (q | k | v), dequantised by
    qkv_scale.  head_dim defaults to a third of the row width / heads.
    threads > 1 runs sequences on that many host threads."""
    lib = _load()
    qkv = _c(qkv, np.int8)
    m, ld = qkv.shape
    assert m == batch * seq
    if head_dim is None:
        assert ld % (3 * heads) == 0
        head_dim = ld // (3 * heads)
    d = heads * head_dim
    out = np.empty((m, d), dtype=np.float64)
    if m == 0:
        return out
    dp = ctypes.POINTER(ctypes.c_double)

    def run(b0, b1):
        if b1 <= b0:
            return 0
        q = qkv[b0 * seq:b1 * seq]
        o = out[b0 * seq:b1 * seq]
        return lib.oracle_attention(b1 - b0, seq, heads, head_dim, _ptr(q, ctypes.c_int8), ld,
                                    float(np.float32(qkv_scale)), o.ctypes.data_as(dp))

    threads = max(1, min(int(threads), batch))
    bounds = [batch * i // threads for i in range(threads + 1)]
    if threads == 1:
        rcs = [run(0, batch)]
    else:
        with ThreadPoolExecutor(threads) as ex:
            rcs = list(ex.map(lambda i: run(bounds[i], bounds[i + 1]), range(threads)))
    if any(rcs):
        raise ValueError("oracle_attention: bad sizes")
    return out


def attention(qkv: np.ndarray, qkv_scale, batch: int, seq: int, ctx_scale, heads: int = HEADS) -> np.ndarray:
    """attention_f32, requantised to int8 with ctx_scale."""
    return requant_f32(attention_f32(qkv, qkv_scale, batch, seq, heads), ctx_scale)


CHAIN_STAGES = ("qkv", "ctx", "attn_out", "ffn1", "ffn2")


def layer_chain(x0: np.ndarray, weights, out_scales: dict, batch: int, seq: int, threads: int = 8) -> dict:
    """The int8 outputs of every stage of one encoder layer for input x0
    [M][768]; weights = the four linears' BsrWeight (QKV, attention output,
    FFN1, FFN2), out_scales = the frozen output scales per stage."""
    wq, wo, w1, w2 = weights
    dense = [weight_dense(w) for w in weights]
    out = {}
    out["qkv"] = linear(x0, dense[0], wq.scales, wq.bias, I8, out_scales["qkv"], threads=threads)
    out["ctx"] = attention(out["qkv"], out_scales["qkv"], batch, seq, out_scales["ctx"])
    out["attn_out"] = linear(out["ctx"], dense[1], wo.scales, wo.bias, I8, out_scales["attn_out"], threads=threads)
    out["ffn1"] = linear(out["attn_out"], dense[2], w1.scales, w1.bias, I8_GELU, out_scales["ffn1"], threads=threads)
    out["ffn2"] = linear(out["ffn1"], dense[3], w2.scales, w2.bias, I8, out_scales["ffn2"], threads=threads)
    return out


def calibrate_chain(x0: np.ndarray, weights, batch: int, seq: int, threads: int = 8) -> dict:
    """Post-training calibration of the chain's output scales: each stage's
    scale is max |y| / 127 (in fp32) of its unquantised output y on these
    inputs, stage by stage, so that every stage sees the int8 input the
    chain will give it."""
    wq, wo, w1, w2 = weights
    dense = [weight_dense(w) for w in weights]

    def scale_of(y) -> float:
        return float(np.float32(np.max(np.abs(y))) / np.float32(127.0))

    s = {}
    s["qkv"] = scale_of(linear(x0, dense[0], wq.scales, wq.bias, F32, threads=threads))
    qkv = linear(x0, dense[0], wq.scales, wq.bias, I8, s["qkv"], threads=threads)
    ctx_f = attention_f32(qkv, s["qkv"], batch, seq)
    s["ctx"] = scale_of(ctx_f)
    ctx = requant_f32(ctx_f, s["ctx"])
    s["attn_out"] = scale_of(linear(ctx, dense[1], wo.scales, wo.bias, F32, threads=threads))
    o = linear(ctx, dense[1], wo.scales, wo.bias, I8, s["attn_out"], threads=threads)
    s["ffn1"] = scale_of(linear(o, dense[2], w1.scales, w1.bias, F32_GELU, threads=threads))
    f1 = linear(o, dense[2], w1.scales, w1.bias, I8_GELU, s["ffn1"], threads=threads)
    s["ffn2"] = scale_of(linear(f1, dense[3], w2.scales, w2.bias, F32, threads=threads))
    return s
