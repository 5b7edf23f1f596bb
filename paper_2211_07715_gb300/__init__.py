"""Block-sparse INT8 linear layer on GB300 -- Python binding of libbsgemm.so.

The layer is the hot path of the inference engine of "Fast DistilBERT on
CPUs" (arXiv 2211.07715): int8 activations times an int8 weight that is
sparse in blocks of 4 output rows x 1 input column, exact int32
accumulation, and a fused dequantise + bias (+ GELU) (+ requantise)
epilogue.  All arithmetic runs in the CUDA kernels of libbsgemm.so; this
module only marshals arguments (PyTorch provides device memory and
streams).  There is no CPU fallback: importing fails loudly if the library
has not been built (``python paper_2211_07715_gb300/build.py`` or
``__graft_entry__.build()``).

The functions below carry the C names (``bsgemm_create``, ``bsgemm_run``,
...); :class:`SparseInt8Linear` wraps one handle.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libbsgemm.so")

BLOCK = 4
OUT_I32, OUT_F32, OUT_F32_GELU, OUT_I8, OUT_I8_GELU, OUT_F32_RESID = 0, 1, 2, 3, 4, 5
ERR_INVALID, ERR_UNSUPPORTED, ERR_CUDA = -1, -2, -3
STATUS_TIMEOUT = 1  # BSGEMM_STATUS_TIMEOUT: a bounded wait on an asynchronous copy gave up
STATIC_SCRATCH_BYTES = 16 << 20  # BSGEMM_STATIC_SCRATCH_BYTES: the token-tile scratch of bsgemm_run_static


class BsgemmError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"bsgemm error {code}: {msg}")
        self.code = code


ACT_READY = 1  # BSGEMM_ACT_READY: act may be read while the stream's previous kernel finishes


class Epilogue(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("out_scale", ctypes.c_float), ("flags", ctypes.c_uint32),
                ("residual", ctypes.c_void_p), ("residual_scale", ctypes.c_float)]


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with `python paper_2211_07715_gb300/build.py`")
    lib = ctypes.CDLL(LIB_PATH)
    vp = ctypes.c_void_p
    lib.bsgemm_create.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, vp, vp, vp, vp]
    lib.bsgemm_create.restype = vp
    lib.bsgemm_create_1x4.argtypes = [ctypes.c_int, ctypes.c_int, vp, vp, vp, vp]
    lib.bsgemm_create_1x4.restype = vp
    lib.bsgemm_create_2to4.argtypes = [ctypes.c_int, ctypes.c_int, vp, vp, vp, vp]
    lib.bsgemm_create_2to4.restype = vp
    lib.bsgemm_create_tc.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, vp, vp, vp, vp]
    lib.bsgemm_create_tc.restype = vp
    lib.bsgemm_run.argtypes = [vp, vp, ctypes.c_int, vp, Epilogue, vp]
    lib.bsgemm_run.restype = ctypes.c_int
    lib.bsgemm_destroy.argtypes = [vp]
    lib.bsgemm_destroy.restype = None
    lib.bsgemm_last_error.argtypes = []
    lib.bsgemm_last_error.restype = ctypes.c_char_p
    lib.bsgemm_last_status.argtypes = []
    lib.bsgemm_last_status.restype = ctypes.c_int
    lib.bsgemm_max_k.argtypes = []
    lib.bsgemm_max_k.restype = ctypes.c_int
    lib.bsgemm_info.argtypes = [vp, ctypes.POINTER(ctypes.c_int64), ctypes.c_int]
    lib.bsgemm_info.restype = ctypes.c_int
    lib.bsgemm_workspace_bytes.argtypes = [vp, ctypes.c_int]
    lib.bsgemm_workspace_bytes.restype = ctypes.c_size_t
    lib.bsgemm_run_ws.argtypes = [vp, vp, ctypes.c_int, vp, Epilogue, vp, ctypes.c_size_t, vp]
    lib.bsgemm_run_ws.restype = ctypes.c_int
    lib.bsgemm_run_static.argtypes = [vp, vp, ctypes.c_int, vp, Epilogue, vp]
    lib.bsgemm_run_static.restype = ctypes.c_int
    lib.bsgemm_tile_activations.argtypes = [vp, vp, ctypes.c_int, vp, ctypes.c_size_t, vp]
    lib.bsgemm_tile_activations.restype = ctypes.c_int
    lib.bsgemm_run_kmajor.argtypes = [vp, vp, ctypes.c_int, ctypes.c_int, vp, Epilogue, vp]
    lib.bsgemm_run_kmajor.restype = ctypes.c_int
    lib.bsgemm_run_tiled.argtypes = [vp, vp, ctypes.c_size_t, ctypes.c_int, vp, Epilogue, vp]
    lib.bsgemm_run_tiled.restype = ctypes.c_int
    lib.bsgemm_host_workspace_bytes.argtypes = [vp, ctypes.c_int, ctypes.c_int32]
    lib.bsgemm_host_workspace_bytes.restype = ctypes.c_size_t
    lib.bsgemm_run_host.argtypes = [vp, vp, ctypes.c_int, vp, Epilogue, vp, ctypes.c_size_t, vp]
    lib.bsgemm_run_host.restype = ctypes.c_int
    lib.bsgemm_block_prune.argtypes = [ctypes.c_int, ctypes.c_int, vp, ctypes.c_double, vp, vp]
    lib.bsgemm_block_prune.restype = ctypes.c_int64
    lib.bsgemm_layernorm.argtypes = [vp, ctypes.c_int, ctypes.c_int, vp, vp, ctypes.c_float, vp, Epilogue, vp]
    lib.bsgemm_layernorm.restype = ctypes.c_int
    lib.bsgemm_attention.argtypes = [vp, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                     ctypes.c_float, vp, Epilogue, vp]
    lib.bsgemm_attention.restype = ctypes.c_int
    lib.bsgemm_device_status.argtypes = [vp, ctypes.c_int]
    lib.bsgemm_device_status.restype = ctypes.c_int
    lib.bsgemm_attention_status.argtypes = [ctypes.c_int]
    lib.bsgemm_attention_status.restype = ctypes.c_int
    lib.bsgemm_set_test_hooks.argtypes = [ctypes.c_uint32]
    lib.bsgemm_set_test_hooks.restype = ctypes.c_uint32
    lib.bsgemm_int8_peak.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
    lib.bsgemm_int8_peak.restype = ctypes.c_int
    return lib


_lib = _load()

EXPORTED = ("bsgemm_create", "bsgemm_create_1x4", "bsgemm_create_2to4", "bsgemm_create_tc", "bsgemm_run", "bsgemm_run_ws", "bsgemm_run_static", "bsgemm_workspace_bytes",
            "bsgemm_tile_activations", "bsgemm_run_tiled", "bsgemm_run_kmajor",
            "bsgemm_host_workspace_bytes", "bsgemm_run_host", "bsgemm_block_prune", "bsgemm_layernorm",
            "bsgemm_attention", "bsgemm_destroy",
            "bsgemm_last_error", "bsgemm_last_status", "bsgemm_device_status", "bsgemm_max_k", "bsgemm_info",
            "bsgemm_set_test_hooks", "bsgemm_int8_peak", "bsgemm_attention_status")


def _epi(kind: int, out_scale: float, flags: int = 0, residual: int = 0, residual_scale: float = 1.0) -> Epilogue:
    return Epilogue(int(kind), float(out_scale), int(flags), residual or None, float(residual_scale))


def bsgemm_last_error() -> str:
    return _lib.bsgemm_last_error().decode()


def bsgemm_last_status() -> int:
    return int(_lib.bsgemm_last_status())


def bsgemm_max_k() -> int:
    return int(_lib.bsgemm_max_k())


def _host_array(a, dtype) -> np.ndarray:
    if hasattr(a, "detach"):  # a torch tensor
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def bsgemm_create(n_out: int, k_in: int, block: int, indices, values, scales, bias=None) -> int:
    """Create a handle from host arrays (see include/bsgemm.h); raises on failure."""
    indices = _host_array(indices, np.int32)
    values = _host_array(values, np.int8)
    scales = _host_array(scales, np.float32)
    bias = None if bias is None else _host_array(bias, np.float32)
    h = _lib.bsgemm_create(int(n_out), int(k_in), int(block), indices.ctypes.data, values.ctypes.data,
                           scales.ctypes.data, None if bias is None else bias.ctypes.data)
    if not h:
        raise BsgemmError(bsgemm_last_status(), bsgemm_last_error())
    return h


def bsgemm_create_tc(n_out: int, k_in: int, block: int, indices, values, scales, bias=None) -> int:
    """As bsgemm_create, and with N and K multiples of 128 (K <= 4096) the
    row-major runs go dense over K to the tensor cores (see include/bsgemm.h)."""
    indices = _host_array(indices, np.int32)
    values = _host_array(values, np.int8)
    scales = _host_array(scales, np.float32)
    bias = None if bias is None else _host_array(bias, np.float32)
    h = _lib.bsgemm_create_tc(int(n_out), int(k_in), int(block), indices.ctypes.data, values.ctypes.data,
                              scales.ctypes.data, None if bias is None else bias.ctypes.data)
    if not h:
        raise BsgemmError(bsgemm_last_status(), bsgemm_last_error())
    return h


def bsgemm_create_1x4(n_out: int, k_in: int, indices, values, scales, bias=None) -> int:
    """Handle of a weight sparse in 1 x 4 blocks: indices = indptr [N + 1]
    then colgrp [nnz]; values int8 [nnz][4] (see include/bsgemm.h)."""
    indices = _host_array(indices, np.int32)
    values = _host_array(values, np.int8)
    scales = _host_array(scales, np.float32)
    bias = None if bias is None else _host_array(bias, np.float32)
    h = _lib.bsgemm_create_1x4(int(n_out), int(k_in), indices.ctypes.data, values.ctypes.data, scales.ctypes.data,
                               None if bias is None else bias.ctypes.data)
    if not h:
        raise BsgemmError(bsgemm_last_status(), bsgemm_last_error())
    return h


def bsgemm_create_2to4(n_out: int, k_in: int, values, idx, scales, bias=None) -> int:
    """Handle of a 2:4-sparse weight: values int8 and idx uint8 [N][K/2]."""
    values = _host_array(values, np.int8)
    idx = _host_array(idx, np.uint8)
    scales = _host_array(scales, np.float32)
    bias = None if bias is None else _host_array(bias, np.float32)
    h = _lib.bsgemm_create_2to4(int(n_out), int(k_in), values.ctypes.data, idx.ctypes.data, scales.ctypes.data,
                                None if bias is None else bias.ctypes.data)
    if not h:
        raise BsgemmError(bsgemm_last_status(), bsgemm_last_error())
    return h


def bsgemm_run(h: int, act_ptr: int, m: int, out_ptr: int, kind: int, out_scale: float = 1.0,
               stream: int = 0, flags: int = 0, residual_ptr: int = 0, residual_scale: float = 1.0) -> None:
    """Enqueue one run on `stream` (raw device pointers); raises on failure."""
    rc = _lib.bsgemm_run(h, act_ptr, int(m), out_ptr, _epi(kind, out_scale, flags, residual_ptr, residual_scale),
                         stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_run_ws(h: int, act_ptr: int, m: int, out_ptr: int, kind: int, out_scale: float, ws_ptr: int,
                  ws_bytes: int, stream: int = 0, flags: int = 0, residual_ptr: int = 0,
                  residual_scale: float = 1.0) -> None:
    """Enqueue a run with a device workspace (used only by the shapes that
    need the relayout kernel); raises on failure."""
    rc = _lib.bsgemm_run_ws(h, act_ptr, int(m), out_ptr, _epi(kind, out_scale, flags, residual_ptr, residual_scale),
                            ws_ptr, int(ws_bytes), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_run_static(h: int, act_ptr: int, m: int, out_ptr: int, kind: int, out_scale: float = 1.0,
                      stream: int = 0) -> None:
    """The fast path with the library's fixed device scratch: allocates
    nothing; calls overlapping in time on one device race (see the header)."""
    rc = _lib.bsgemm_run_static(h, act_ptr, int(m), out_ptr, _epi(kind, out_scale), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_run_kmajor(h: int, act_t_ptr: int, m: int, ld: int, out_ptr: int, kind: int, out_scale: float = 1.0,
                      stream: int = 0, flags: int = 0) -> None:
    """The layer on K-major activations X^T [K][M] (row stride ld bytes)."""
    rc = _lib.bsgemm_run_kmajor(h, act_t_ptr, int(m), int(ld), out_ptr,
                                _epi(kind, out_scale, flags), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_tile_activations(h: int, act_ptr: int, m: int, tiles_ptr: int, tiles_bytes: int, stream: int = 0) -> None:
    rc = _lib.bsgemm_tile_activations(h, act_ptr, int(m), tiles_ptr, int(tiles_bytes), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_run_tiled(h: int, tiles_ptr: int, tiles_bytes: int, m: int, out_ptr: int, kind: int, out_scale: float,
                     stream: int = 0) -> None:
    rc = _lib.bsgemm_run_tiled(h, tiles_ptr, int(tiles_bytes), int(m), out_ptr, _epi(kind, out_scale),
                               stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_run_host(h: int, act_ptr: int, m: int, out_ptr: int, kind: int, out_scale: float, ws_ptr: int,
                    ws_bytes: int, stream: int = 0) -> None:
    """Enqueue the end-to-end call: HOST act and out, a DEVICE workspace."""
    rc = _lib.bsgemm_run_host(h, act_ptr, int(m), out_ptr, _epi(kind, out_scale), ws_ptr,
                              int(ws_bytes), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def bsgemm_host_workspace_bytes(h: int, m: int, kind: int) -> int:
    return int(_lib.bsgemm_host_workspace_bytes(h, int(m), int(kind)))


def bsgemm_block_prune(n_out: int, k_in: int, w_ptr: int, sparsity: float, keep_ptr: int, stream: int = 0) -> int:
    """Average-magnitude 4x1 block pruning on the device (raw pointers);
    returns the number of kept blocks, raises on failure."""
    rc = _lib.bsgemm_block_prune(int(n_out), int(k_in), w_ptr, float(sparsity), keep_ptr, stream)
    if rc < 0:
        raise BsgemmError(int(rc), bsgemm_last_error())
    return int(rc)


def block_prune(w, sparsity: float, stream=None):
    """Keep-mask [N/4][K] (uint8 CUDA tensor, 1 = kept) of the App. A.1
    pruning of the fp32 CUDA weight `w` [N][K] to the given sparsity."""
    import torch
    if w.dtype != torch.float32 or not w.is_cuda or not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous fp32 CUDA tensor [N][K]")
    n_out, k_in = w.shape
    if n_out % BLOCK:
        raise ValueError("N must be a multiple of 4")
    keep = torch.empty((n_out // BLOCK, k_in), dtype=torch.uint8, device=w.device)
    s = torch.cuda.current_stream() if stream is None else stream
    bsgemm_block_prune(n_out, k_in, w.data_ptr(), sparsity, keep.data_ptr(), s.cuda_stream)
    return keep


def bsgemm_layernorm(z_ptr: int, m: int, n: int, gamma_ptr: int, beta_ptr: int, eps: float, out_ptr: int, kind: int,
                     out_scale: float = 1.0, stream: int = 0) -> None:
    """Enqueue the row-wise LayerNorm of z [M][N] fp32 (raw device pointers)."""
    rc = _lib.bsgemm_layernorm(z_ptr, int(m), int(n), gamma_ptr, beta_ptr, float(eps), out_ptr, _epi(kind, out_scale),
                               stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def layernorm(z, gamma, beta, eps: float, kind: int = OUT_F32, out_scale: float = 1.0, stream=None):
    """LayerNorm of each row of the CUDA fp32 tensor z [M][N] (gamma, beta:
    CUDA fp32 [N]); returns a new CUDA tensor, float32 or int8 by kind."""
    import torch
    for t, name in ((z, "z"), (gamma, "gamma"), (beta, "beta")):
        if t.dtype != torch.float32 or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA float32 tensor")
    m, n = z.shape
    if tuple(gamma.shape) != (n,) or tuple(beta.shape) != (n,):
        raise ValueError("gamma and beta must be [N]")
    out = torch.empty((m, n), dtype=torch.int8 if kind == OUT_I8 else torch.float32, device=z.device)
    s = torch.cuda.current_stream() if stream is None else stream
    bsgemm_layernorm(z.data_ptr(), m, n, gamma.data_ptr(), beta.data_ptr(), eps, out.data_ptr(), kind, out_scale,
                     s.cuda_stream)
    return out


ATTN_MAX_SEQ = 512  # BSGEMM_ATTN_MAX_SEQ
ATTN_HEAD_DIM = 64


def bsgemm_attention(qkv_ptr: int, batch: int, seq: int, heads: int, head_dim: int, ld: int, qkv_scale: float,
                     out_ptr: int, kind: int, out_scale: float = 1.0, stream: int = 0, flags: int = 0) -> None:
    """Enqueue multi-head self-attention on the int8 QKV rows (raw device
    pointers; rows of ld bytes holding q | k | v).  flags: 0 or ACT_READY
    (qkv was complete before the stream's previous kernel began)."""
    rc = _lib.bsgemm_attention(qkv_ptr, int(batch), int(seq), int(heads), int(head_dim), int(ld), float(qkv_scale),
                               out_ptr, _epi(kind, out_scale, flags), stream)
    if rc != 0:
        raise BsgemmError(rc, bsgemm_last_error())


def attention(qkv, batch: int, seq: int, heads: int, qkv_scale: float, kind: int = OUT_F32, out_scale: float = 1.0,
              out=None, stream=None, flags: int = 0):
    """Multi-head self-attention (head width 64) on the CUDA int8 tensor qkv
    [batch * seq][>= 3 * heads * 64] (the QKV linear's output, q | k | v;
    its row stride may be padded to a multiple of 16).  Returns the context
    [batch * seq][heads * 64], float32 or int8 by kind (or fills `out`).
    flags: 0 or ACT_READY (qkv was complete before the stream's previous
    kernel began)."""
    import torch
    if qkv.dtype != torch.int8 or not qkv.is_cuda or qkv.dim() != 2 or qkv.stride(1) != 1:
        raise ValueError("qkv must be a CUDA int8 [M][row] tensor with unit column stride")
    m = qkv.shape[0]
    if m != batch * seq:
        raise ValueError("qkv must have batch * seq rows")
    d = heads * ATTN_HEAD_DIM
    if qkv.shape[1] < 3 * d:
        raise ValueError("qkv rows must hold q, k and v (3 * heads * 64 bytes)")
    dtype = torch.int8 if kind == OUT_I8 else torch.float32
    if out is None:
        out = torch.empty((m, d), dtype=dtype, device=qkv.device)
    elif out.dtype != dtype or tuple(out.shape) != (m, d) or not out.is_contiguous():
        raise ValueError(f"out must be a contiguous {dtype} [{m}][{d}] tensor")
    s = torch.cuda.current_stream() if stream is None else stream
    bsgemm_attention(qkv.data_ptr(), batch, seq, heads, ATTN_HEAD_DIM, qkv.stride(0), qkv_scale, out.data_ptr(), kind,
                     out_scale, s.cuda_stream, flags)
    return out


def bsgemm_workspace_bytes(h: int, m: int) -> int:
    return int(_lib.bsgemm_workspace_bytes(h, int(m)))


def bsgemm_device_status(h: int, clear: bool = False) -> int:
    rc = _lib.bsgemm_device_status(h, 1 if clear else 0)
    if rc < 0:
        raise BsgemmError(rc, bsgemm_last_error())
    return rc


TEST_SKIP_TILE_COPY = 1  # BSGEMM_TEST_SKIP_TILE_COPY
TEST_STALL_PRUNE_CTA = 2  # BSGEMM_TEST_STALL_PRUNE_CTA
TEST_ATTN_SKIP_MMA = 4  # BSGEMM_TEST_ATTN_SKIP_MMA


def bsgemm_attention_status(clear: bool = False) -> int:
    """The current device's attention status word (STATUS_TIMEOUT when a
    wait of the attention kernel gave up); synchronises the device."""
    rc = _lib.bsgemm_attention_status(1 if clear else 0)
    if rc < 0:
        raise BsgemmError(rc, bsgemm_last_error())
    return rc


def bsgemm_set_test_hooks(bits: int) -> int:
    """Make the kernels' bounded waits give up on purpose (tests of the
    failure path only); returns the previous bits."""
    return int(_lib.bsgemm_set_test_hooks(int(bits)))


def bsgemm_int8_peak(unit: int, iters: int = 4000) -> float:
    """Measured peak of an int8 dot-product unit in TOPS: unit 0 = dp4a,
    1 = mma.sync m16n8k32 s8 (synchronises the device)."""
    v = ctypes.c_double(0.0)
    rc = _lib.bsgemm_int8_peak(int(unit), int(iters), ctypes.byref(v))
    if rc != 0:
        raise BsgemmError(rc, "int8 peak probe failed")
    return float(v.value)


def bsgemm_destroy(h: int) -> None:
    _lib.bsgemm_destroy(h)


def bsgemm_info(h: int) -> dict:
    buf = (ctypes.c_int64 * 7)()
    rc = _lib.bsgemm_info(h, buf, 7)
    if rc < 0:
        raise BsgemmError(rc, bsgemm_last_error())
    keys = ("n_out", "k_in", "nnzb", "quads", "tile_m", "ctas", "device_bytes")
    return dict(zip(keys, (int(v) for v in buf)))


_OUT_DTYPES = {OUT_I32: "int32", OUT_F32: "float32", OUT_F32_GELU: "float32", OUT_I8: "int8", OUT_I8_GELU: "int8",
               OUT_F32_RESID: "float32"}


def dense_to_blocks(w: np.ndarray, keep=None):
    """Block-compress a dense int8 weight [N][K] (any N: the last block-row
    takes the N % 4 remaining rows, its missing rows read as zeros).  Stores
    the 4x1 blocks where `keep` [ceil(N/4)][K] is true (a mask from
    block_prune; its pruned blocks are dropped whatever they hold), or
    without a mask every block that holds a nonzero value.  Returns
    (indptr, colidx, values)."""
    w = _host_array(w, np.int8)
    n_out, k_in = w.shape
    nbr = -(-n_out // BLOCK)
    if n_out % BLOCK:
        w = np.concatenate([w, np.zeros((nbr * BLOCK - n_out, k_in), np.int8)])
    blocks = w.reshape(nbr, BLOCK, k_in)                      # [r][i][k]
    if keep is None:
        keep = (blocks != 0).any(axis=1)                      # [r][k]
    else:
        keep = _host_array(keep, np.uint8).astype(bool)
        if keep.shape != (nbr, k_in):
            raise ValueError(f"keep must have shape {(nbr, k_in)}")
    r_idx, k_idx = np.nonzero(keep)                           # row-major: sorted by r, then k
    indptr = np.zeros(nbr + 1, np.int32)
    np.cumsum(keep.sum(axis=1), out=indptr[1:])
    values = np.ascontiguousarray(blocks[r_idx, :, k_idx], dtype=np.int8)  # [nnzb][4]
    return indptr, k_idx.astype(np.int32), values


def dense_from_blocks_1x4(n_out: int, k_in: int, indptr, colgrp, values) -> np.ndarray:
    """Dense int8 W [N][K] of a weight sparse in 1 x 4 blocks: one output row
    x 4 consecutive input columns (K a multiple of 4).  Row n holds blocks
    indptr[n] .. indptr[n+1]-1; block e covers columns 4 colgrp[e] ..
    4 colgrp[e] + 3 with values[e][0..3].  Checks the arrays the way
    bsgemm_create checks its own (ValueError)."""
    indptr = _host_array(indptr, np.int32).reshape(-1)
    colgrp = _host_array(colgrp, np.int32).reshape(-1)
    values = _host_array(values, np.int8).reshape(-1, 4)
    if n_out < 1 or k_in < 4 or k_in % 4:
        raise ValueError("need N >= 1 and K a positive multiple of 4")
    if indptr.shape != (n_out + 1,) or indptr[0] != 0 or (np.diff(indptr) < 0).any():
        raise ValueError("indptr must hold N + 1 non-decreasing entries from 0")
    nnz = int(indptr[-1])
    if colgrp.shape != (nnz,) or values.shape != (nnz, 4):
        raise ValueError("colgrp and values must hold indptr[N] blocks")
    if nnz and (colgrp.min() < 0 or colgrp.max() >= k_in // 4):
        raise ValueError("column groups must lie in [0, K / 4)")
    rows = np.repeat(np.arange(n_out), np.diff(indptr))
    if nnz > 1:
        same_row = rows[1:] == rows[:-1]
        if (same_row & (colgrp[1:] <= colgrp[:-1])).any():
            raise ValueError("column groups must increase strictly within a row")
    w = np.zeros((n_out, k_in), np.int8)
    w[rows[:, None], 4 * colgrp[:, None] + np.arange(4)] = values
    return w


def dense_from_2to4(values, idx) -> np.ndarray:
    """Dense int8 W [N][K] of a 2:4-sparse weight: values and idx [N][K/2]
    hold, per output row and group g of 4 input columns, two values at the
    in-group positions idx[n][2g], idx[n][2g+1] (0 <= idx < 4, strictly
    increasing).  ValueError on bad indices."""
    values = _host_array(values, np.int8)
    idx = _host_array(idx, np.uint8)
    if values.ndim != 2 or idx.shape != values.shape or values.shape[1] % 2:
        raise ValueError("values and idx must be [N][K/2] with K a multiple of 4")
    n_out, half = values.shape
    pairs = idx.reshape(n_out, half // 2, 2)
    if (idx >= 4).any() or (pairs[:, :, 0] >= pairs[:, :, 1]).any():
        raise ValueError("in-group positions must lie in [0, 4) and increase within each group")
    cols = 4 * (np.arange(half) // 2)[None, :] + idx.astype(np.int64)
    w = np.zeros((n_out, 2 * half), np.int8)
    w[np.arange(n_out)[:, None], cols] = values
    return w


class SparseInt8Linear:
    """One block-sparse int8 linear layer resident on the current CUDA device."""

    def __init__(self, n_out: int, k_in: int, indptr, colidx, values, scales, bias=None, tensor_cores: bool = False):
        """tensor_cores: create through bsgemm_create_tc (the weight also run
        dense over K on the tensor cores when N and K are multiples of 128)."""
        indices = np.concatenate([_host_array(indptr, np.int32), _host_array(colidx, np.int32)])
        self.n_out, self.k_in = int(n_out), int(k_in)
        create = bsgemm_create_tc if tensor_cores else bsgemm_create
        self._h = create(n_out, k_in, BLOCK, indices, values, scales, bias)
        self.info = bsgemm_info(self._h)

    @classmethod
    def from_dense(cls, w, scales, bias=None, keep=None, tensor_cores: bool = False) -> "SparseInt8Linear":
        """From a dense int8 weight [N][K]; `keep` [N/4][K] (e.g. from
        block_prune) selects the stored blocks."""
        w = _host_array(w, np.int8)
        indptr, colidx, values = dense_to_blocks(w, keep)
        return cls(w.shape[0], w.shape[1], indptr, colidx, values, scales, bias, tensor_cores=tensor_cores)

    @classmethod
    def _of_handle(cls, h: int, n_out: int, k_in: int) -> "SparseInt8Linear":
        self = cls.__new__(cls)
        self.n_out, self.k_in = int(n_out), int(k_in)
        self._h = h
        self.info = bsgemm_info(h)
        return self

    @classmethod
    def from_blocks_1x4(cls, n_out: int, k_in: int, indptr, colgrp, values, scales, bias=None) -> "SparseInt8Linear":
        """A weight sparse in 1 x 4 blocks (one output row x 4 consecutive
        input columns; block e of row n covers columns 4 colgrp[e] ..
        4 colgrp[e] + 3), run natively by the layer kernel's 1 x 4 form
        (bsgemm_create_1x4): one dot-4 per block and token."""
        indices = np.concatenate([_host_array(indptr, np.int32), _host_array(colgrp, np.int32)])
        return cls._of_handle(bsgemm_create_1x4(n_out, k_in, indices, values, scales, bias), n_out, k_in)

    @classmethod
    def from_2to4(cls, values, idx, scales, bias=None) -> "SparseInt8Linear":
        """A 2:4-sparse weight (values, idx [N][K/2]) through
        bsgemm_create_2to4: on the sparse tensor cores when N and K are
        multiples of 128 (K <= 4096), else as the 4 x 1 blocks that hold its
        values (~94% of all blocks for random 2:4 patterns)."""
        values = np.asarray(values)
        n_out, k_in = values.shape[0], 2 * values.shape[1]
        return cls._of_handle(bsgemm_create_2to4(n_out, k_in, values, idx, scales, bias), n_out, k_in)

    def workspace_bytes(self, m: int) -> int:
        return bsgemm_workspace_bytes(self._h, m)

    def run(self, x, out, kind: int, out_scale: float = 1.0, stream=None, workspace=None,
            act_ready: bool = False, residual=None, residual_scale: float = 1.0) -> None:
        """out[M][N] = epilogue(x[M][K] W^T); both CUDA tensors, contiguous.

        With K % 16 == 0 and x 16-byte aligned this is one kernel that stages
        x itself (the workspace is then unused); otherwise the workspace --
        the given uint8 CUDA tensor, or (workspace=None) one drawn from
        PyTorch's caching allocator on the same stream -- takes the relaid
        tiles, and workspace=False gathers them with per-thread loads
        instead.  act_ready: x was complete before the stream's previous
        kernel began (BSGEMM_ACT_READY).  OUT_F32_RESID adds residual_scale *
        residual (a contiguous CUDA int8 [M][N] tensor) to the dequantised
        value (the residual add before LayerNorm)."""
        import torch
        if x.dtype != torch.int8 or not x.is_cuda or not x.is_contiguous() or x.dim() != 2 or x.shape[1] != self.k_in:
            raise ValueError("x must be a contiguous CUDA int8 tensor [M][K]")
        if (not out.is_cuda or not out.is_contiguous() or tuple(out.shape) != (x.shape[0], self.n_out)
                or str(out.dtype).split(".")[-1] != _OUT_DTYPES[kind]):
            raise ValueError(f"out must be a contiguous CUDA {_OUT_DTYPES[kind]} tensor [M][N]")
        s = torch.cuda.current_stream() if stream is None else stream
        m = x.shape[0]
        flags = ACT_READY if act_ready else 0
        res_ptr = 0
        if kind == OUT_F32_RESID:
            if (residual is None or residual.dtype != torch.int8 or not residual.is_cuda
                    or not residual.is_contiguous() or tuple(residual.shape) != (m, self.n_out)):
                raise ValueError("OUT_F32_RESID needs a contiguous CUDA int8 residual [M][N]")
            res_ptr = residual.data_ptr()
        if workspace is False or m == 0:
            bsgemm_run(self._h, x.data_ptr(), m, out.data_ptr(), kind, out_scale, s.cuda_stream, flags, res_ptr,
                       residual_scale)
            return
        need = self.workspace_bytes(m)
        if workspace is None:
            with torch.cuda.stream(s):
                workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
        if workspace.numel() * workspace.element_size() < need:
            raise ValueError(f"workspace must hold {need} bytes")
        bsgemm_run_ws(self._h, x.data_ptr(), m, out.data_ptr(), kind, out_scale, workspace.data_ptr(),
                      workspace.numel() * workspace.element_size(), s.cuda_stream, flags, res_ptr, residual_scale)

    def run_kmajor(self, xt, out, kind: int, out_scale: float = 1.0, stream=None) -> None:
        """out[M][N] = epilogue(X W^T) from K-major activations: xt is a CUDA
        int8 tensor [K][M] whose rows are 16-byte aligned (row stride a
        multiple of 16 bytes, M <= stride); out a contiguous CUDA [M][N]."""
        import torch
        if (xt.dtype != torch.int8 or not xt.is_cuda or xt.dim() != 2 or xt.shape[0] != self.k_in
                or xt.stride(1) != 1):
            raise ValueError("xt must be a CUDA int8 tensor [K][M] with unit column stride")
        m = xt.shape[1]
        if (not out.is_cuda or not out.is_contiguous() or tuple(out.shape) != (m, self.n_out)
                or str(out.dtype).split(".")[-1] != _OUT_DTYPES[kind]):
            raise ValueError(f"out must be a contiguous CUDA {_OUT_DTYPES[kind]} tensor [M][N]")
        s = torch.cuda.current_stream() if stream is None else stream
        bsgemm_run_kmajor(self._h, xt.data_ptr(), m, xt.stride(0), out.data_ptr(), kind, out_scale, s.cuda_stream)

    def __call__(self, x, kind: int, out_scale: float = 1.0, stream=None, out=None, sync: bool = True):
        """Allocate the output (unless `out` is given) and run.

        A CUDA `x` stays on the device.  A CPU `x` takes the end-to-end path
        (bsgemm_run_host): it is copied in, the layer runs, and the result is
        copied back into `out` (a CPU tensor, pinned for an asynchronous
        copy) or a new one.  With sync=False and pinned `x` and `out`, the
        call only enqueues on `stream` (default: the current stream): the
        caller synchronises that stream before reading `out`, and leaves `x`
        unchanged until then.  The device workspace comes from PyTorch's
        caching allocator on that stream.
        """
        import torch
        dtype = getattr(torch, _OUT_DTYPES[kind])
        s = torch.cuda.current_stream() if stream is None else stream
        if x.is_cuda:
            if out is None:
                out = torch.empty((x.shape[0], self.n_out), dtype=dtype, device=x.device)
            self.run(x, out, kind, out_scale, s)
            return out
        if x.dtype != torch.int8 or not x.is_contiguous() or x.dim() != 2 or x.shape[1] != self.k_in:
            raise ValueError("x must be a contiguous int8 tensor [M][K]")
        m = x.shape[0]
        pinned = x.is_pinned()
        if out is None:
            out = torch.empty((m, self.n_out), dtype=dtype, pin_memory=pinned)
        elif out.is_cuda or out.dtype != dtype or tuple(out.shape) != (m, self.n_out) or not out.is_contiguous():
            raise ValueError(f"out must be a contiguous CPU {dtype} tensor of shape {(m, self.n_out)}")
        if not sync and not (pinned and out.is_pinned()):
            raise ValueError("sync=False needs a pinned x and a pinned out")
        if m == 0:
            return out
        need = bsgemm_host_workspace_bytes(self._h, m, kind)
        with torch.cuda.stream(s):
            ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        bsgemm_run_host(self._h, x.data_ptr(), m, out.data_ptr(), kind, out_scale, ws.data_ptr(), need, s.cuda_stream)
        if sync:
            s.synchronize()
        return out

    def close(self) -> None:
        if getattr(self, "_h", None):
            bsgemm_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
