/*
 * bsgemm.h -- C ABI of the block-sparse INT8 linear layer on one GB300
 * (sm_103a): the hot path of the inference engine of "Fast DistilBERT on
 * CPUs" (arXiv 2211.07715), re-designed for the GPU.
 *
 * The layer computes, for int8 activations X [M][K] and an int8 weight
 * W [N][K] that is sparse in blocks of 4 consecutive output rows x 1 input
 * column (App. A.1; "constant block size 4", App. A.3.4):
 *
 *   acc[m][n] = sum_k X[m][k] * W[n][k]                  exact int32
 *                 (Sec. 3 "Sparse GEMM operators", Algorithm 1's dot-4)
 *   y[m][n]   = fmaf((float)acc[m][n], scales[n], bias[n])
 *   out       = acc | y | GELU(y) | q(y) | q(GELU(y))
 *                 (the fused post-operators of App. A.3.3 / Algorithm 1's
 *                  "downconvert and post-operator fusion")
 *
 * with q(v) = saturate_s8(round_half_even(v * (1.0f / out_scale))) and
 * GELU the erf form 0.5 y (1 + erf(y / sqrt 2)) evaluated in fp32 by the
 * Abramowitz & Stegun 7.1.28 rational approximation of erf (|error| <=
 * 3e-7), by one fixed IEEE op sequence so that int8 results are
 * reproducible bit for bit.
 *
 * Threading: every function may be called from any host thread.  A handle
 * is immutable after bsgemm_create, so one handle (one copy of the weights
 * in device memory) may serve concurrent bsgemm_run calls on several
 * streams -- the GPU form of the paper's weight sharing across parallel
 * instances (App. A.3.2).
 *
 * Errors: functions returning int give 0 on success or a negative
 * BSGEMM_ERR_* code; bsgemm_create returns NULL on failure.  In both cases
 * bsgemm_last_error() describes the last failure on the calling thread.
 */
#ifndef BSGEMM_H_
#define BSGEMM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BSGEMM_BLOCK 4 /* output rows per block (App. A.1) */

/* Return codes. */
#define BSGEMM_OK 0
#define BSGEMM_ERR_INVALID (-1)     /* a pointer, size or value is not allowed */
#define BSGEMM_ERR_UNSUPPORTED (-2) /* valid, but outside what this build runs */
#define BSGEMM_ERR_CUDA (-3)        /* a CUDA call failed (message has details) */

/* Epilogue kinds: what bsgemm_run writes to `out` (App. A.3.3 post-ops). */
typedef enum {
    BSGEMM_OUT_I32 = 0,      /* int32 acc                               */
    BSGEMM_OUT_F32 = 1,      /* float y = fmaf((float)acc, s[n], b[n])   */
    BSGEMM_OUT_F32_GELU = 2, /* float GELU(y)                           */
    BSGEMM_OUT_I8 = 3,       /* int8  q(y)                              */
    BSGEMM_OUT_I8_GELU = 4,  /* int8  q(GELU(y))                        */
    BSGEMM_OUT_F32_RESID = 5 /* float z = y + residual_scale * residual */
} bsgemm_out_kind;

typedef struct {
    int32_t kind;    /* a bsgemm_out_kind                                    */
    float out_scale; /* int8 kinds only: finite and > 0; the library         */
                     /* multiplies by 1.0f / out_scale (one fp32 division)   */
    uint32_t flags;  /* 0 or BSGEMM_ACT_READY; other bits are invalid        */
    const int8_t* residual; /* BSGEMM_OUT_F32_RESID only: DEVICE int8 [M][N], */
                            /* 4-byte aligned (the sub-layer's input that the */
                            /* encoder adds before LayerNorm, Sec. 3)         */
    float residual_scale;   /* its scale, finite                              */
} bsgemm_epilogue;

/*
 * BSGEMM_ACT_READY: act was complete before the kernel that precedes this
 * call on the stream began (an upload, or the output of work that has
 * finished), so the layer kernel may start reading it while that kernel
 * still runs (the kernels are launched with programmatic dependent launch).
 * Without the flag act is read only after the preceding kernel has
 * completed, which is right whenever that kernel writes act (a layer
 * chain).  Outputs are written after the preceding kernel in either case.
 * It changes nothing on the paths that stage relaid tiles.
 */
#define BSGEMM_ACT_READY 1u

typedef struct bsgemm_ctx* bsgemm_t; /* opaque handle */

/*
 * bsgemm_create -- build the device form of a block-compressed weight.
 *
 * Block-compressed layout (App. A.1 blocks; App. A.3.4 "the sparse weight is
 * compressed and the mask is used"), all HOST memory, read during the call
 * only (the caller keeps ownership and may free them on return):
 *   N        output features, 1 <= N <= BSGEMM_MAX_N.  Block-row r holds rows 4r..4r+3;
 *            when N % 4 != 0 the last block-row, r = ceil(N/4) - 1, holds
 *            the N % 4 remaining rows and values[j][i] of its rows
 *            4r + i >= N are ignored (App. A.3.4 notes that such N need
 *            padding and leaves it out; here the block-row is zero-padded
 *            at create time and only channels < N are stored).
 *   K        input features, 1 <= K <= bsgemm_max_k().
 *   block    must be 4.
 *   indices  int32: indptr[R + 1] followed by colidx[nnzb], R =
 *            ceil(N/4), nnzb = indptr[R].  Block j of block-row r (indptr[r] <= j <
 *            indptr[r+1]) lies in column colidx[j]; columns strictly
 *            increase within a block-row; indptr[0] = 0.
 *   values   int8 [nnzb][4]: values[j][i] = W[4r + i][colidx[j]].  A stored
 *            block may hold zeros; any int8 value is allowed.
 *   scales   float [N]: per-output-channel dequantisation scale (the product
 *            of the activation and weight scales); must be finite.
 *   bias     float [N], or NULL for zeros; must be finite.
 * The call allocates device memory on the CURRENT CUDA device, copies the
 * repacked weights there and synchronises.  Returns NULL on failure.
 *
 * Other block shapes: bsgemm_create_1x4 and bsgemm_create_2to4 below; the
 * same weight run dense on the tensor cores: bsgemm_create_tc.
 */
#define BSGEMM_MAX_N (4 * 65535) /* block-row indices are 16-bit inside the kernel */
bsgemm_t bsgemm_create(int N, int K, int block, const int32_t* indices, const int8_t* values,
                       const float* scales, const float* bias);

/*
 * bsgemm_create_1x4 -- a weight sparse in 1 x 4 blocks: one output row x 4
 * consecutive input columns (the paper's 4 x 1 blocks turned along K; its
 * App. A.3.4 leaves other block shapes to padding and regrouping).  The
 * layer kernel runs them natively: each block is one dot-4 of a token's 4
 * consecutive activations with the block's 4 weights, with no zero padding
 * of the block's work.  HOST arrays, read during the call only:
 *   N        output features, 1 <= N <= 65535 (any N; rows are independent).
 *   K        input features, a multiple of 4, 4 <= K <= bsgemm_max_k().
 *   indices  int32: indptr[N + 1] followed by colgrp[nnz], nnz = indptr[N]:
 *            block e of row n (indptr[n] <= e < indptr[n + 1]) covers
 *            columns 4 colgrp[e] .. 4 colgrp[e] + 3; colgrp strictly
 *            increases within a row and lies in [0, K/4).
 *   values   int8 [nnz][4]: values[e][i] = W[n][4 colgrp[e] + i].
 *   scales, bias  as for bsgemm_create.
 * Runs take every bsgemm_run* call and epilogue kind except
 * BSGEMM_OUT_F32_RESID (BSGEMM_ERR_UNSUPPORTED).  bsgemm_info()[2] is nnz.
 * Returns NULL on failure (bsgemm_last_error / bsgemm_last_status).
 */
bsgemm_t bsgemm_create_1x4(int N, int K, const int32_t* indices, const int8_t* values, const float* scales,
                           const float* bias);

/*
 * bsgemm_create_2to4 -- a weight with 2:4 structured sparsity along K (two
 * values in every group of 4 consecutive input columns of every row, the
 * pattern of sparse tensor cores that Sec. 1 cites as related work).  HOST
 * arrays [N][K/2], read during the call only: values int8 and idx uint8,
 * where values[n][2j + t] is W[n][4j + idx[n][2j + t]]; idx[n][2j] <
 * idx[n][2j + 1] <= 3 (a value may be 0).  K a multiple of 4, at most
 * bsgemm_max_k().  With N and K multiples of 128 the runs of row-major activations
 * (bsgemm_run, _run_ws, _run_static, _run_host), every kind but
 * BSGEMM_OUT_F32_RESID, go to the sparse tensor cores (tcgen05.mma.sp: the
 * stored values as f16 with their positions, the activations widened to
 * f16, exact fp32 partial sums of at most 1024 products added in int32:
 * the int32 result bit for bit); the handle then holds a second device
 * allocation of N K + N K / 32 bytes for those operands.  Other shapes and
 * runs go through the 4 x 1 blocks that hold the values (block (r, k)
 * stored when one of rows 4r..4r+3 is nonzero in column k; about 1.9x the
 * multiply-adds of the 2:4 values for random patterns).  scales, bias and
 * the result as for bsgemm_create.
 */
bsgemm_t bsgemm_create_2to4(int N, int K, const int8_t* values, const uint8_t* idx, const float* scales,
                            const float* bias);

/*
 * bsgemm_create_tc -- the block-compressed weight of bsgemm_create (same
 * arguments, same validation, same result), also laid out to run DENSE
 * over K on the tensor cores: the contraction of Algorithm 1 with every
 * column multiplied, zeros included (tcgen05.mma kind::f16 on the int8
 * values as f16, the activations widened to f16, exact fp32 partial sums
 * of at most 1024 products added in int32: the int32 result bit for bit).
 * With N and K multiples of 128 (K <= bsgemm_max_k() as for every
 * handle) the runs of row-major activations (bsgemm_run, _run_ws,
 * _run_static, _run_host), every kind but BSGEMM_OUT_F32_RESID, take that
 * path, and the handle holds a second
 * device allocation of 2 N K bytes (the f16 image); other shapes and runs
 * take the block-sparse kernel.  This is the tensor-core alternative to
 * the block-sparse int8 kernel, for comparison: its time does not fall
 * with sparsity.
 */
bsgemm_t bsgemm_create_tc(int N, int K, int block, const int32_t* indices, const int8_t* values,
                          const float* scales, const float* bias);

/*
 * bsgemm_run -- out = epilogue(X * W^T) on `stream`.
 *   act     DEVICE pointer, int8 [M][K] row-major (row stride K bytes).
 *   M       tokens, M >= 0; M = 0 is a no-op returning BSGEMM_OK.
 *   out     DEVICE pointer, [M][N] row-major of int32 / float / int8 by
 *           epi.kind; 16-byte aligned; must not overlap act.
 *   epi     epilogue kind and, for int8 kinds, the output scale.
 *   stream  a cudaStream_t (NULL = the legacy default stream).
 * Asynchronous: returns after enqueueing one kernel launch; allocates
 * nothing, does not synchronise and keeps no reference to act or out.  The
 * current device must be the one the handle was created on.  When K is a
 * multiple of 16 and act is 16-byte aligned (the fast path) the kernel
 * brings each 64-token tile of act into shared memory by tensor copies and
 * transposes it there; otherwise it gathers the tile with per-thread loads.
 * Returns BSGEMM_OK, BSGEMM_ERR_INVALID (NULL handle or pointers, M < 0,
 * bad kind, bad out_scale, misaligned out, wrong device) or
 * BSGEMM_ERR_CUDA (launch failure).
 */
int bsgemm_run(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* stream);

/*
 * bsgemm_workspace_bytes -- device workspace bsgemm_run_ws needs for M
 * tokens: a token-tiled, column-major copy of the activations
 * (ceil(M / T) * round_up(K, 16) * T bytes, T = bsgemm_info()[4]).
 * Returns 0 for M <= 0 or a NULL handle.
 */
size_t bsgemm_workspace_bytes(bsgemm_t h, int M);

/*
 * bsgemm_run_ws -- bsgemm_run with a caller-owned DEVICE workspace of at
 * least bsgemm_workspace_bytes(h, M) bytes, 16-byte aligned.  On bsgemm_run's
 * fast path (K % 16 == 0, act 16-byte aligned) it is that one kernel and the
 * workspace is not touched.  Otherwise it enqueues two kernels on `stream`:
 * one rewrites act as token tiles into the workspace, the second streams
 * each tile into shared memory with one bulk (TMA) copy and computes the
 * layer (faster than bsgemm_run's per-thread gather for those shapes).  The
 * workspace is scratch: its contents are undefined afterwards, and two runs
 * in flight at the same time need two workspaces.  Same results, return
 * codes and asynchrony as bsgemm_run; a workspace that is NULL, too small or
 * misaligned returns BSGEMM_ERR_INVALID.
 */
int bsgemm_run_ws(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                  size_t workspace_bytes, void* stream);

/*
 * bsgemm_run_static -- bsgemm_run_ws without a caller workspace and without
 * any allocation: on bsgemm_run's fast path nothing but that kernel runs;
 * otherwise the token tiles go to a fixed scratch array of
 * BSGEMM_STATIC_SCRATCH_BYTES (16 MiB) that the library holds in device
 * memory, one per device.  The paper has no counterpart; this entry point
 * serves callers that must not allocate at run time.
 *   Limit, only where the scratch is used (K % 16 != 0, or act not 16-byte
 *   aligned): bsgemm_workspace_bytes(h, M) <= BSGEMM_STATIC_SCRATCH_BYTES,
 *   i.e. M <= floor(16 MiB / (round_up(K, 16) * T)) * T tokens
 *   (T = bsgemm_info()[4]; M <= 5440 at K = 3072, M <= 21824 at K = 768).
 *   A larger M there returns BSGEMM_ERR_INVALID (use bsgemm_run_ws); on the
 *   fast path any M is accepted.
 *   Set-up: the first call on each device looks up the scratch array's
 *   address (cudaGetSymbolAddress) with that device current and caches it;
 *   make that first call before any stream capture.
 *   Races: every call on a device uses the same scratch, whatever the
 *   handle, stream or thread.  Two calls whose kernels overlap in time race
 *   and give undefined output; serialise them (one stream, or events).
 *   Nothing has to start at zero: each run writes every scratch byte it
 *   reads.
 * Results, return codes, asynchrony and the other arguments are those of
 * bsgemm_run_ws.
 */
#define BSGEMM_STATIC_SCRATCH_BYTES (16u << 20)
int bsgemm_run_static(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* stream);

/*
 * bsgemm_run_kmajor -- bsgemm_run on activations stored K-major: act_t is
 * X^T, int8 [K][M] with row stride ld bytes (row k = input feature k of the
 * M tokens, tokens contiguous), the input layout of Algorithm 1, whose
 * inner loop reads a k-block of input rows that each hold n-block
 * consecutive tokens.  Each 64-token tile then comes into shared memory by
 * tensor copies that land it directly in the kernel's layout: no transpose
 * and no relayout, one kernel, no scratch.
 *   act_t  DEVICE, 16-byte aligned; ld >= M and ld % 16 == 0.
 *   out    DEVICE [M][N] row-major as for bsgemm_run.
 * Results, asynchrony and the other return codes are bsgemm_run's.
 */
int bsgemm_run_kmajor(bsgemm_t h, const int8_t* act_t, int M, int ld, void* out, bsgemm_epilogue epi, void* stream);

/*
 * The two steps of bsgemm_run_ws, for callers that keep activations in the
 * token-tiled layout between layers or time the steps apart:
 *   bsgemm_tile_activations -- act [M][K] (DEVICE) -> token tiles in
 *     `tiles` (DEVICE, >= bsgemm_workspace_bytes(h, M) bytes, 16-byte
 *     aligned): tile t = tokens tT..tT+T-1, stored column by column (all T
 *     tokens' bytes of column k, then of column k+1, ...), columns padded to
 *     round_up(K, 16) and tokens past M with zeros, T = bsgemm_info()[4].
 *   bsgemm_run_tiled -- the layer from such tiles (one kernel).
 * Both are asynchronous on `stream` and return BSGEMM_OK or BSGEMM_ERR_*.
 */
int bsgemm_tile_activations(bsgemm_t h, const int8_t* act, int M, void* tiles, size_t tiles_bytes, void* stream);
int bsgemm_run_tiled(bsgemm_t h, const void* tiles, size_t tiles_bytes, int M, void* out, bsgemm_epilogue epi,
                     void* stream);

/*
 * bsgemm_run_host -- the end-to-end call on HOST buffers: copy act in, run
 * the layer (as bsgemm_run_ws does), copy the result out, all
 * enqueued on `stream`.  The paper's engine (Sec. 3) runs on the CPU and
 * takes and returns tensors in host memory; this is that call on the GPU,
 * with the transfers over the host link inside it.
 *   act        HOST int8 [M][K] row-major.
 *   out        HOST [M][N] row-major of the epilogue's type.
 *              Both should be page-locked (cudaHostAlloc/cudaHostRegister):
 *              then the two copies are asynchronous.  Pageable buffers
 *              work, with CUDA's pageable-copy behaviour (the calling
 *              thread blocks on the copies).
 *   workspace  DEVICE, >= bsgemm_host_workspace_bytes(h, M, epi.kind)
 *              bytes, 16-byte aligned: the activations' copy, their token
 *              tiles and the device result, each at a 256-byte aligned
 *              offset.  Scratch as for bsgemm_run_ws: two calls in flight
 *              at the same time need two workspaces.
 * Returns after enqueueing (two copies, one or two kernels); `out` holds the
 * result once `stream` has completed, and `act` must not change before
 * then.  Return codes as bsgemm_run_ws, plus BSGEMM_ERR_CUDA if a copy
 * cannot be enqueued.
 */
size_t bsgemm_host_workspace_bytes(bsgemm_t h, int M, int32_t kind);
int bsgemm_run_host(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                    size_t workspace_bytes, void* stream);

/*
 * bsgemm_block_prune -- the create-side pruning step (App. A.1): score each
 * 4x1 block of a dense weight by the mean magnitude of its 4 values and
 * prune the lowest-scoring ones until the sparsity ratio is reached.
 *   N, K      weight shape; N a multiple of 4, N >= 4, K >= 1.
 *   W         DEVICE float [N][K] row-major; every value finite.
 *   sparsity  fraction of blocks pruned, 0 <= sparsity <= 1: the number
 *             pruned is floor(sparsity * (N/4 * K) + 0.5).
 *   keep      DEVICE uint8 [N/4][K]: written 1 for a kept block, 0 for a
 *             pruned one.
 * Scores are computed in double as (((|w0| + |w1|) + |w2|) + |w3|) / 4,
 * w_i = W[4r + i][k], in that order; equal scores prune the lower block
 * index r * K + k first, so the mask is unique.  Runs on `stream` on the
 * current device with stream-ordered scratch (8 bytes per block) and
 * synchronises `stream` before returning.  Returns the number of kept
 * blocks, or BSGEMM_ERR_INVALID (bad shape, pointer or sparsity, or a
 * non-finite weight; `keep` is then undefined) or BSGEMM_ERR_CUDA.
 */
int64_t bsgemm_block_prune(int N, int K, const float* W, double sparsity, uint8_t* keep, void* stream);

/*
 * bsgemm_layernorm -- LayerNorm of each row of z (the post-operator that
 * Sec. 3's optimized INT8 graph fuses after the output projection and FFN2;
 * with BSGEMM_OUT_F32_RESID the residual add before it happens in the
 * linear's epilogue):
 *   out[m][n] = (z[m][n] - mean_m) / sqrt(var_m + eps) * gamma[n] + beta[n]
 * in fp32: the row mean as the first value plus the mean of the
 * deviations from it, the variance from the centred squares, then one fmaf
 * with gamma and beta; for int8 output requantised as the linear's
 * epilogue does.
 *   z      DEVICE float [M][N];  gamma, beta DEVICE float [N].
 *   out    DEVICE [M][N], float (epi.kind BSGEMM_OUT_F32) or int8
 *          (BSGEMM_OUT_I8, epi.out_scale as for bsgemm_run); must not overlap z.
 *   eps    >= 0, finite.
 * One kernel (a warp a row) on `stream`, asynchronous; M = 0 is a no-op.
 * Returns BSGEMM_OK, BSGEMM_ERR_INVALID or BSGEMM_ERR_CUDA.
 */
int bsgemm_layernorm(const float* z, int M, int N, const float* gamma, const float* beta, float eps, void* out,
                     bsgemm_epilogue epi, void* stream);

/*
 * bsgemm_attention -- multi-head self-attention on the int8 output of the
 * QKV linear: the two Matmuls and the softmax between the QKV and output
 * projections of Sec. 3's optimized INT8 graph (the paper leaves their form
 * implicit; this is scaled dot-product attention, no mask).  For sequence
 * b, head h and query t:
 *   s_j   = (q_t . k_j) * qkv_scale^2 / sqrt(head_dim)   (q . k exact, int32)
 *   out_t = sum_j exp(s_j - max s) v_j * qkv_scale / sum_j exp(s_j - max s)
 * in fp32 after the exact dot product; for int8 output requantised as the
 * linear's epilogue does.
 *   qkv    DEVICE int8, rows of ld bytes: token row m = b * seq + t holds
 *          q (bytes 0 .. d-1), k (d .. 2d-1) and v (2d .. 3d-1), d = heads
 *          * head_dim; head h is bytes h * head_dim .. of each third (the
 *          QKV linear's int8 output, ld = 3d).  16-byte aligned.
 *   ld     >= 3d, a multiple of 16.
 *   qkv_scale  the int8 scale of q, k and v: finite, > 0, with
 *          qkv_scale^2 / sqrt(head_dim) a normal fp32 number below 2^100.
 *   out    DEVICE [batch * seq][d], float (epi.kind BSGEMM_OUT_F32) or
 *          int8 (BSGEMM_OUT_I8, epi.out_scale as for bsgemm_run);
 *          16-byte aligned; must not overlap qkv.  epi.flags may be
 *          BSGEMM_ACT_READY (qkv was complete before the stream's
 *          preceding kernel began: the kernel then reads it while that
 *          kernel still runs; out is written after it either way).  Other
 *          epi fields unused.
 * head_dim must be 64 and seq <= BSGEMM_ATTN_MAX_SEQ (else
 * BSGEMM_ERR_UNSUPPORTED); 1 <= heads <= 65535, 0 <= batch <= 65535, seq >=
 * 1 unless batch = 0 (a no-op).  One kernel on `stream`, asynchronous.
 * Returns BSGEMM_OK, BSGEMM_ERR_INVALID, BSGEMM_ERR_UNSUPPORTED or
 * BSGEMM_ERR_CUDA.
 */
#define BSGEMM_ATTN_MAX_SEQ 512
int bsgemm_attention(const int8_t* qkv, int batch, int seq, int heads, int head_dim, int ld, float qkv_scale,
                     void* out, bsgemm_epilogue epi, void* stream);

/*
 * bsgemm_attention_status -- read (and with clear != 0, reset) the current
 * device's attention status word: 0 when every wait of the attention
 * kernel's launches completed; BSGEMM_STATUS_TIMEOUT when one gave up (a
 * tensor-core MMA did not complete within the wait's limit; that launch's
 * out is incomplete).  Synchronises the device.  Returns the status, or a
 * negative BSGEMM_ERR_* code.
 */
int bsgemm_attention_status(int clear);

/*
 * bsgemm_device_status -- read (and with clear != 0, reset) the handle's
 * device status word.  0 means every wait in the kernels completed; bit 0
 * (BSGEMM_STATUS_TIMEOUT) means a bounded wait on an asynchronous copy gave
 * up and that run's output is incomplete.  Synchronises the device.  Returns
 * the status, or a negative BSGEMM_ERR_* code.
 */
#define BSGEMM_STATUS_TIMEOUT 1
int bsgemm_device_status(bsgemm_t h, int clear);

/*
 * bsgemm_set_test_hooks -- make the bounded waits give up on purpose, so
 * that a test can check the failure path without faulting or hanging a GPU
 * (the paper has no counterpart; its engine runs on a CPU).  The bits apply
 * to every later launch in the process until they are set back to 0:
 *   BSGEMM_TEST_SKIP_TILE_COPY: the layer kernel issues no copy of a token
 *     tile and gives each wait on one up after 64 polls.  No copy is then in
 *     flight when a CTA leaves; the run's output is undefined and the
 *     handle's device status gets BSGEMM_STATUS_TIMEOUT.  Staging by
 *     per-thread loads (no copies) is unaffected.
 *   BSGEMM_TEST_STALL_PRUNE_CTA: CTA 0 of the pruning kernel leaves before
 *     its first grid barrier and the other CTAs give that barrier up after
 *     4096 polls; every CTA returns and bsgemm_block_prune returns
 *     BSGEMM_ERR_CUDA (keep is undefined).
 *   BSGEMM_TEST_ATTN_SKIP_MMA: the attention kernel issues no tensor-core
 *     MMA and gives each wait on one up after 64 polls (nothing is then in
 *     flight when a CTA leaves); out is undefined and
 *     bsgemm_attention_status reports BSGEMM_STATUS_TIMEOUT.
 * Not for production use.  Returns the previous bits.
 */
#define BSGEMM_TEST_SKIP_TILE_COPY 1u
#define BSGEMM_TEST_STALL_PRUNE_CTA 2u
#define BSGEMM_TEST_ATTN_SKIP_MMA 4u
uint32_t bsgemm_set_test_hooks(uint32_t bits);

/*
 * bsgemm_destroy -- free the handle and its device memory.  The caller must
 * make sure no bsgemm_run on this handle is still executing (cudaFree
 * itself waits for the device).  NULL is ignored.
 */
void bsgemm_destroy(bsgemm_t h);

/*
 * bsgemm_int8_peak -- measure the peak rate of one int8 dot-product unit of
 * the current device, the denominator of the layer's roofline (the layer is
 * Algorithm 1's int8 dot-4 contraction; the paper has no counterpart of
 * this measurement).  unit 0: dp4a (4 int8 multiply-adds into int32 per lane,
 * the unit the layer kernel runs on); unit 1: mma.sync m16n8k32 s8 x s8 ->
 * s32 (the warp-level tensor-core instruction).  A probe kernel runs `iters`
 * loop iterations on every SM, four times; *tops receives the best of the
 * last three as 10^12 ops/s (2 ops per multiply-add).  Allocates a few bytes
 * of device memory and synchronises the device: a measurement helper, not
 * for use while other work runs.  Returns BSGEMM_OK, BSGEMM_ERR_INVALID
 * (unit not 0 or 1, iters < 1, tops NULL) or BSGEMM_ERR_CUDA.
 */
int bsgemm_int8_peak(int unit, int iters, double* tops);

/* Message for the last failure on the calling thread ("" if none).  The
 * string stays valid until the next bsgemm_* call on this thread. */
const char* bsgemm_last_error(void);

/* Code (BSGEMM_OK or BSGEMM_ERR_*) of the last bsgemm_* call on the calling
 * thread; tells why bsgemm_create returned NULL. */
int bsgemm_last_status(void);

/* Largest K bsgemm_create accepts in this build (bounded by the shared
 * memory that holds one token tile of activations for all of K). */
int bsgemm_max_k(void);

/*
 * bsgemm_info -- describe a handle, for benchmarks and tests.  Fills up to
 * `n` entries of `out` with: [0] N, [1] K, [2] nnzb (stored blocks),
 * [3] padded quads (groups of 4 stored blocks of one block-row, the unit of
 * the inner loop; the last quad of a block-row is padded with zero-weight
 * entries), [4] token-tile height of the kernel, [5] CTAs of a launch once
 * M is large enough to fill the GPU (SMs x resident CTAs per SM), [6] device
 * bytes held by the handle (the tensor-core operands' allocation included).
 * Returns the number of entries available (7), or BSGEMM_ERR_INVALID.
 */
int bsgemm_info(bsgemm_t h, int64_t* out, int n);

#ifdef __cplusplus
}
#endif

#endif /* BSGEMM_H_ */
