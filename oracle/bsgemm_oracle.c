/*
 * CPU oracle for the block-sparse INT8 linear layer of "Fast DistilBERT on
 * CPUs" (arXiv 2211.07715).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * definition that the CUDA path is checked against.  Only the test suite, the
 * smoke check and the benchmark's CPU-baseline leg may load it.  It shares no
 * code, header, table or helper with the CUDA library, and the CUDA library
 * never calls it.
 *
 * What it computes (paper Sec. 3 "Sparse GEMM operators", App. A.3.4 and
 * Algorithm 1): a dense int8 input times a weight that is sparse in blocks of
 * 4 consecutive output rows x 1 input column (App. A.1), accumulated exactly
 * in int32 (the VNNI dot-4 of Algorithm 1), followed by the fused post-ops
 * (App. A.3.3: bias and further post-operators fused into the InnerProduct):
 * per-output-channel dequantisation + bias, optional erf-GELU, optional
 * requantisation to int8.
 *
 * Readings of the paper used here (the paper leaves these open):
 *   - block orientation: 4 consecutive output rows x 1 column (App. A.1);
 *   - activations and weights are signed int8, symmetric, no zero point
 *     (the u8 x s8 of vpdpbusd in Algorithm 1 is an ISA artefact);
 *   - scales[n] is the combined activation x weight scale of channel n;
 *   - dequantisation is y = fmaf((float)acc, scale[n], bias[n]) in fp32;
 *   - requantisation is q = saturate_s8(round_half_even(y * inv_out_scale))
 *     with inv_out_scale = 1.0f / out_scale computed once in fp32;
 *   - the epilogue runs once after the full K reduction (Algorithm 1 prints
 *     it inside the k loop; that placement is read as a typesetting slip).
 *
 * Precision: the accumulator is exact (int64 here, range-checked to int32).
 * fp32-output epilogues are given in fp64 (the exact value the fp32 kernel
 * approximates).  Where floating point decides an integer (requantisation),
 * the decision is taken in fp32, the precision the kernel computes in, by the
 * op sequence stated next to each function.
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off -fPIC -shared (no -ffast-math:
 * every fp32 operation below must be a single IEEE round-to-nearest-even op).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_BLOCK 4

/* Output kinds, numbered as in the library's public header (both follow the
 * same five epilogues; the numbering is an interface, not shared code). */
enum { O_I32 = 0, O_F32 = 1, O_F32_GELU = 2, O_I8 = 3, O_I8_GELU = 4 };

/* ---------------------------------------------------------------------- */
/* Block-compressed weight format (App. A.1: 1-D blocks of 4 along the     */
/* output dimension; App. A.3.4: "the sparse weight is compressed and the  */
/* mask is used").                                                          */
/*                                                                          */
/* indptr[N/4 + 1], colidx[nnzb], values[nnzb][4]: block j of block-row r   */
/* (indptr[r] <= j < indptr[r+1]) sits in column colidx[j] and holds the    */
/* weights of output rows 4r+0..4r+3 in that column.                        */
/* Returns 0, or -1 when the arrays do not describe a valid matrix.         */
/* ---------------------------------------------------------------------- */
int oracle_bsr_to_dense(int N, int K, const int32_t* indptr, const int32_t* colidx,
                        const int8_t* values, int8_t* W /* [N][K] */) {
    if (N < 0 || K < 0 || N % ORACLE_BLOCK != 0) return -1;
    int nbr = N / ORACLE_BLOCK;
    if (indptr[0] != 0) return -1;
    memset(W, 0, (size_t)N * (size_t)K);
    for (int r = 0; r < nbr; ++r) {
        if (indptr[r + 1] < indptr[r]) return -1;
        for (int j = indptr[r]; j < indptr[r + 1]; ++j) {
            int k = colidx[j];
            if (k < 0 || k >= K) return -1;
            if (j > indptr[r] && colidx[j - 1] >= k) return -1; /* sorted, unique */
            for (int i = 0; i < ORACLE_BLOCK; ++i)
                W[(size_t)(ORACLE_BLOCK * r + i) * K + k] = values[(size_t)j * ORACLE_BLOCK + i];
        }
    }
    return 0;
}

/* Dense -> block-compressed, keeping exactly the blocks whose mask entry is
 * nonzero (mask[r][k], r < N/4).  A kept block may contain zero values.
 * Returns nnzb; indptr must hold N/4+1 entries, colidx/values room for all
 * kept blocks (pass NULL for both to only count). */
int oracle_dense_to_bsr(int N, int K, const int8_t* W, const uint8_t* mask,
                        int32_t* indptr, int32_t* colidx, int8_t* values) {
    int nbr = N / ORACLE_BLOCK, nnzb = 0;
    if (indptr) indptr[0] = 0;
    for (int r = 0; r < nbr; ++r) {
        for (int k = 0; k < K; ++k) {
            if (!mask[(size_t)r * K + k]) continue;
            if (colidx) colidx[nnzb] = k;
            if (values)
                for (int i = 0; i < ORACLE_BLOCK; ++i)
                    values[(size_t)nnzb * ORACLE_BLOCK + i] = W[(size_t)(ORACLE_BLOCK * r + i) * K + k];
            ++nnzb;
        }
        if (indptr) indptr[r + 1] = nnzb;
    }
    return nnzb;
}

/* ---------------------------------------------------------------------- */
/* Accumulation (Sec. 3: "the kernel uses VNNI to produce the intermediate */
/* output"; Algorithm 1: vpdpbusd dot-4 into int32).                        */
/* acc[m][n] = sum_k X[m][k] * W[n][k] over the decompressed W, every k,    */
/* no skipping.  Rows m in [row0, row1) only.  Returns 0, or -2 if a sum    */
/* leaves the int32 range (the kernel's accumulator would wrap).            */
/* ---------------------------------------------------------------------- */
int oracle_acc(int M, int N, int K, const int8_t* X /* [M][K] */, const int8_t* W /* [N][K] */,
               int32_t* acc /* [M][N] */, int row0, int row1) {
    (void)M;
    for (int m = row0; m < row1; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t s = 0;
            for (int k = 0; k < K; ++k)
                s += (int64_t)X[(size_t)m * K + k] * (int64_t)W[(size_t)n * K + k];
            if (s > INT32_MAX || s < INT32_MIN) return -2;
            acc[(size_t)m * N + n] = (int32_t)s;
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Epilogue pieces (Sec. 3: "add bias C as the final output"; App. A.3.3:  */
/* post-operators fused into the InnerProduct; Algorithm 1: "downconvert   */
/* and post-operator fusion").                                              */
/* ---------------------------------------------------------------------- */

/* Dequantisation in fp32, the precision the requantisation decision is
 * taken in: int32 -> fp32 (round to nearest even), then one fused
 * multiply-add with a single rounding. */
float oracle_dequant_f32(int32_t acc, float scale, float bias) {
    return fmaf((float)acc, scale, bias);
}

/* Exact-valued reference for fp32 outputs: acc * scale + bias in fp64. */
double oracle_dequant_f64(int32_t acc, float scale, float bias) {
    return (double)acc * (double)scale + (double)bias;
}

/* erf-form GELU in fp64: 0.5 y (1 + erf(y / sqrt 2)). */
double oracle_gelu_f64(double y) {
    return 0.5 * y * (1.0 + erf(y / sqrt(2.0)));
}

/* 1/b for 1 <= b < 2^25 by Newton's method for the reciprocal, as a fixed
 * sequence of IEEE fp32 operations (round to nearest even), so that every
 * machine gets the same bits:
 *   b = m 2^E with 1 <= m < 2 (exact, from the bits of b)
 *   y0 = fma(-8/17, m, 24/17)   (the minimax straight line for 1/m on [1, 2),
 *                                relative error <= 1/17; both constants rounded
 *                                to fp32: 0x1.e1e1e2p-2, 0x1.69696ap+0)
 *   y_{i+1} = fma(y_i, fma(-m, y_i, 1), y_i),  i = 0, 1, 2
 *                               (each step squares the relative error:
 *                                1/17 -> 3.5e-3 -> 1.2e-5 -> 1.5e-10)
 *   1/b = y3 * 2^-E             (exact: a power of two, result normal)
 * The result is within about half an ulp of 1/b; it need not be the
 * correctly rounded quotient. */
float oracle_recip_f32(float b) {
    uint32_t bits;
    memcpy(&bits, &b, sizeof bits);
    const int E = (int)((bits >> 23) & 0xffu) - 127;
    const uint32_t mbits = (bits & 0x7fffffu) | (127u << 23);
    float m;
    memcpy(&m, &mbits, sizeof m);
    float y = fmaf(-0x1.e1e1e2p-2f, m, 0x1.69696ap+0f);
    for (int i = 0; i < 3; ++i) {
        const float e = fmaf(-m, y, 1.0f);
        y = fmaf(y, e, y);
    }
    const uint32_t sbits = (uint32_t)(127 - E) << 23;
    float s2;
    memcpy(&s2, &sbits, sizeof s2);
    return y * s2;
}

/* erf-form GELU evaluated in fp32 by a fixed op sequence, so that an int8
 * result decided from it is reproducible on any IEEE machine.  erf comes from
 * Abramowitz & Stegun, Handbook of Mathematical Functions, formula 7.1.28:
 *   erf(x) = 1 - (1 + a1 x + a2 x^2 + a3 x^3 + a4 x^4 + a5 x^5 + a6 x^6)^-16,
 *   x >= 0, |error| <= 3e-7, and erf(-x) = -erf(x).
 * Op sequence (each step one IEEE fp32 operation, round to nearest even):
 *   x  = y * 0.70710678f            (1/sqrt 2 rounded to fp32)
 *   ax = |x|
 *   h  = fma(ax, a6, a5); h = fma(ax, h, a4); h = fma(ax, h, a3);
 *   h  = fma(ax, h, a2);  h = fma(ax, h, a1); p = fma(ax, h, 1)
 *   p2 = p*p; p4 = p2*p2; p8 = p4*p4; p16 = p8*p8
 *   e  = 1 if p16 >= 2^25, else 1 - recip(p16)  (recip: Newton's method
 *        above; from p16 = 2^25 on, 1 - 1/p16 rounds to 1 in fp32 for the
 *        exact quotient too: 1 - 2^-25 is a tie, rounded to even)
 *   erf = (x < 0) ? -e : e
 *   g  = (0.5 * y) * (1 + erf)                                            */
float oracle_gelu_f32(float y) {
    const float a1 = 0.0705230784f, a2 = 0.0422820123f, a3 = 0.0092705272f;
    const float a4 = 0.0001520143f, a5 = 0.0002765672f, a6 = 0.0000430638f;
    float x = y * 0.70710678f;
    float ax = fabsf(x);
    float h = fmaf(ax, a6, a5);
    h = fmaf(ax, h, a4);
    h = fmaf(ax, h, a3);
    h = fmaf(ax, h, a2);
    h = fmaf(ax, h, a1);
    float p = fmaf(ax, h, 1.0f);
    float p2 = p * p;
    float p4 = p2 * p2;
    float p8 = p4 * p4;
    float p16 = p8 * p8;
    float e = (p16 >= 0x1p25f) ? 1.0f : 1.0f - oracle_recip_f32(p16);
    float erfv = (x < 0.0f) ? -e : e;
    float half_y = 0.5f * y;
    float one_plus = 1.0f + erfv;
    return half_y * one_plus;
}

/* Requantisation: t = v * inv (one fp32 multiply), then round half to even
 * and saturate to [-128, 127]. */
int8_t oracle_requant(float v, float inv_out_scale) {
    float t = v * inv_out_scale;
    float r = nearbyintf(t); /* default rounding mode: to nearest, ties to even */
    if (r > 127.0f) return 127;
    if (r < -128.0f) return -128;
    return (int8_t)r;
}

/* ---------------------------------------------------------------------- */
/* The whole linear layer for rows [row0, row1): accumulation then the      */
/* epilogue `kind` per element.  Output element type by kind:               */
/*   I32 -> int32 acc;  F32 -> double y;  F32_GELU -> double GELU(y);       */
/*   I8 -> int8 requant(fp32 y);  I8_GELU -> int8 requant(gelu_f32(fp32 y)). */
/* bias may be NULL (zeros).  Returns 0, -1 bad kind/scale, -2 overflow.    */
/* ---------------------------------------------------------------------- */
int oracle_linear(int M, int N, int K, const int8_t* X, const int8_t* W, const float* scales,
                  const float* bias, int kind, float out_scale, void* out, int row0, int row1) {
    if (kind < O_I32 || kind > O_I8_GELU) return -1;
    float inv = 0.0f;
    if (kind == O_I8 || kind == O_I8_GELU) {
        if (!(out_scale > 0.0f) || !isfinite(out_scale)) return -1;
        inv = 1.0f / out_scale;
    }
    int32_t* acc = (int32_t*)malloc(sizeof(int32_t) * (size_t)N);
    if (!acc) return -3;
    for (int m = row0; m < row1; ++m) {
        /* one row at a time so that a row sample needs O(N) scratch */
        int rc = oracle_acc(M, N, K, X + (size_t)m * K, W, acc, 0, 1);
        if (rc) { free(acc); return rc; }
        for (int n = 0; n < N; ++n) {
            size_t o = (size_t)m * N + n;
            float b = bias ? bias[n] : 0.0f;
            switch (kind) {
            case O_I32: ((int32_t*)out)[o] = acc[n]; break;
            case O_F32: ((double*)out)[o] = oracle_dequant_f64(acc[n], scales[n], b); break;
            case O_F32_GELU:
                ((double*)out)[o] = oracle_gelu_f64(oracle_dequant_f64(acc[n], scales[n], b));
                break;
            case O_I8:
                ((int8_t*)out)[o] = oracle_requant(oracle_dequant_f32(acc[n], scales[n], b), inv);
                break;
            case O_I8_GELU:
                ((int8_t*)out)[o] =
                    oracle_requant(oracle_gelu_f32(oracle_dequant_f32(acc[n], scales[n], b)), inv);
                break;
            }
        }
    }
    free(acc);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Residual add before LayerNorm (the post-operators the optimized INT8     */
/* graph fuses after an InnerProduct, Sec. 3 "Graph optimization"; the     */
/* encoder adds the sub-layer's input before its LayerNorm).  For rows      */
/* [row0, row1) of the layer:                                               */
/*   y = fmaf((float)acc, scale[n], bias[n])            (fp32, as above)    */
/*   z = y + (res_scale * (float)r[m][n])               (two fp32 ops,     */
/*                                                       multiply first)    */
/* r is the int8 residual [M][N] (the sub-layer's input in the int8 chain)  */
/* with its per-tensor scale.  Writes z (fp32) to out[M][N].                */
/* Returns 0, -2 on accumulator overflow, -3 out of memory.                 */
/* ---------------------------------------------------------------------- */
int oracle_linear_resid(int M, int N, int K, const int8_t* X, const int8_t* W, const float* scales,
                        const float* bias, const int8_t* R, float res_scale, float* out, int row0, int row1) {
    int32_t* acc = (int32_t*)malloc(sizeof(int32_t) * (size_t)(N > 0 ? N : 1));
    if (!acc) return -3;
    for (int m = row0; m < row1; ++m) {
        int rc = oracle_acc(M, N, K, X + (size_t)m * K, W, acc, 0, 1);
        if (rc) { free(acc); return rc; }
        for (int n = 0; n < N; ++n) {
            size_t o = (size_t)m * N + n;
            float y = oracle_dequant_f32(acc[n], scales[n], bias ? bias[n] : 0.0f);
            float rs = res_scale * (float)R[o];
            out[o] = y + rs;
        }
    }
    free(acc);
    return 0;
}

/* LayerNorm over the N channels of each row (the LayerNorm the optimized    */
/* INT8 graph fuses, Sec. 3 "Graph optimization"):                          */
/*   mu = (1/N) sum_n z[n],  var = (1/N) sum_n (z[n] - mu)^2,                */
/*   out[n] = (z[n] - mu) / sqrt(var + eps) * gamma[n] + beta[n],            */
/* in fp64 (the exact value the fp32 kernel approximates; the paper fixes    */
/* no summation order).  Two passes over the row: the mean, then the         */
/* centred squares.                                                         */
void oracle_layernorm(int M, int N, const float* Z, const float* gamma, const float* beta, double eps,
                      double* out) {
    for (int m = 0; m < M; ++m) {
        const float* z = Z + (size_t)m * N;
        double sum = 0.0;
        for (int n = 0; n < N; ++n) sum += (double)z[n];
        double mu = sum / (double)N;
        double sq = 0.0;
        for (int n = 0; n < N; ++n) {
            double d = (double)z[n] - mu;
            sq += d * d;
        }
        double var = sq / (double)N;
        double inv_sd = 1.0 / sqrt(var + eps);
        for (int n = 0; n < N; ++n)
            out[(size_t)m * N + n] = ((double)z[n] - mu) * inv_sd * (double)gamma[n] + (double)beta[n];
    }
}

/* ---------------------------------------------------------------------- */
/* Block-wise pruning with the average-magnitude heuristic (App. A.1): the  */
/* score of a 4x1 block is the mean |w| of its four weights; the blocks     */
/* with the lowest scores are pruned until the required sparsity ratio is   */
/* reached.  Number pruned = round(sparsity * total), halves away from 0.   */
/* Equal scores: the block with the lower index r*K + k is pruned first.    */
/* Writes keep[r][k] = 1 for kept blocks.  Returns the number kept.         */
/* ---------------------------------------------------------------------- */
typedef struct { double score; int64_t id; } oracle_scored;

static int cmp_scored(const void* a, const void* b) {
    const oracle_scored* x = (const oracle_scored*)a;
    const oracle_scored* y = (const oracle_scored*)b;
    if (x->score < y->score) return -1;
    if (x->score > y->score) return 1;
    return (x->id < y->id) ? -1 : (x->id > y->id);
}

int64_t oracle_block_prune(int N, int K, const float* W /* [N][K] */, double sparsity,
                           uint8_t* keep /* [N/4][K] */) {
    int nbr = N / ORACLE_BLOCK;
    int64_t total = (int64_t)nbr * K;
    oracle_scored* s = (oracle_scored*)malloc(sizeof(oracle_scored) * (size_t)(total ? total : 1));
    if (!s) return -1;
    for (int r = 0; r < nbr; ++r)
        for (int k = 0; k < K; ++k) {
            double sum = 0.0;
            for (int i = 0; i < ORACLE_BLOCK; ++i) sum += fabs((double)W[(size_t)(ORACLE_BLOCK * r + i) * K + k]);
            s[(int64_t)r * K + k].score = sum / ORACLE_BLOCK;
            s[(int64_t)r * K + k].id = (int64_t)r * K + k;
        }
    qsort(s, (size_t)total, sizeof(oracle_scored), cmp_scored);
    int64_t npruned = (int64_t)floor(sparsity * (double)total + 0.5);
    if (npruned > total) npruned = total;
    if (npruned < 0) npruned = 0;
    for (int64_t i = 0; i < total; ++i) keep[s[i].id] = (i >= npruned);
    free(s);
    return total - npruned;
}

/* ---------------------------------------------------------------------- */
/* Multi-head self-attention on the int8 QKV projection: the two Matmuls   */
/* and the softmax between the QKV and output linears of the INT8 graph    */
/* (Sec. 3 "Graph optimization" fuses post-operators into InnerProduct and */
/* Matmul alike).  The paper does not write attention out; this is the     */
/* standard scaled dot-product form over the heads of DistilBERT:          */
/*   row m = b * seq + t of QKV holds q | k | v, each heads * hd wide,     */
/*   int8 times qkv_scale;                                                 */
/*   for sequence b, head h and query t (columns h*hd .. h*hd + hd - 1):   */
/*     s_j   = (q_t . k_j) / sqrt(hd)                 j = 0 .. seq - 1     */
/*     p_j   = exp(s_j - max_j s_j) / sum_j exp(s_j - max_j s_j)           */
/*     out_t = sum_j p_j v_j                                               */
/* in fp64; every position of a sequence is a token (no mask).  Rows of   */
/* QKV are ld bytes apart; out is [batch * seq][heads * hd].  Returns 0,   */
/* or -1 on bad sizes / allocation failure.                                */
/* ---------------------------------------------------------------------- */
int oracle_attention(int batch, int seq, int heads, int hd, const int8_t* QKV, int ld, float qkv_scale,
                     double* out) {
    const int d = heads * hd;
    if (batch < 0 || seq < 1 || heads < 1 || hd < 1 || ld < 3 * d) return -1;
    double* s = (double*)malloc(sizeof(double) * (size_t)seq);
    if (!s) return -1;
    const double scale = (double)qkv_scale;
    const double inv_sqrt_hd = 1.0 / sqrt((double)hd);
    for (int b = 0; b < batch; ++b)
        for (int h = 0; h < heads; ++h)
            for (int t = 0; t < seq; ++t) {
                const int8_t* q = QKV + (size_t)(b * seq + t) * ld + h * hd;
                double smax = -INFINITY;
                for (int j = 0; j < seq; ++j) {
                    const int8_t* k = QKV + (size_t)(b * seq + j) * ld + d + h * hd;
                    double dot = 0.0;
                    for (int c = 0; c < hd; ++c) dot += ((double)q[c] * scale) * ((double)k[c] * scale);
                    s[j] = dot * inv_sqrt_hd;
                    if (s[j] > smax) smax = s[j];
                }
                double sum = 0.0;
                for (int j = 0; j < seq; ++j) {
                    s[j] = exp(s[j] - smax);
                    sum += s[j];
                }
                double* o = out + (size_t)(b * seq + t) * d + h * hd;
                for (int c = 0; c < hd; ++c) {
                    double acc = 0.0;
                    for (int j = 0; j < seq; ++j) {
                        const int8_t* v = QKV + (size_t)(b * seq + j) * ld + 2 * d + h * hd;
                        acc += (s[j] / sum) * ((double)v[c] * scale);
                    }
                    o[c] = acc;
                }
            }
    free(s);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Weights sparse in 1 x 4 blocks (one output row x 4 consecutive input    */
/* columns): the variant block shape along the reduction dimension, where  */
/* one block is exactly one dot-4 (the k_block = 4 of Algorithm 1 within   */
/* a single output row).  Row n holds blocks indptr[n] .. indptr[n+1]-1;   */
/* block e covers columns 4 colgrp[e] .. 4 colgrp[e] + 3 with values       */
/* values[e][0..3] in column order.  Decompresses into the dense W [N][K]  */
/* (K a multiple of 4).  Returns 0, or -1 if the arrays are invalid        */
/* (indptr not starting at 0 / decreasing, a group outside [0, K/4), or    */
/* groups of a row not strictly increasing).                               */
/* ---------------------------------------------------------------------- */
int oracle_bsr1x4_to_dense(int N, int K, const int32_t* indptr, const int32_t* colgrp, const int8_t* values,
                           int8_t* W) {
    if (N < 1 || K < 4 || K % 4 != 0 || indptr[0] != 0) return -1;
    memset(W, 0, (size_t)N * K);
    for (int n = 0; n < N; ++n) {
        if (indptr[n + 1] < indptr[n]) return -1;
        for (int32_t e = indptr[n]; e < indptr[n + 1]; ++e) {
            const int32_t j = colgrp[e];
            if (j < 0 || j >= K / 4) return -1;
            if (e > indptr[n] && colgrp[e - 1] >= j) return -1;
            for (int i = 0; i < 4; ++i) W[(size_t)n * K + 4 * j + i] = values[4 * (size_t)e + i];
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Weights with 2:4 structured sparsity along the input dimension: in each */
/* output row, each group of 4 consecutive input columns holds at most 2   */
/* nonzero weights (the pattern of sparse tensor cores the paper cites as  */
/* related work, Sec. 1).  Compressed form per row n and group g: two      */
/* values values[n][2g + t] at the in-group positions idx[n][2g + t]       */
/* (t = 0, 1; 0 <= idx < 4, strictly increasing within the group).         */
/* Decompresses into the dense W [N][K] (K a multiple of 4).  Returns 0,   */
/* or -1 on an invalid index.                                              */
/* ---------------------------------------------------------------------- */
int oracle_2to4_to_dense(int N, int K, const int8_t* values, const uint8_t* idx, int8_t* W) {
    if (N < 1 || K < 4 || K % 4 != 0) return -1;
    memset(W, 0, (size_t)N * K);
    const int half = K / 2;
    for (int n = 0; n < N; ++n)
        for (int g = 0; g < K / 4; ++g) {
            const uint8_t i0 = idx[(size_t)n * half + 2 * g], i1 = idx[(size_t)n * half + 2 * g + 1];
            if (i0 >= 4 || i1 >= 4 || i0 >= i1) return -1;
            W[(size_t)n * K + 4 * g + i0] = values[(size_t)n * half + 2 * g];
            W[(size_t)n * K + 4 * g + i1] = values[(size_t)n * half + 2 * g + 1];
        }
    return 0;
}
