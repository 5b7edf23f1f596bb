// Multi-head self-attention on the int8 output of the QKV linear: the two
// Matmuls and the softmax between the QKV and output projections of the
// optimized INT8 graph (Sec. 3 "Graph optimization").  The paper does not
// write the attention out; this is the standard scaled dot-product form.
// For sequence b, head h (64 channels) and query t:
//   s_j   = (q_t . k_j) * c,          c = qkv_scale^2 / sqrt(64)
//   e_j   = exp(s_j - max_j s_j)
//   out_t = (sum_j e_j v_j) * (qkv_scale / sum_j e_j)
// No attention mask: every position of a sequence is a token.
//
// Both contractions run on the fifth-generation tensor cores (tcgen05.mma
// kind::f16, f16 operands, fp32 accumulators in tensor memory):
//   * q k^T is exact: int8 values are exact in f16, the products (< 2^14)
//     are exact, and every partial sum of 64 of them stays below 2^24, so
//     the fp32 accumulator holds the int32 dot product;
//   * P v takes each weight in two f16 parts (e = hi + lo + r, |r| <= 2^-22
//     e + 2^-25) against the exact f16 v, two MMAs per K step.
// The softmax runs online over blocks of 128 keys in fp32: a thread keeps
// its query's running maximum m of the exact dot products and its running
// sum l; e_j = 2^((d_j - m) c log2(e)) with d_j - m exact, so the only
// roundings inside the exponent are those of c log2(e) and of one product.
// When m grows, the context and l are scaled by the same factor.
//
// One CTA = 128 queries of one (sequence, head), 4 warps; thread i owns
// query i = tensor-memory lane i.  Tensor memory (256 columns, so two CTAs
// share an SM): S/P in columns 0-127 (the block's scores, then its weights
// written back in place as f16 pairs: for keys 32c .. 32c + 31 the high
// parts in columns 32c .. 32c + 15, the low parts in 32c + 16 .. 32c + 31),
// the context O in 128-191, the CTA's queries (f16 pairs) in 192-223.  The
// head's keys and values (seq <= BSGEMM_ATTN_MAX_SEQ, padded with zeros to
// whole blocks) are staged once into shared memory as f16 rows of 64 with
// the 128-byte swizzle: K is the K-major B operand of q k^T, V the MN-major
// B operand of P v.  Per block one thread issues the 4 MMAs of S = Q K_b^T
// (N = 128, K = 64) and, after the threads have written P, the 16 of O +=
// P_hi V_b + P_lo V_b (N = 64, K = 128); completions arrive on two
// mbarriers, every wait bounded.
#include <cfloat>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda_fp16.h>

#include "bsgemm.h"
#include "bsgemm_device.cuh"
#include "bsgemm_internal.h"
#include "bsgemm_tcgen05.cuh"

namespace bsg {
namespace {

constexpr int kAttnThreads = 128;     // 4 warps, one query (TMEM lane) each
constexpr int kAttnQ = 128;           // queries per CTA
constexpr int kKeyBlock = 128;        // keys per online-softmax block
constexpr uint32_t kBlockBytes = 16384;  // 128 rows x 64 f16
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0, kColO = 128, kColQ = 192;
constexpr uint32_t kIdescS = f16_idesc(128, 128, false);  // S = Q K_b^T
constexpr uint32_t kIdescPV = f16_idesc(128, 64, true);   // O += P V_b

// Bit 0 set when a wait of the attention kernel gave up (per device).
__device__ unsigned g_attn_status;

__device__ __forceinline__ int4 ld_nc16(const int8_t* p) {
    return __ldg(reinterpret_cast<const int4*>(p));
}

// Two int8 values (bytes sel of the biased word u = w ^ 0x80808080) as an
// f16 pair, exactly: 0x64uu is the f16 1024 + uu, minus 1152 = the value.
__device__ __forceinline__ uint32_t s8x2_f16x2(uint32_t u, uint32_t sel) {
    const uint32_t b = __byte_perm(u, 0x64646464u, sel);
    __half2 h;
    memcpy(&h, &b, sizeof(h));
    h = __hsub2(h, __half2(__ushort_as_half(0x6480u), __ushort_as_half(0x6480u)));  // 1152
    uint32_t r;
    memcpy(&r, &h, sizeof(r));
    return r;
}

// 16 int8 values -> 8 f16 pairs, in order.
__device__ __forceinline__ void widen16(int4 v, uint32_t (&o)[8]) {
    const uint32_t w[4] = {static_cast<uint32_t>(v.x) ^ 0x80808080u, static_cast<uint32_t>(v.y) ^ 0x80808080u,
                           static_cast<uint32_t>(v.z) ^ 0x80808080u, static_cast<uint32_t>(v.w) ^ 0x80808080u};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        o[2 * q] = s8x2_f16x2(w[q], 0x4140u);
        o[2 * q + 1] = s8x2_f16x2(w[q], 0x4342u);
    }
}

// Rows 0 .. rows-1 (a multiple of 128) of one third of the head (src = its
// row 0, rows ld bytes apart) into a swizzled f16 tile; rows >= seq are
// zeros.  Row j, 16-byte chunk c (f16 8c .. 8c + 7) at j * 128 + (c ^ (j %
// 8)) * 16.
__device__ __forceinline__ void stage_rows(unsigned char* tile, const int8_t* src, int seq, int rows, int ld,
                                           int tid) {
    for (int u0 = 0; u0 < 4 * rows; u0 += 4 * kAttnThreads) {
        int4 v[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int u = u0 + k * kAttnThreads + tid, j = u >> 2, ch = u & 3;
            v[k] = j < seq ? ld_nc16(src + static_cast<long long>(j) * ld + 16 * ch) : make_int4(0, 0, 0, 0);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int u = u0 + k * kAttnThreads + tid, j = u >> 2, ch = u & 3;
            uint32_t o[8];
            widen16(v[k], o);
            unsigned char* row = tile + static_cast<uint32_t>(j) * 128u;
            *reinterpret_cast<uint4*>(row + ((static_cast<uint32_t>(2 * ch) ^ (j & 7)) << 4)) =
                make_uint4(o[0], o[1], o[2], o[3]);
            *reinterpret_cast<uint4*>(row + ((static_cast<uint32_t>(2 * ch + 1) ^ (j & 7)) << 4)) =
                make_uint4(o[4], o[5], o[6], o[7]);
        }
    }
}

__device__ __forceinline__ uint32_t pack2_s8(float v0, float v1, float inv) {
    const int q0 = __float2int_rn(__fmul_rn(v0, inv)), q1 = __float2int_rn(__fmul_rn(v1, inv));
    uint32_t d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(0));
    return d;  // q0 in byte 0, q1 in byte 1
}

// The f16 pair (a, b) -> u32 (a in the low half), and back.
__device__ __forceinline__ uint32_t f16x2_bits(float a, float b) {
    const __half2 h = __floats2half2_rn(a, b);
    uint32_t r;
    memcpy(&r, &h, sizeof(r));
    return r;
}
__device__ __forceinline__ float2 f16x2_float2(uint32_t u) {
    __half2 h;
    memcpy(&h, &u, sizeof(h));
    return __half22float2(h);
}

// c2 = c log2(e).  skip_mma (a test hook) issues no MMA, so that every wait
// gives up after wait_limit polls with nothing in flight.
__global__ void __launch_bounds__(kAttnThreads, 2)
attention_kernel(const int8_t* __restrict__ qkv, int seq, int d, int ld, float c2, float vscale, int kind,
                 float inv_out_scale, void* __restrict__ out, unsigned wait_limit, int skip_mma) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* sm =
        reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int nkb = (seq + kKeyBlock - 1) / kKeyBlock;
    unsigned char* Ks = sm;                                  // [nkb * 128][64] f16, swizzled
    unsigned char* Vs = sm + nkb * kBlockBytes;              // [nkb * 128][64] f16, swizzled
    unsigned char* misc = sm + 2 * nkb * kBlockBytes;
    const uint32_t bar_s = smem_addr(misc);                  // S_b complete
    const uint32_t bar_o = bar_s + 8;                        // P_b V_b complete
    const int tid = threadIdx.x, warp = tid >> 5;
    const int q0 = blockIdx.x * kAttnQ;
    const int h = blockIdx.y;
    const long long row0 = static_cast<long long>(blockIdx.z) * seq;  // first token row of the sequence
    const int8_t* head = qkv + row0 * ld + h * 64;

    if (tid == 0) mbar_init_n(bar_s, 2);
    __syncwarp();
    if (warp == 0) tmem_alloc(bar_s + 16, kTmemCols);
    stage_rows(Ks, head + d, seq, nkb * kKeyBlock, ld, tid);
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = *reinterpret_cast<volatile uint32_t*>(misc + 16);
    const uint32_t lane = tm + (static_cast<uint32_t>(32 * warp) << 16);  // this warp's quarter of the lanes

    // The thread's query as f16 pairs into its lane.
    {
        const int q = q0 + tid;
        uint32_t v[32];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int4 x = q < seq ? ld_nc16(head + static_cast<long long>(q) * ld + 16 * k) : make_int4(0, 0, 0, 0);
            uint32_t o[8];
            widen16(x, o);
#pragma unroll
            for (int i = 0; i < 8; ++i) v[8 * k + i] = o[i];
        }
        tmem_st32(lane + kColQ, v);
        tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    const uint32_t ks = smem_addr(Ks), vs = smem_addr(Vs);
    auto issue_s = [&](int b) {
#pragma unroll
        for (int t = 0; t < 4; ++t)
            mma_f16_ts(tm + kColS, tm + kColQ + 8 * t, sw128_desc(ks + b * kBlockBytes + 32 * t, 16, 1024), kIdescS,
                       t > 0);
        tc_commit(bar_s);
    };
    if (tid == 0 && !skip_mma) issue_s(0);
    // The values land while the first scores are computed; they are visible
    // to the MMAs after the block's barrier below.
    stage_rows(Vs, head + 2 * d, seq, nkb * kKeyBlock, ld, tid);
    fence_proxy_async();

    float m = -INFINITY;  // running maximum of the exact dot products
    float l = 0.0f;       // running sum of the weights
    bool ok = true;
    for (int b = 0; b < nkb; ++b) {
        ok &= mbar_wait(bar_s, b & 1, wait_limit);
        __syncwarp();
        tc_fence_after();
        float s[kKeyBlock];
        {
            uint32_t r[4][32];
#pragma unroll
            for (int k = 0; k < 4; ++k) tmem_ld32(lane + kColS + 32 * k, r[k]);
#pragma unroll
            for (int k = 0; k < 4; ++k) tmem_wait_ld(r[k]);
#pragma unroll
            for (int k = 0; k < 4; ++k)
#pragma unroll
                for (int i = 0; i < 32; ++i) s[32 * k + i] = __uint_as_float(r[k][i]);
        }
        const int valid = seq - b * kKeyBlock;  // keys of the block inside the sequence, >= 1
        if (valid < kKeyBlock) {
#pragma unroll
            for (int j = 0; j < kKeyBlock; ++j)
                if (j >= valid) s[j] = -INFINITY;
        }
        float bm = s[0];
#pragma unroll
        for (int j = 1; j < kKeyBlock; ++j) bm = fmaxf(bm, s[j]);
        const float mn = fmaxf(m, bm);  // finite: the block has a key
        // A larger maximum scales the context and the sum by the same
        // factor (1 for the lanes whose maximum did not move); tensor-memory
        // loads and stores are warp-wide, so the whole warp takes the branch.
        if (b > 0 && __any_sync(0xffffffffu, mn > m)) {
            const float alpha = exp2f(__fmul_rn(__fsub_rn(m, mn), c2));
            l = __fmul_rn(l, alpha);
            uint32_t o[2][32];
            tmem_ld32(lane + kColO, o[0]);
            tmem_ld32(lane + kColO + 32, o[1]);
            tmem_wait_ld(o[0]);
            tmem_wait_ld(o[1]);
#pragma unroll
            for (int k = 0; k < 2; ++k)
#pragma unroll
                for (int i = 0; i < 32; ++i) o[k][i] = __float_as_uint(__fmul_rn(__uint_as_float(o[k][i]), alpha));
            tmem_st32(lane + kColO, o[0]);
            tmem_st32(lane + kColO + 32, o[1]);
        }
        m = mn;
        // Weights of keys 32 cc .. 32 cc + 31: high f16 parts into columns
        // 32 cc .. + 15, low parts into 32 cc + 16 .. + 31 (over the scores).
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            uint32_t p[32];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const float e0 = exp2f(__fmul_rn(__fsub_rn(s[32 * cc + 2 * e], m), c2));
                const float e1 = exp2f(__fmul_rn(__fsub_rn(s[32 * cc + 2 * e + 1], m), c2));
                l = __fadd_rn(__fadd_rn(l, e0), e1);
                const uint32_t hi = f16x2_bits(e0, e1);
                const float2 hf = f16x2_float2(hi);
                p[e] = hi;
                p[16 + e] = f16x2_bits(__fsub_rn(e0, hf.x), __fsub_rn(e1, hf.y));
            }
            tmem_st32(lane + kColS + 32 * cc, p);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !skip_mma) {
            tc_fence_after();
#pragma unroll
            for (int t = 0; t < 8; ++t) {  // keys 16 t .. 16 t + 15 of the block
                const uint64_t bd = sw128_desc(vs + b * kBlockBytes + 2048 * t, 1024, 1024);
                const uint32_t a = tm + kColS + 32 * (t >> 1) + 8 * (t & 1);
                mma_f16_ts(tm + kColO, a, bd, kIdescPV, (b > 0 || t > 0) ? 1u : 0u);
                mma_f16_ts(tm + kColO, a + 16, bd, kIdescPV, 1u);
            }
            tc_commit(bar_o);
            if (b + 1 < nkb) {  // the next scores overwrite P_b: wait until it is consumed
                ok &= mbar_wait(bar_o, b & 1, wait_limit);
                tc_fence_after();
                issue_s(b + 1);
            }
        }
    }

    // Context row: O / l * qkv_scale.
    ok &= mbar_wait(bar_o, (nkb - 1) & 1, wait_limit);
    __syncwarp();
    tc_fence_after();
    uint32_t o[2][32];
    tmem_ld32(lane + kColO, o[0]);
    tmem_ld32(lane + kColO + 32, o[1]);
    tmem_wait_ld(o[0]);
    tmem_wait_ld(o[1]);
    const int r = q0 + tid;
    if (r < seq) {
        const float f = __fdiv_rn(vscale, l);
        const long long base = (row0 + r) * d + h * 64;
        if (kind == 3) {
            uint4* dst = reinterpret_cast<uint4*>(static_cast<int8_t*>(out) + base);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                uint32_t w[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int j = 16 * k + 4 * i;
                    const float y0 = __fmul_rn(__uint_as_float(o[j >> 5][j & 31]), f);
                    const float y1 = __fmul_rn(__uint_as_float(o[(j + 1) >> 5][(j + 1) & 31]), f);
                    const float y2 = __fmul_rn(__uint_as_float(o[(j + 2) >> 5][(j + 2) & 31]), f);
                    const float y3 = __fmul_rn(__uint_as_float(o[(j + 3) >> 5][(j + 3) & 31]), f);
                    w[i] = pack2_s8(y0, y1, inv_out_scale) | (pack2_s8(y2, y3, inv_out_scale) << 16);
                }
                dst[k] = make_uint4(w[0], w[1], w[2], w[3]);
            }
        } else {
            float4* dst = reinterpret_cast<float4*>(static_cast<float*>(out) + base);
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int j = 4 * k;
                dst[k] = make_float4(__fmul_rn(__uint_as_float(o[j >> 5][j & 31]), f),
                                     __fmul_rn(__uint_as_float(o[(j + 1) >> 5][(j + 1) & 31]), f),
                                     __fmul_rn(__uint_as_float(o[(j + 2) >> 5][(j + 2) & 31]), f),
                                     __fmul_rn(__uint_as_float(o[(j + 3) >> 5][(j + 3) & 31]), f));
            }
        }
    }
    if (!ok) atomicOr(&g_attn_status, static_cast<unsigned>(kStatusTimeout));
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, kTmemCols);
}

}  // namespace

size_t attention_smem_bytes(int seq) {
    const size_t nkb = (static_cast<size_t>(seq) + kKeyBlock - 1) / kKeyBlock;
    return 2 * nkb * kBlockBytes + 1024 + 64;  // K and V tiles, 1024-byte alignment, barriers + TMEM address
}

cudaError_t launch_attention(const int8_t* qkv, int batch, int seq, int heads, int ld, float score_scale,
                             float qkv_scale, int kind, float inv_out_scale, void* out, cudaStream_t s) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static bool ready[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!ready[dev]) {
            e = cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     static_cast<int>(attention_smem_bytes(BSGEMM_ATTN_MAX_SEQ)));
            if (e != cudaSuccess) return e;
            ready[dev] = true;
        }
    }
    const float c2 = static_cast<float>(static_cast<double>(score_scale) * 1.4426950408889634);  // c log2(e)
    const bool skip = (test_hooks() & BSGEMM_TEST_ATTN_SKIP_MMA) != 0;
    const dim3 grid(static_cast<unsigned>((seq + kAttnQ - 1) / kAttnQ), static_cast<unsigned>(heads),
                    static_cast<unsigned>(batch));
    attention_kernel<<<grid, kAttnThreads, attention_smem_bytes(seq), s>>>(
        qkv, seq, heads * 64, ld, c2, qkv_scale, kind, inv_out_scale, out, skip ? 64u : kWaitLimit, skip ? 1 : 0);
    return cudaGetLastError();
}

cudaError_t attention_status(bool clear, unsigned* v) {
    cudaError_t e = cudaMemcpyFromSymbol(v, g_attn_status, sizeof(unsigned));
    if (e == cudaSuccess && clear && *v != 0) {
        const unsigned zero = 0;
        e = cudaMemcpyToSymbol(g_attn_status, &zero, sizeof(unsigned));
    }
    return e;
}

}  // namespace bsg
