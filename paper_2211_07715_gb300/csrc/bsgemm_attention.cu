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
// Both contractions run on the tensor cores (mma.sync m16n8k16, bf16
// operands, fp32 accumulation):
//   * q k^T is exact: int8 values are exact in bf16, the products (< 2^14)
//     are exact, and every partial sum of 64 of them stays below 2^24, so
//     the fp32 accumulator holds the int32 dot product;
//   * P v takes P in two bf16 parts (p = hi + lo + r, |r| <= 2^-16 p) against
//     the exact bf16 v, two MMAs per tile.
// The softmax is taken online over blocks of 64 keys (running row maximum m
// and sum l; when m grows, the context accumulator and l are scaled by the
// same factor exp(m_old - m_new)), in fp32.
//
// One CTA = 64 queries of one (sequence, head), 4 warps of 16 queries.  The
// head's keys and values for the whole sequence (seq <= BSGEMM_ATTN_MAX_SEQ,
// padded to whole 64-key blocks with zeros) and the CTA's queries are
// staged once into shared memory as bf16 rows of 64 (128 bytes, 16-byte
// chunks XOR-swizzled by the row so that 8 consecutive rows of one chunk
// lie in different banks); `ldmatrix` reads the MMA fragments: plain for
// the queries and keys, transposed for the values.  The scores and
// probabilities of a 16 x 64 block live in registers (the MMA output
// layout of a score tile is the input layout of the P v MMA).
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda_bf16.h>

#include "bsgemm.h"
#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kAttnThreads = 128;  // 4 warps x 16 queries
constexpr int kAttnQ = 64;         // queries per CTA
constexpr int kKeyBlock = 64;      // keys per online-softmax block

__device__ __forceinline__ int4 ld_nc16(const int8_t* p) {
    return __ldg(reinterpret_cast<const int4*>(p));
}

// Byte offset of 16-byte chunk c (bf16 elements 8c .. 8c+7) of row r in a
// swizzled tile of 64-element bf16 rows.
__device__ __forceinline__ uint32_t tile_off(int r, int c) {
    return (static_cast<uint32_t>(r) << 7) | (static_cast<uint32_t>(c ^ (r & 7)) << 4);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint32_t bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    uint32_t u;
    memcpy(&u, &v, sizeof(u));
    return u;
}

// The bf16 pair of bf16x2(lo, hi) back in fp32.
__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// Byte k of w (w holds int8 values XOR 0x80, i.e. v + 128 as unsigned
// bytes) as the float v: 0x4B0000uu is 2^23 + uu exactly.
template <int k>
__device__ __forceinline__ float widen_s8(uint32_t w) {
    return __fsub_rn(__int_as_float(static_cast<int>(__byte_perm(w, 0x4B000000u, 0x7440u + k))), 8388736.0f);
}

// 16 int8 values (elements 16 ch .. 16 ch + 15 of row r) -> bf16 chunks
// 2 ch and 2 ch + 1 of that row.
__device__ __forceinline__ void store_row16(unsigned char* tile, int r, int ch, int4 v) {
    const uint32_t w[4] = {static_cast<uint32_t>(v.x) ^ 0x80808080u, static_cast<uint32_t>(v.y) ^ 0x80808080u,
                           static_cast<uint32_t>(v.z) ^ 0x80808080u, static_cast<uint32_t>(v.w) ^ 0x80808080u};
    uint32_t o[8];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        o[2 * q] = bf16x2(widen_s8<0>(w[q]), widen_s8<1>(w[q]));
        o[2 * q + 1] = bf16x2(widen_s8<2>(w[q]), widen_s8<3>(w[q]));
    }
    *reinterpret_cast<int4*>(tile + tile_off(r, 2 * ch)) = make_int4(o[0], o[1], o[2], o[3]);
    *reinterpret_cast<int4*>(tile + tile_off(r, 2 * ch + 1)) = make_int4(o[4], o[5], o[6], o[7]);
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// d += A B for one m16n8k16 tile: A 16 x 16 (4 registers of bf16 pairs), B
// 16 x 8 (2 registers), d 16 x 8 fp32 (rows g and g + 8, columns 2 t4 and
// 2 t4 + 1 of lane 4 g + t4).
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
                 "{%8, %9}, {%0, %1, %2, %3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack2_s8(float v0, float v1, float inv) {
    const int q0 = __float2int_rn(__fmul_rn(v0, inv)), q1 = __float2int_rn(__fmul_rn(v1, inv));
    uint32_t d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(0));
    return d;  // q0 in byte 0, q1 in byte 1
}

__global__ void __launch_bounds__(kAttnThreads, 2)
attention_kernel(const int8_t* __restrict__ qkv, int seq, int d, int ld, float c, float vscale, int kind,
                 float inv_out_scale, void* __restrict__ out) {
    extern __shared__ __align__(128) unsigned char smem[];
    const int nkb = (seq + kKeyBlock - 1) / kKeyBlock;
    const int seq_pad = nkb * kKeyBlock;
    unsigned char* Ks = smem;                    // [seq_pad][64] bf16
    unsigned char* Vs = smem + 128 * seq_pad;    // [seq_pad][64] bf16
    unsigned char* Qs = smem + 256 * seq_pad;    // [64][64] bf16

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q0 = blockIdx.x * kAttnQ;
    const int h = blockIdx.y;
    const long long row0 = static_cast<long long>(blockIdx.z) * seq;  // first token row of the sequence
    const int8_t* head = qkv + row0 * ld + h * 64;

    // 1. Queries, keys and values of the head -> bf16 tiles (rows past the
    //    sequence are zeros).
    const int4 zero = make_int4(0, 0, 0, 0);
    for (int u = tid; u < 4 * kAttnQ; u += kAttnThreads) {
        const int i = u >> 2, ch = u & 3;
        const int4 v = q0 + i < seq ? ld_nc16(head + static_cast<long long>(q0 + i) * ld + 16 * ch) : zero;
        store_row16(Qs, i, ch, v);
    }
    for (int u = tid; u < 4 * seq_pad; u += kAttnThreads) {
        const int j = u >> 2, ch = u & 3;
        int4 kv = zero, vv = zero;
        if (j < seq) {
            const int8_t* row = head + static_cast<long long>(j) * ld + 16 * ch;
            kv = ld_nc16(row + d);
            vv = ld_nc16(row + 2 * d);
        }
        store_row16(Ks, j, ch, kv);
        store_row16(Vs, j, ch, vv);
    }
    __syncthreads();

    // 2. The warp's 16 queries as A fragments (4 chunks of 16 channels).
    uint32_t qa[4][4];
    {
        const int r = 16 * warp + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
        for (int kc = 0; kc < 4; ++kc)
            ldsm_x4(smem_u32(Qs + tile_off(r, 2 * kc + (lane >> 4))), qa[kc][0], qa[kc][1], qa[kc][2], qa[kc][3]);
    }
    const int t4 = lane & 3;
    float o[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.0f;
    float m0 = -INFINITY, m1 = -INFINITY;  // running maxima of rows g and g + 8
    float l0 = 0.0f, l1 = 0.0f;            // this lane's part of the running sums

    for (int kb = 0; kb < nkb; ++kb) {
        const int key0 = kb * kKeyBlock;
        // scores of keys key0 + 8 nt .. + 7
        float s[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.0f;
#pragma unroll
            for (int kcp = 0; kcp < 2; ++kcp) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(smem_u32(Ks + tile_off(key0 + 8 * nt + (lane & 7), 4 * kcp + (lane >> 3))), b0, b1, b2, b3);
                mma_bf16(s[nt], qa[2 * kcp], b0, b1);
                mma_bf16(s[nt], qa[2 * kcp + 1], b2, b3);
            }
        }
        float bm0 = -INFINITY, bm1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = key0 + 8 * nt + 2 * t4 + (e & 1);
                s[nt][e] = key < seq ? __fmul_rn(s[nt][e], c) : -INFINITY;
            }
            bm0 = fmaxf(bm0, fmaxf(s[nt][0], s[nt][1]));
            bm1 = fmaxf(bm1, fmaxf(s[nt][2], s[nt][3]));
        }
        bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
        bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
        bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
        bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
        const float mn0 = fmaxf(m0, bm0), mn1 = fmaxf(m1, bm1);  // finite: key0 < seq
        const float a0 = expf(__fsub_rn(m0, mn0)), a1 = expf(__fsub_rn(m1, mn1));  // 0 in the first block
        m0 = mn0;
        m1 = mn1;
        l0 = __fmul_rn(l0, a0);
        l1 = __fmul_rn(l1, a1);
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            o[n][0] = __fmul_rn(o[n][0], a0), o[n][1] = __fmul_rn(o[n][1], a0);
            o[n][2] = __fmul_rn(o[n][2], a1), o[n][3] = __fmul_rn(o[n][3], a1);
        }
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            s[nt][0] = expf(__fsub_rn(s[nt][0], mn0)), s[nt][1] = expf(__fsub_rn(s[nt][1], mn0));
            s[nt][2] = expf(__fsub_rn(s[nt][2], mn1)), s[nt][3] = expf(__fsub_rn(s[nt][3], mn1));
            l0 = __fadd_rn(l0, __fadd_rn(s[nt][0], s[nt][1]));
            l1 = __fadd_rn(l1, __fadd_rn(s[nt][2], s[nt][3]));
        }
        // context += P v, 32 keys (two k-chunks of 16) per transposed ldmatrix
#pragma unroll
        for (int kkp = 0; kkp < 2; ++kkp) {
            uint32_t hi[2][4], lo[2][4];
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const int nt = 2 * (2 * kkp + x);
                const float* p[4] = {&s[nt][0], &s[nt][2], &s[nt + 1][0], &s[nt + 1][2]};
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    hi[x][r] = bf16x2(p[r][0], p[r][1]);
                    lo[x][r] = bf16x2(__fsub_rn(p[r][0], bf16_lo(hi[x][r])), __fsub_rn(p[r][1], bf16_hi(hi[x][r])));
                }
            }
#pragma unroll
            for (int n = 0; n < 8; ++n) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(smem_u32(Vs + tile_off(key0 + 32 * kkp + 8 * (lane >> 3) + (lane & 7), n)), b0, b1, b2, b3);
                mma_bf16(o[n], hi[0], b0, b1);
                mma_bf16(o[n], lo[0], b0, b1);
                mma_bf16(o[n], hi[1], b2, b3);
                mma_bf16(o[n], lo[1], b2, b3);
            }
        }
    }

    // 3. Row sums over the quad, scale, store rows g and g + 8.
    l0 = __fadd_rn(l0, __shfl_xor_sync(0xffffffffu, l0, 1));
    l0 = __fadd_rn(l0, __shfl_xor_sync(0xffffffffu, l0, 2));
    l1 = __fadd_rn(l1, __shfl_xor_sync(0xffffffffu, l1, 1));
    l1 = __fadd_rn(l1, __shfl_xor_sync(0xffffffffu, l1, 2));
    const float f0 = __fdiv_rn(vscale, l0), f1 = __fdiv_rn(vscale, l1);
    const int ra = q0 + 16 * warp + (lane >> 2);
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const int r = ra + 8 * half;
        if (r >= seq) continue;
        const float f = half ? f1 : f0;
        const long long base = (row0 + r) * d + h * 64 + 2 * t4;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            const float y0 = __fmul_rn(o[n][2 * half], f), y1 = __fmul_rn(o[n][2 * half + 1], f);
            if (kind == 3) {
                *reinterpret_cast<uint16_t*>(static_cast<int8_t*>(out) + base + 8 * n) =
                    static_cast<uint16_t>(pack2_s8(y0, y1, inv_out_scale));
            } else {
                *reinterpret_cast<float2*>(static_cast<float*>(out) + base + 8 * n) = make_float2(y0, y1);
            }
        }
    }
}

}  // namespace

size_t attention_smem_bytes(int seq) {
    const size_t seq_pad = (static_cast<size_t>(seq) + kKeyBlock - 1) / kKeyBlock * kKeyBlock;
    return 256 * seq_pad + 128 * kAttnQ;  // keys and values, queries: bf16 rows of 64
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
    const dim3 grid(static_cast<unsigned>((seq + kAttnQ - 1) / kAttnQ), static_cast<unsigned>(heads),
                    static_cast<unsigned>(batch));
    attention_kernel<<<grid, kAttnThreads, attention_smem_bytes(seq), s>>>(qkv, seq, heads * 64, ld, score_scale,
                                                                         qkv_scale, kind, inv_out_scale, out);
    return cudaGetLastError();
}

}  // namespace bsg
