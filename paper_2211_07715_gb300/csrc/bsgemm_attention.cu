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
// The softmax runs online over blocks of 64 keys in fp32.  A thread's
// weights are e_j = 2^fl(d_j c2 - M) (one fused multiply-add; c2 = c
// log2(e), d_j the exact dot product) against a reference M = fl(m c2) of a
// maximum m of the dot products seen so far.  M moves only when a block's
// maximum exceeds it by more than 8 (log2 units), so the weights stay below
// 2^8 and rescaling is rare; when it moves, the context and the running sum
// are scaled by the same 2^(M_old - M_new), the difference taken exactly.
// The rounding of M thus scales every weight by one factor that the context
// and the sum share, and the exponent carries only the roundings of c2 and
// of the fused product.
//
// One CTA = 128 queries of one (sequence, head): 8 compute warps and one
// MMA warp.  Compute warps w and w + 4 share the 32 queries of tensor-memory
// lane quarter w (thread i % 128 owns query i = lane i): each takes 32 of a
// block's 64 keys and 32 of the context's 64 columns, and the two exchange
// their block maxima through shared memory and keep their running sums of
// the weights in registers.  Tensor memory (256 columns, so two CTAs share
// an SM): two score buffers in columns 0-63 and 64-127 (block b uses
// buffer b % 2: its scores, then its weights written back in place as f16
// pairs -- for keys 32c .. 32c + 31 of the block the high parts in columns
// 32c .. + 15 of the buffer, the low parts in 32c + 16 .. + 31), the context
// O in 128-191, the CTA's queries (f16 pairs) in 192-223.  The head's keys
// and values (seq <= BSGEMM_ATTN_MAX_SEQ, padded with zeros to whole blocks)
// are copied into shared memory as int8 (cp.async, no registers) and widened
// there into f16 rows of 64 with the 128-byte swizzle: K is the K-major B
// operand of q k^T, V the MN-major B operand of P v.
//
// One thread of the MMA warp issues S_0 and S_1 (S_b = Q K_b^T: N = 64, K =
// 64), then per block b: waits until the compute threads have written P_b,
// issues O += P_b,hi V_b + P_b,lo V_b (8 MMAs) and right behind them
// S_(b+2) into the same buffer: the MMAs one thread issues run in issue
// order, so S_(b+2) writes the buffer only after P_b V_b has read it.  The
// compute warps thus work on block b + 1 while the tensor cores consume
// block b, and wait for the tensor cores only where the running maximum
// grows (a rescale of O needs the previous block's P v complete).
// mbarriers, two of each kind (one per buffer, so that no wait can fall two
// phases behind): S_b complete, P_b written (256 arrivals), P_b V_b
// complete; and one for the queries written to tensor memory (128
// arrivals).  Every wait is bounded.

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

constexpr int kCompute = 256;         // 8 compute warps, two per query (TMEM lane)
constexpr int kAttnThreads = kCompute + 32;  // + the MMA warp
constexpr int kAttnQ = 128;           // queries per CTA
constexpr int kKeyBlock = 64;         // keys per online-softmax block
constexpr uint32_t kBlockBytes = 8192;   // 64 rows x 64 f16
constexpr int kMaxRows = (BSGEMM_ATTN_MAX_SEQ + kKeyBlock - 1) / kKeyBlock * kKeyBlock;
constexpr int kMaxHalfUnits = (2 * kMaxRows + kCompute - 1) / kCompute;  // 16-byte units of V's second half a thread
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0, kColO = 128, kColQ = 192;  // score buffers at kColS and kColS + 64
constexpr uint32_t kIdescS = f16_idesc(128, 64, false);  // S = Q K_b^T
constexpr uint32_t kIdescPV = f16_idesc(128, 64, true);  // O += P V_b
constexpr float kLazy = 8.0f;  // largest weight 2^kLazy: the reference maximum moves past that

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

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(bar) : "memory");
}

// 16 bytes global -> shared without registers (zeros when src_bytes is 0).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
// Wait until at most N of this thread's committed groups are in flight.
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }
// Barrier of the 8 compute warps (the MMA warp does not take part).
__device__ __forceinline__ void compute_sync() { asm volatile("bar.sync 5, 256;\n" ::: "memory"); }

// Rows [j0, j1) of int8 rows (64 bytes each, row-major from `src`) widened
// into the swizzled f16 tile `tile` (row j, 16-byte chunk c at j * 128 + (c
// ^ (j % 8)) * 16); thread t takes 16-byte units t, t + 256, ... (at most
// NU of them: all loads first, then the widening and stores).
__device__ __forceinline__ void store_unit(unsigned char* tile, int u, int4 v) {
    const int j = u >> 2, ch = u & 3;
    uint32_t o[8];
    widen16(v, o);
    unsigned char* row = tile + static_cast<uint32_t>(j) * 128u;
    *reinterpret_cast<uint4*>(row + ((static_cast<uint32_t>(2 * ch) ^ (j & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
    *reinterpret_cast<uint4*>(row + ((static_cast<uint32_t>(2 * ch + 1) ^ (j & 7)) << 4)) =
        make_uint4(o[4], o[5], o[6], o[7]);
}
template <int NU>
__device__ __forceinline__ void widen_rows(unsigned char* tile, const unsigned char* src, int j0, int j1, int tid) {
    int4 v[NU];
#pragma unroll
    for (int i = 0; i < NU; ++i) {
        const int u = 4 * j0 + tid + i * kCompute;
        v[i] = u < 4 * j1 ? *reinterpret_cast<const int4*>(src + 16 * u) : make_int4(0, 0, 0, 0);
    }
#pragma unroll
    for (int i = 0; i < NU; ++i) {
        const int u = 4 * j0 + tid + i * kCompute;
        if (u < 4 * j1) store_unit(tile, u, v[i]);
    }
}

__device__ __forceinline__ uint32_t pack2_s8(float v0, float v1, float inv) {
    const int q0 = __float2int_rn(__fmul_rn(v0, inv)), q1 = __float2int_rn(__fmul_rn(v1, inv));
    uint32_t d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(0));
    return d;  // q0 in byte 0, q1 in byte 1
}

// 2^t for t <= 0 on the special-function unit: ex2.approx.ftz.f32, within 2
// ulp of the exact value wherever the result is a normal fp32 number
// (checked on GB300 over every fp32 t in [-126, 0]); below that the result
// flushes to 0, an absolute error under 2^-126.
__device__ __forceinline__ float ex2(float t) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(t));
    return y;
}

// Two fp32 lanes at once (sm_100+ packed instructions, each lane rounded
// as the scalar instruction rounds): a * b + c, a + b, a - b; and the
// largest of three values.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 r;
    asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mov.b64 rc, {%6, %7};\n"
        " fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}\n"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 r;
    asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
        " add.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}\n"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
    float2 r;
    asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
        " sub.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}\n"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
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

// 64-thread barrier (id 1 + qq) of the two compute warps of lane quarter qq.
__device__ __forceinline__ void pair_sync(int qq) {
    switch (qq) {
        case 0: asm volatile("bar.sync 1, 64;\n" ::: "memory"); break;
        case 1: asm volatile("bar.sync 2, 64;\n" ::: "memory"); break;
        case 2: asm volatile("bar.sync 3, 64;\n" ::: "memory"); break;
        default: asm volatile("bar.sync 4, 64;\n" ::: "memory"); break;
    }
}

// c2 = c log2(e).  skip_mma (a test hook) issues no MMA, so that every wait
// on one gives up after wait_limit polls with nothing in flight.
__global__ void __launch_bounds__(kAttnThreads, 2)
attention_kernel(const int8_t* __restrict__ qkv, int seq, int d, int ld, float c2, float vscale, int kind,
                 float inv_out_scale, void* __restrict__ out, unsigned wait_limit, int skip_mma, int act_ready) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* sm =
        reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int nkb = (seq + kKeyBlock - 1) / kKeyBlock;
    const int rows = nkb * kKeyBlock;
    unsigned char* Ks = sm;                                  // [rows][64] f16, swizzled
    unsigned char* Vs = sm + nkb * kBlockBytes;              // [rows][64] f16, swizzled
    unsigned char* misc = sm + 2 * nkb * kBlockBytes;
    float* red = reinterpret_cast<float*>(misc + 64);        // [2 blocks][2 halves][128 queries]
    const uint32_t bar_s = smem_addr(misc);  // [2] S_b complete (buffer b % 2)
    const uint32_t bar_p = bar_s + 16;       // [2] P_b written: one arrival per compute thread
    const uint32_t bar_o = bar_s + 32;       // [2] P_b V_b complete
    const uint32_t bar_q = bar_s + 48;       // queries in tensor memory: one arrival per thread of warps 0-3
    const int tid = threadIdx.x, warp = tid >> 5;
    const int q0 = blockIdx.x * kAttnQ;
    const int h = blockIdx.y;
    const long long row0 = static_cast<long long>(blockIdx.z) * seq;  // first token row of the sequence
    const int8_t* head = qkv + row0 * ld + h * 64;
    const bool mma_warp = warp == kCompute / 32;
    const int qq = warp & 3, hh = (warp >> 2) & 1;  // lane quarter; half of the keys and of the context
    const int qi = tid & (kAttnQ - 1);               // the thread's query within the CTA (= its lane)

    // The kernel is launched with programmatic dependent launch: it lets the
    // next kernel launch at once, and reads qkv only after the preceding
    // kernel has completed -- unless act_ready says qkv was complete before
    // that kernel began; global writes always come after it.
    griddep_launch_dependents();

    // 1. Barriers and tensor memory (MMA warp); the head's keys and values
    //    copied as int8 into the value tile's space (keys in its first half,
    //    values in its second) and the query loaded (warps 0-3), all issued
    //    at once; the keys widened into their f16 tile (compute warps).
    if (mma_warp) {
        if (tid == kCompute) {
            mbar_init_n(bar_s, 2);
            mbar_init(bar_p, kCompute);
            mbar_init(bar_p + 8, kCompute);
            mbar_init_n(bar_o, 2);
            mbar_init(bar_q, kAttnQ);
        }
        __syncwarp();
        tmem_alloc(bar_s + 56, kTmemCols);
    }
    int4 qv[4];
    if (!mma_warp) {
        if (!act_ready) griddep_wait();
        const int q = q0 + qi;
#pragma unroll
        for (int k = 0; k < 4; ++k)
            qv[k] = (hh == 0 && q < seq) ? ld_nc16(head + static_cast<long long>(q) * ld + 16 * k)
                                         : make_int4(0, 0, 0, 0);
        // unit u of part p (0 = keys, 1 = values): row u / 4, 16-byte chunk u % 4,
        // to Vs + p * rows * 64 + 16 u (zeros past the sequence); one
        // commit group per part, so the keys widen while the values land
        const uint32_t vs8 = smem_addr(Vs);
#pragma unroll
        for (int p = 0; p < 2; ++p) {
            for (int u = tid; u < 4 * rows; u += kCompute) {
                const int j = u >> 2;
                const int8_t* src = head + (p + 1) * d + static_cast<long long>(j < seq ? j : 0) * ld + 16 * (u & 3);
                cp_async16(vs8 + static_cast<uint32_t>(p * rows * 64 + 16 * u), src, j < seq ? 16u : 0u);
            }
            cp_async_commit();
        }
        cp_async_wait<1>();
        compute_sync();  // every thread's copies of the keys have landed
        widen_rows<4 * kMaxRows / kCompute>(Ks, Vs, 0, rows, tid);
        fence_proxy_async();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = *reinterpret_cast<volatile uint32_t*>(misc + 56);
    const uint32_t lane = tm + (static_cast<uint32_t>(32 * qq) << 16);  // this warp's lane quarter

    // 2. The query as f16 pairs into its lane (warps 0-3).
    if (!mma_warp) {
        if (hh == 0) {
            uint32_t v[32];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                uint32_t o[8];
                widen16(qv[k], o);
#pragma unroll
                for (int i2 = 0; i2 < 8; ++i2) v[8 * k + i2] = o[i2];
            }
            tmem_st32(lane + kColQ, v);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(bar_q);
        }
    }

    bool ok = true;
    if (mma_warp) {
        // 3a. MMA issue (one thread).
        if (tid == kCompute) {
            const uint32_t ks = smem_addr(Ks), vs = smem_addr(Vs);
            auto issue_s = [&](int b) {
                const uint32_t buf = tm + kColS + 64u * static_cast<uint32_t>(b & 1);
#pragma unroll
                for (int t = 0; t < 4; ++t)
                    mma_f16_ts(buf, tm + kColQ + 8 * t, sw128_desc(ks + b * kBlockBytes + 32 * t, 16, 1024), kIdescS,
                               t > 0);
                tc_commit(bar_s + 8u * static_cast<uint32_t>(b & 1));
            };
            ok &= mbar_wait(bar_q, 0, wait_limit);
            tc_fence_after();
            if (!skip_mma) {
                issue_s(0);
                if (nkb > 1) issue_s(1);
            }
            for (int b = 0; b < nkb; ++b) {
                const uint32_t x = static_cast<uint32_t>(b & 1), ph = static_cast<uint32_t>(b >> 1) & 1u;
                ok &= mbar_wait(bar_p + 8u * x, ph, wait_limit);
                tc_fence_after();
                if (!skip_mma) {
#pragma unroll
                    for (int t = 0; t < 4; ++t) {  // keys 16 t .. 16 t + 15 of the block
                        const uint64_t bd = sw128_desc(vs + b * kBlockBytes + 2048 * t, 1024, 1024);
                        const uint32_t a = tm + kColS + 64u * x + 32 * (t >> 1) + 8 * (t & 1);
                        mma_f16_ts(tm + kColO, a, bd, kIdescPV, (b > 0 || t > 0) ? 1u : 0u);
                        mma_f16_ts(tm + kColO, a + 16, bd, kIdescPV, 1u);
                    }
                    tc_commit(bar_o + 8u * x);
                }
                // S_(b+2) overwrites P_b.  MMAs issued by one thread run in
                // issue order, so it follows P_b V_b without a wait here.
                if (b + 2 < nkb && !skip_mma) issue_s(b + 2);
            }
        }
        __syncwarp();
    } else {
        // 3b. Compute warps: the values widened in place, then the softmax
        //     block by block over the warp's 32 keys of each block.  The
        //     int8 values sit at Vs + rows * 64: rows below rows / 2 widen
        //     into the keys' int8 space (free now), the others over their
        //     own int8 bytes, so those are read into registers first.
        {
            cp_async_wait<0>();
            compute_sync();  // every thread's copies of the values have landed
            const unsigned char* v8 = Vs + rows * 64;
            const int half = rows / 2;
            int4 hv[kMaxHalfUnits];  // the second half's int8 bytes, loaded with the first half's
#pragma unroll
            for (int i = 0; i < kMaxHalfUnits; ++i) {
                const int u = 4 * half + i * kCompute + tid;
                hv[i] = u < 4 * rows ? *reinterpret_cast<const int4*>(v8 + 16 * u) : make_int4(0, 0, 0, 0);
            }
            widen_rows<kMaxHalfUnits>(Vs, v8, 0, half, tid);
            compute_sync();  // every read of the second half's int8 bytes is done
#pragma unroll
            for (int i = 0; i < kMaxHalfUnits; ++i) {
                const int u = 4 * half + i * kCompute + tid;
                if (u < 4 * rows) store_unit(Vs, u, hv[i]);
            }
        }
        fence_proxy_async();  // visible to the MMAs once P_0 is announced
        // The weights are 2^(s c2 - M) against a reference M = fl(m c2) of a
        // maximum m of the dot products seen so far, which moves only when
        // the block maximum exceeds it by more than kLazy (log2 units), so
        // the weights stay below 2^kLazy.  A rounding error of M scales all
        // the weights taken against it by one factor, which the context and
        // the sum share.
        float mref = 0.0f;                      // M
        float lq[4] = {0.0f, 0.0f, 0.0f, 0.0f};  // running sum of the warp's weights, in 4 parts
        for (int b = 0; b < nkb; ++b) {
            const uint32_t x = static_cast<uint32_t>(b & 1), ph = static_cast<uint32_t>(b >> 1) & 1u;
            const uint32_t buf = lane + kColS + 64u * x + 32u * static_cast<uint32_t>(hh);
            ok &= mbar_wait(bar_s + 8u * x, ph, wait_limit);
            __syncwarp();
            tc_fence_after();
            float s[32];
            {
                uint32_t r[32];
                tmem_ld32(buf, r);
                tmem_wait_ld(r);
#pragma unroll
                for (int i2 = 0; i2 < 32; ++i2) s[i2] = __uint_as_float(r[i2]);
            }
            const int valid = seq - b * kKeyBlock - 32 * hh;  // of the warp's 32 keys, inside the sequence
            if (valid < 32) {
#pragma unroll
                for (int j2 = 0; j2 < 32; ++j2)
                    if (j2 >= valid) s[j2] = -INFINITY;
            }
            float bq[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
            for (int j2 = 4; j2 < 32; j2 += 8)
#pragma unroll
                for (int k = 0; k < 4; ++k) bq[k] = max3(bq[k], s[j2 + k], s[j2 + 4 + k]);
            float* rb = red + 256 * (b & 1);
            rb[128 * hh + qi] = fmaxf(max3(bq[0], bq[1], bq[2]), bq[3]);
            pair_sync(qq);
            // The block's maximum, scaled (finite: the block has a key).
            const float bm = __fmul_rn(fmaxf(rb[qi], rb[128 + qi]), c2);
            if (b == 0) {
                mref = bm;
            } else {
                // A reference that moves scales the context and the sum by
                // alpha = 2^(M_old - M_new) once the previous block's P v is
                // complete (alpha = 1 for the lanes whose reference stays);
                // tensor-memory loads and stores are warp-wide, so the whole
                // warp takes the branch.
                const bool move = __fsub_rn(bm, mref) > kLazy;
                if (__any_sync(0xffffffffu, move)) {
                    const uint32_t xp = static_cast<uint32_t>((b - 1) & 1), php = static_cast<uint32_t>((b - 1) >> 1) & 1u;
                    ok &= mbar_wait(bar_o + 8u * xp, php, wait_limit);
                    __syncwarp();
                    tc_fence_after();
                    // M_old - M_new exactly, as d_hi + d_lo (Knuth's TwoSum)
                    const float dh = __fsub_rn(mref, bm);
                    const float bb = __fsub_rn(dh, mref);
                    const float dl = __fadd_rn(__fsub_rn(mref, __fsub_rn(dh, bb)), __fsub_rn(-bm, bb));
                    const float alpha = move ? __fmul_rn(exp2f(dh), exp2f(dl)) : 1.0f;
                    if (move) mref = bm;
#pragma unroll
                    for (int k = 0; k < 4; ++k) lq[k] = __fmul_rn(lq[k], alpha);
                    uint32_t o[32];
                    const uint32_t oc = lane + kColO + 32u * static_cast<uint32_t>(hh);
                    tmem_ld32(oc, o);
                    tmem_wait_ld(o);
#pragma unroll
                    for (int i2 = 0; i2 < 32; ++i2) o[i2] = __float_as_uint(__fmul_rn(__uint_as_float(o[i2]), alpha));
                    tmem_st32(oc, o);
                }
            }
            // The warp's 32 weights: high f16 parts into the first 16 of its
            // columns, low parts into the last 16 (over the scores).
            // (pairs of lanes: the packed fp32 instructions round each lane
            // as the scalar ones do, so the values are those of one lane at a
            // time; the sums go to lq[0], lq[1] for even e, lq[2], lq[3] for
            // odd e, as before)
            uint32_t p[32];
            float2 l01 = make_float2(lq[0], lq[1]), l23 = make_float2(lq[2], lq[3]);
            const float2 c22 = make_float2(c2, c2), nm2 = make_float2(-mref, -mref);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const float2 t = fma2(make_float2(s[2 * e], s[2 * e + 1]), c22, nm2);
                const float2 ee = make_float2(ex2(t.x), ex2(t.y));
                if (e & 1) l23 = add2(l23, ee);
                else l01 = add2(l01, ee);
                const uint32_t hi = f16x2_bits(ee.x, ee.y);
                const float2 lo = sub2(ee, f16x2_float2(hi));
                p[e] = hi;
                p[16 + e] = f16x2_bits(lo.x, lo.y);
            }
            lq[0] = l01.x;
            lq[1] = l01.y;
            lq[2] = l23.x;
            lq[3] = l23.y;
            tmem_st32(buf, p);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(bar_p + 8u * x);
        }

        // 4. Context: the warp's 32 columns of O / l * qkv_scale, once the
        //    last P v is complete (which completes every earlier one); l =
        //    the two warps' sums.
        float* rl = red + 512;
        rl[128 * hh + qi] = __fadd_rn(__fadd_rn(lq[0], lq[1]), __fadd_rn(lq[2], lq[3]));
        ok &= mbar_wait(bar_o + 8u * static_cast<uint32_t>((nkb - 1) & 1), static_cast<uint32_t>((nkb - 1) >> 1) & 1u,
                        wait_limit);
        __syncwarp();
        tc_fence_after();
        uint32_t o[32];
        tmem_ld32(lane + kColO + 32u * static_cast<uint32_t>(hh), o);
        tmem_wait_ld(o);
        pair_sync(qq);
        const int r = q0 + qi;
        griddep_wait();  // the output is written after the preceding kernel
        if (r < seq) {
            const float l = __fadd_rn(rl[qi], rl[128 + qi]);
            const float f = __fdiv_rn(vscale, l);
            const long long base = (row0 + r) * d + h * 64 + 32 * hh;
            if (kind == 3) {
                uint4* dst = reinterpret_cast<uint4*>(static_cast<int8_t*>(out) + base);
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    uint32_t w[4];
#pragma unroll
                    for (int i2 = 0; i2 < 4; ++i2) {
                        const int j2 = 16 * k + 4 * i2;
                        w[i2] = pack2_s8(__fmul_rn(__uint_as_float(o[j2]), f), __fmul_rn(__uint_as_float(o[j2 + 1]), f),
                                         inv_out_scale) |
                                (pack2_s8(__fmul_rn(__uint_as_float(o[j2 + 2]), f),
                                          __fmul_rn(__uint_as_float(o[j2 + 3]), f), inv_out_scale)
                                 << 16);
                    }
                    dst[k] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            } else {
                float4* dst = reinterpret_cast<float4*>(static_cast<float*>(out) + base);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    dst[k] = make_float4(__fmul_rn(__uint_as_float(o[4 * k]), f), __fmul_rn(__uint_as_float(o[4 * k + 1]), f),
                                         __fmul_rn(__uint_as_float(o[4 * k + 2]), f),
                                         __fmul_rn(__uint_as_float(o[4 * k + 3]), f));
            }
        }
    }
    if (!ok) {
        griddep_wait();
        atomicOr(&g_attn_status, static_cast<unsigned>(kStatusTimeout));
    }
    tc_fence_before();
    __syncthreads();
    if (mma_warp) tmem_dealloc(tm, kTmemCols);
}

}  // namespace

size_t attention_smem_bytes(int seq) {
    const size_t nkb = (static_cast<size_t>(seq) + kKeyBlock - 1) / kKeyBlock;
    // K and V tiles, 1024-byte alignment, 7 barriers + TMEM address, the
    // block maxima [2][2][128] and the sums [2][128]
    return 2 * nkb * kBlockBytes + 1024 + 64 + 4 * (512 + 256);
}

cudaError_t launch_attention(const int8_t* qkv, int batch, int seq, int heads, int ld, float score_scale,
                             float qkv_scale, int kind, float inv_out_scale, void* out, bool act_ready, cudaStream_t s) {
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
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = attention_smem_bytes(seq);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, attention_kernel, qkv, seq, heads * 64, ld, c2, qkv_scale, kind, inv_out_scale, out,
                           skip ? 64u : kWaitLimit, skip ? 1 : 0, act_ready ? 1 : 0);
    return e != cudaSuccess ? e : cudaGetLastError();
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
