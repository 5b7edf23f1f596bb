// Block-sparse INT8 linear on sm_103a: gather + dp4a + fused epilogue.
//
// What the kernel computes is the layer of Sec. 3 "Sparse GEMM operators"
// (Algorithm 1, App. A.3.4): a dense int8 input times a weight sparse in
// 4x1 blocks (4 output rows x 1 input column, App. A.1), int32 dot-4
// accumulation, then the fused post-operators (App. A.3.3): dequantise +
// bias, optional erf-GELU, optional requantise to int8.
//
// GB300 design (not a translation of the paper's AVX-512 loop nest):
//
// * Unit of work: (token tile t, block-row r) -- MT tokens x 4 output
//   channels, reduced over the block-row's stored columns.  Units are
//   ordered tile-major and split into one contiguous, cost-balanced range per
//   CTA of a persistent grid (CTAs = SMs x resident CTAs), so every SM gets
//   the same number of quads regardless of M.
// * The CTA stages its token tile of the activations for ALL of K in shared
//   memory, transposed to "k-major" rows (row k holds the MT tokens' bytes at
//   column k), once per tile; every block-row of the tile then gathers from
//   it.  This is the re-organisation of the input by the mask that
//   Algorithm 1 does with vpermt2d/vpshufb, done once per tile instead of
//   once per block.
// * Lanes own 4 consecutive tokens.  For one quad (4 stored columns k0..k3 of
//   one block-row) a lane reads 4 words (one per column, 4 tokens each),
//   transposes the 4x4 bytes with 8 byte-permutes into one dot-4 operand per
//   token, and issues 16 dp4a (4 tokens x 4 channels) against the quad's 4
//   weight words -- the analogue of Algorithm 1's broadcast weight block A,
//   re-organised input block B and 4 vpdpbusd.  GB300 runs int8 dot products
//   at the same rate on dp4a as on its int8 MMA paths, so no tensor-core path
//   is faster here (the 4-channel block cannot fill an MMA tile).
// * A CTA's quads are split evenly between its lane groups; a block-row that
//   straddles a split point is summed in a shared-memory slot (int32 atomics)
//   and finished after a barrier.  All sums are exact int32.
// * The epilogue runs in registers: int32 -> fp32 (RNE), one fma with scale
//   and bias, optional GELU by a fixed fp32 op sequence (A&S 7.1.28 erf),
//   optional requantise (fp32 multiply, round half to even, saturate).
#include <cstdint>
#include <cuda_runtime.h>

#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kSmemOptin = 232448;  // sm_103 opt-in shared memory per block

__host__ __device__ constexpr int groups_per_cta(int MT) { return kThreads / (MT / 4); }
__host__ __device__ constexpr int slot_words(int MT) { return 16 * (MT / 4); }

// 4x4 byte transpose.  In: a/b/c/d = bytes (x0..x3) of rows 0..3.  Out:
// t_i = (a_i, b_i, c_i, d_i).
__device__ __forceinline__ void transpose4(uint32_t a, uint32_t b, uint32_t c, uint32_t d,
                                           uint32_t& t0, uint32_t& t1, uint32_t& t2, uint32_t& t3) {
    const uint32_t ab_lo = __byte_perm(a, b, 0x5140);  // a0 b0 a1 b1
    const uint32_t ab_hi = __byte_perm(a, b, 0x7362);  // a2 b2 a3 b3
    const uint32_t cd_lo = __byte_perm(c, d, 0x5140);  // c0 d0 c1 d1
    const uint32_t cd_hi = __byte_perm(c, d, 0x7362);  // c2 d2 c3 d3
    t0 = __byte_perm(ab_lo, cd_lo, 0x5410);            // a0 b0 c0 d0
    t1 = __byte_perm(ab_lo, cd_lo, 0x7632);            // a1 b1 c1 d1
    t2 = __byte_perm(ab_hi, cd_hi, 0x5410);            // a2 b2 c2 d2
    t3 = __byte_perm(ab_hi, cd_hi, 0x7632);            // a3 b3 c3 d3
}

// erf-form GELU in fp32 by a fixed sequence of IEEE round-to-nearest ops.
// erf(|x|) = 1 - p(|x|)^-16, p = 1 + a1 x + ... + a6 x^6 (Abramowitz &
// Stegun 7.1.28, |error| <= 3e-7); p^16 by four squarings.
__device__ __forceinline__ float gelu_f32(float y) {
    const float x = __fmul_rn(y, 0.70710678f);
    const float ax = fabsf(x);
    float h = __fmaf_rn(ax, 0.0000430638f, 0.0002765672f);
    h = __fmaf_rn(ax, h, 0.0001520143f);
    h = __fmaf_rn(ax, h, 0.0092705272f);
    h = __fmaf_rn(ax, h, 0.0422820123f);
    h = __fmaf_rn(ax, h, 0.0705230784f);
    const float p = __fmaf_rn(ax, h, 1.0f);
    const float p2 = __fmul_rn(p, p);
    const float p4 = __fmul_rn(p2, p2);
    const float p8 = __fmul_rn(p4, p4);
    const float p16 = __fmul_rn(p8, p8);
    const float e = __fsub_rn(1.0f, __fdiv_rn(1.0f, p16));
    const float erf_x = (x < 0.0f) ? -e : e;
    return __fmul_rn(__fmul_rn(0.5f, y), __fadd_rn(1.0f, erf_x));
}

// fp32 -> int8: one fp32 multiply, round half to even, saturate.
__device__ __forceinline__ uint32_t requant_s8(float v, float inv) {
    int q = __float2int_rn(__fmul_rn(v, inv));
    q = max(-128, min(127, q));
    return static_cast<uint32_t>(q) & 0xffu;
}

// Epilogue for one lane: tokens m_first..m_first+3 (rows < M only) x the 4
// channels of block-row r.  acc[i * 4 + c] = token i, channel c.
template <int KIND>
__device__ __forceinline__ void store_tile(const DeviceWeights& w, const LaunchArgs& a, long long m_first,
                                           int r, const int (&acc)[16]) {
    const int N = w.N;
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f), b = s;
    if (KIND != 0) {
        s = __ldg(reinterpret_cast<const float4*>(w.scale) + r);
        b = __ldg(reinterpret_cast<const float4*>(w.bias) + r);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const long long m = m_first + i;
        if (m >= a.M) break;
        const size_t o = static_cast<size_t>(m) * N + 4 * r;
        const int* v = acc + 4 * i;
        if (KIND == 0) {
            *reinterpret_cast<int4*>(static_cast<int32_t*>(a.out) + o) = make_int4(v[0], v[1], v[2], v[3]);
        } else {
            float y0 = __fmaf_rn(__int2float_rn(v[0]), s.x, b.x);
            float y1 = __fmaf_rn(__int2float_rn(v[1]), s.y, b.y);
            float y2 = __fmaf_rn(__int2float_rn(v[2]), s.z, b.z);
            float y3 = __fmaf_rn(__int2float_rn(v[3]), s.w, b.w);
            if (KIND == 2 || KIND == 4) {
                y0 = gelu_f32(y0);
                y1 = gelu_f32(y1);
                y2 = gelu_f32(y2);
                y3 = gelu_f32(y3);
            }
            if (KIND == 1 || KIND == 2) {
                *reinterpret_cast<float4*>(static_cast<float*>(a.out) + o) = make_float4(y0, y1, y2, y3);
            } else {
                const float inv = a.inv_out_scale;
                const uint32_t packed = requant_s8(y0, inv) | (requant_s8(y1, inv) << 8) |
                                        (requant_s8(y2, inv) << 16) | (requant_s8(y3, inv) << 24);
                *reinterpret_cast<uint32_t*>(static_cast<int8_t*>(a.out) + o) = packed;
            }
        }
    }
}

// Last block-row r in [lo, hi) with qptr[r] <= q, given qptr[lo] <= q < qptr[hi].
__device__ __forceinline__ int row_of(const int32_t* qptr, int lo, int hi, int q) {
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(qptr + mid) <= q) lo = mid; else hi = mid;
    }
    return lo;
}

// Stage activations rows m0..m0+MT-1, all K columns, into xt as k-major rows
// of MT bytes (word g of row k = tokens 4g..4g+3 at column k).  Rows >= M and
// columns >= K read as zero.
template <int MT>
__device__ __forceinline__ void stage_tile(uint32_t* xt, const LaunchArgs& a, int K, int kpad, long long m0) {
    constexpr int G = MT / 4;
    const int nkc = kpad >> 4;
    for (int id = threadIdx.x; id < G * nkc; id += kThreads) {
        const int g = id % G, kc = id / G;
        uint32_t rw[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const long long m = m0 + 4 * g + i;
            if (m < a.M) {
                const int8_t* src = a.x + static_cast<size_t>(m) * K + 16 * kc;
                if (a.x_vec16) {
                    const int4 v = __ldg(reinterpret_cast<const int4*>(src));
                    rw[i][0] = v.x; rw[i][1] = v.y; rw[i][2] = v.z; rw[i][3] = v.w;
                } else {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        uint32_t word = 0;
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int k = 16 * kc + 4 * j + e;
                            const uint32_t byte = (k < K) ? static_cast<uint8_t>(src[4 * j + e]) : 0u;
                            word |= byte << (8 * e);
                        }
                        rw[i][j] = word;
                    }
                }
            } else {
                rw[i][0] = rw[i][1] = rw[i][2] = rw[i][3] = 0u;
            }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            uint32_t t0, t1, t2, t3;
            transpose4(rw[0][j], rw[1][j], rw[2][j], rw[3][j], t0, t1, t2, t3);
            uint32_t* dst = xt + static_cast<size_t>(16 * kc + 4 * j) * G + g;
            dst[0] = t0;
            dst[G] = t1;
            dst[2 * G] = t2;
            dst[3 * G] = t3;
        }
    }
}

template <int MT, int KIND>
__global__ void __launch_bounds__(kThreads, 1)
bsgemm_kernel(DeviceWeights w, LaunchArgs a, long long ntiles, long long ctile, int grid) {
    constexpr int GL = MT / 4;               // lanes per block-row group
    constexpr int H = groups_per_cta(MT);    // lane groups per CTA
    constexpr int SW = slot_words(MT);       // int32 words per slot
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ long long s_range[2];

    const int K = w.K;
    const int kpad = (K + 15) & ~15;
    uint32_t* xt = reinterpret_cast<uint32_t*>(smem);
    int* slots = reinterpret_cast<int*>(smem + static_cast<size_t>(kpad) * MT);
    const int tid = threadIdx.x;
    const int h = tid / GL, li = tid % GL;
    const long long nbr = w.nbr;

    // This CTA's units: [U(c), U(c+1)), U(c) = first unit whose start cost
    // reaches c * total / grid (unit (t, r) starts at t * ctile + cost[r]).
    if (tid < 2) {
        const long long c = static_cast<long long>(blockIdx.x) + tid;
        const long long target = c * ctile * ntiles / grid;
        const long long t = target / ctile, rem = target - t * ctile;
        int lo = 0, hi = static_cast<int>(nbr);
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(w.cost + mid) >= rem) hi = mid; else lo = mid + 1;
        }
        s_range[tid] = t * nbr + lo;
    }
    __syncthreads();
    long long u = s_range[0];
    const long long u_end = s_range[1];

    while (u < u_end) {
        const long long t = u / nbr;
        const int r_lo = static_cast<int>(u - t * nbr);
        const int r_hi = static_cast<int>(min(nbr, r_lo + (u_end - u)));
        u += r_hi - r_lo;
        const long long m0 = t * MT;

        stage_tile<MT>(xt, a, K, kpad, m0);
        for (int i = tid; i < (H - 1) * SW; i += kThreads) slots[i] = 0;
        __syncthreads();

        const int qa = __ldg(w.qptr + r_lo), qb = __ldg(w.qptr + r_hi);
        const int qn = qb - qa;
        const int q_begin = qa + static_cast<int>(static_cast<long long>(h) * qn / H);
        const int q_end = qa + static_cast<int>(static_cast<long long>(h + 1) * qn / H);
        const long long m_first = m0 + 4 * li;

        if (q_begin < q_end) {
            const uint32_t* xl = xt + li;
            int r = row_of(w.qptr, r_lo, r_hi, q_begin);
            int q = q_begin;
            while (q < q_end) {
                const int rs = __ldg(w.qptr + r), re = __ldg(w.qptr + r + 1);
                const int seg_end = min(re, q_end);
                int acc[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[i] = 0;
                int4 kk = __ldg(w.quads + 2 * q);
                int4 ww = __ldg(w.quads + 2 * q + 1);
                for (; q < seg_end; ++q) {
                    // the quad array carries one padding record, so q + 1 is in bounds
                    const int4 kn = __ldg(w.quads + 2 * q + 2);
                    const int4 wn = __ldg(w.quads + 2 * q + 3);
                    const uint32_t x0 = xl[kk.x * GL], x1 = xl[kk.y * GL];
                    const uint32_t x2 = xl[kk.z * GL], x3 = xl[kk.w * GL];
                    uint32_t t0, t1, t2, t3;
                    transpose4(x0, x1, x2, x3, t0, t1, t2, t3);
                    acc[0] = __dp4a(static_cast<int>(t0), ww.x, acc[0]);
                    acc[1] = __dp4a(static_cast<int>(t0), ww.y, acc[1]);
                    acc[2] = __dp4a(static_cast<int>(t0), ww.z, acc[2]);
                    acc[3] = __dp4a(static_cast<int>(t0), ww.w, acc[3]);
                    acc[4] = __dp4a(static_cast<int>(t1), ww.x, acc[4]);
                    acc[5] = __dp4a(static_cast<int>(t1), ww.y, acc[5]);
                    acc[6] = __dp4a(static_cast<int>(t1), ww.z, acc[6]);
                    acc[7] = __dp4a(static_cast<int>(t1), ww.w, acc[7]);
                    acc[8] = __dp4a(static_cast<int>(t2), ww.x, acc[8]);
                    acc[9] = __dp4a(static_cast<int>(t2), ww.y, acc[9]);
                    acc[10] = __dp4a(static_cast<int>(t2), ww.z, acc[10]);
                    acc[11] = __dp4a(static_cast<int>(t2), ww.w, acc[11]);
                    acc[12] = __dp4a(static_cast<int>(t3), ww.x, acc[12]);
                    acc[13] = __dp4a(static_cast<int>(t3), ww.y, acc[13]);
                    acc[14] = __dp4a(static_cast<int>(t3), ww.z, acc[14]);
                    acc[15] = __dp4a(static_cast<int>(t3), ww.w, acc[15]);
                    kk = kn;
                    ww = wn;
                }
                if (rs >= q_begin && re <= q_end) {
                    store_tile<KIND>(w, a, m_first, r, acc);
                } else {
                    // Block-row shared with other groups: its slot is the first
                    // split point inside it, b = ceil((rs - qa + 1) * H / qn).
                    const long long d = rs - qa;
                    const int b = static_cast<int>(((d + 1) * H + qn - 1) / qn);
                    int* sl = slots + (b - 1) * SW + li;
#pragma unroll
                    for (int i = 0; i < 16; ++i) atomicAdd(sl + i * GL, acc[i]);
                }
                while (r < r_hi && __ldg(w.qptr + r + 1) <= q) ++r;
            }
        }
        __syncthreads();

        // Finish the shared block-rows: group h owns split point b = h + 1.
        if (h < H - 1 && qn > 0) {
            const int b = h + 1;
            const int pb = qa + static_cast<int>(static_cast<long long>(b) * qn / H);
            if (pb < qb) {
                const int r = row_of(w.qptr, r_lo, r_hi, pb);
                const int rs = __ldg(w.qptr + r);
                if (rs < pb) {
                    const long long d = rs - qa;
                    const int bf = static_cast<int>(((d + 1) * H + qn - 1) / qn);
                    if (bf == b) {
                        int acc[16];
                        const int* sl = slots + (b - 1) * SW + li;
#pragma unroll
                        for (int i = 0; i < 16; ++i) acc[i] = sl[i * GL];
                        store_tile<KIND>(w, a, m_first, r, acc);
                    }
                }
            }
        }
        // Block-rows with no stored block: acc = 0.
        for (int r = r_lo + h; r < r_hi; r += H) {
            if (__ldg(w.qptr + r) == __ldg(w.qptr + r + 1)) {
                int acc[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[i] = 0;
                store_tile<KIND>(w, a, m_first, r, acc);
            }
        }
        __syncthreads();
    }
}

template <int MT>
const void* kernel_for(int kind) {
    switch (kind) {
    case 0: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 0>);
    case 1: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 1>);
    case 2: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 2>);
    case 3: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 3>);
    default: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 4>);
    }
}

const void* kernel_ptr(int MT, int kind) { return MT == 128 ? kernel_for<128>(kind) : kernel_for<64>(kind); }

}  // namespace

size_t smem_bytes(int MT, int K) {
    const size_t kpad = (static_cast<size_t>(K) + 15) & ~static_cast<size_t>(15);
    return kpad * MT + static_cast<size_t>(groups_per_cta(MT) - 1) * slot_words(MT) * 4;
}

int tile_for_k(int K) {
    if (K < 1) return 0;
    // static shared memory (the CTA's unit range) takes 16 bytes
    if (smem_bytes(128, K) + 16 <= static_cast<size_t>(kSmemOptin)) return 128;
    if (smem_bytes(64, K) + 16 <= static_cast<size_t>(kSmemOptin)) return 64;
    return 0;
}

int max_k() {
    int k = 16;
    while (tile_for_k(k + 16)) k += 16;
    return k;
}

cudaError_t prepare_kernels(int MT, int K, int* ctas_per_sm) {
    const int smem = static_cast<int>(smem_bytes(MT, K));
    for (int kind = 0; kind < 5; ++kind) {
        cudaError_t e = cudaFuncSetAttribute(kernel_ptr(MT, kind), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemOptin - 16);
        if (e != cudaSuccess) return e;
    }
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, kernel_ptr(MT, 0), kThreads, smem);
}

cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, int MT, int grid, cudaStream_t s) {
    const long long ntiles = (static_cast<long long>(a.M) + MT - 1) / MT;
    const long long ctile = static_cast<long long>(w.Q) + w.nbr;  // cost[nbr]
    const size_t smem = smem_bytes(MT, w.K);
#define BSG_LAUNCH(MTV, KV) \
    bsgemm_kernel<MTV, KV><<<grid, kThreads, smem, s>>>(w, a, ntiles, ctile, grid)
    if (MT == 128) {
        switch (a.kind) {
        case 0: BSG_LAUNCH(128, 0); break;
        case 1: BSG_LAUNCH(128, 1); break;
        case 2: BSG_LAUNCH(128, 2); break;
        case 3: BSG_LAUNCH(128, 3); break;
        default: BSG_LAUNCH(128, 4); break;
        }
    } else {
        switch (a.kind) {
        case 0: BSG_LAUNCH(64, 0); break;
        case 1: BSG_LAUNCH(64, 1); break;
        case 2: BSG_LAUNCH(64, 2); break;
        case 3: BSG_LAUNCH(64, 3); break;
        default: BSG_LAUNCH(64, 4); break;
        }
    }
#undef BSG_LAUNCH
    return cudaGetLastError();
}

}  // namespace bsg
