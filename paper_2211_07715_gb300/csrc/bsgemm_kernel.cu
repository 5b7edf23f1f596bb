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
// * A CTA's quads are split evenly between its 16 warps.  Each warp streams
//   its contiguous range of 32-byte quad records through a two-chunk ring in
//   shared memory (cp.async, 512 bytes per chunk, the next chunk in flight
//   while the current one is consumed).  With 64-token tiles a lane covers
//   only half the warp's width, so the two half-warps take alternate quads
//   of a block-row and add their sums with one shuffle at the row's end.
//   A block-row that straddles a split between warps is summed in a
//   shared-memory slot (int32 atomics) and finished after a barrier.  All
//   sums are exact int32.
// * The epilogue runs in registers: int32 -> fp32 (RNE), one fma with scale
//   and bias, optional GELU by a fixed fp32 op sequence (A&S 7.1.28 erf),
//   optional requantise (fp32 multiply, round half to even, saturate).
#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "bsgemm.h"
#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kSmemOptin = 232448;  // sm_103 opt-in shared memory per block
constexpr int kSlots = kWarps - 1;  // one per split point between warp ranges
// Record ring per warp: kRingSlots chunks of ring_chunk(MT) quad records;
// while one chunk is consumed the next kRingSlots - 1 are in flight.
constexpr int kRingSlots = 4;
__host__ __device__ constexpr int ring_chunk(int MT) { return MT == 64 ? 8 : 16; }

__host__ __device__ constexpr int slot_words(int MT) { return 4 * MT; }  // MT tokens x 4 channels
constexpr size_t ring_bytes(int MT) { return static_cast<size_t>(kWarps) * kRingSlots * ring_chunk(MT) * 32; }

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
    const float e = __fsub_rn(1.0f, __frcp_rn(p16));  // IEEE 1/p16, round to nearest
    const float erf_x = (x < 0.0f) ? -e : e;
    return __fmul_rn(__fmul_rn(0.5f, y), __fadd_rn(1.0f, erf_x));
}

// The same erf-form GELU for fp32 outputs, with the hardware's approximate
// reciprocal (relative error <= 2^-22) in place of the IEEE one: fp32
// outputs are checked against a tolerance, not bit for bit, and the extra
// error stays below 2e-7 |y|.  int8 outputs use gelu_f32, which an int8
// decision must reproduce exactly.
__device__ __forceinline__ float gelu_f32_fast(float y) {
    const float x = y * 0.70710678f;
    const float ax = fabsf(x);
    float h = fmaf(ax, 0.0000430638f, 0.0002765672f);
    h = fmaf(ax, h, 0.0001520143f);
    h = fmaf(ax, h, 0.0092705272f);
    h = fmaf(ax, h, 0.0422820123f);
    h = fmaf(ax, h, 0.0705230784f);
    const float p = fmaf(ax, h, 1.0f);
    const float p2 = p * p, p4 = p2 * p2, p8 = p4 * p4, p16 = p8 * p8;
    float rcp;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(rcp) : "f"(p16));
    const float e = 1.0f - rcp;
    return 0.5f * y * (1.0f + ((x < 0.0f) ? -e : e));
}

// fp32 -> int8: one fp32 multiply, round half to even, saturate.
__device__ __forceinline__ uint32_t requant_s8(float v, float inv) {
    int q = __float2int_rn(__fmul_rn(v, inv));
    q = max(-128, min(127, q));
    return static_cast<uint32_t>(q) & 0xffu;
}

// Epilogue for one lane: tokens m_first + i, i < T (rows < M only), x the
// 4 channels of block-row r (scales s, bias b).  v[i * 4 + c] = token i,
// channel c.
template <int KIND, int T>
__device__ __forceinline__ void store_rows(const DeviceWeights& w, const LaunchArgs& a, long long m_first, int r,
                                           const int (&v)[T * 4], float4 s, float4 b) {
    const int N = w.N;
#pragma unroll
    for (int i = 0; i < T; ++i) {
        const long long m = m_first + i;
        if (m >= a.M) break;
        const size_t o = static_cast<size_t>(m) * N + 4 * r;
        const int* vi = v + 4 * i;
        if (KIND == 0) {
            *reinterpret_cast<int4*>(static_cast<int32_t*>(a.out) + o) = make_int4(vi[0], vi[1], vi[2], vi[3]);
        } else {
            float y0 = __fmaf_rn(__int2float_rn(vi[0]), s.x, b.x);
            float y1 = __fmaf_rn(__int2float_rn(vi[1]), s.y, b.y);
            float y2 = __fmaf_rn(__int2float_rn(vi[2]), s.z, b.z);
            float y3 = __fmaf_rn(__int2float_rn(vi[3]), s.w, b.w);
            if (KIND == 2) {
                y0 = gelu_f32_fast(y0);
                y1 = gelu_f32_fast(y1);
                y2 = gelu_f32_fast(y2);
                y3 = gelu_f32_fast(y3);
            } else if (KIND == 4) {
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

__device__ __forceinline__ float4 load_s4(const float* p, int r) { return __ldg(reinterpret_cast<const float4*>(p) + r); }

// Last index r in [lo, hi) with qp[r] <= q, given qp[lo] <= q < qp[hi]
// (qp: the shared-memory window of quad offsets).
__device__ __forceinline__ int row_of(const int* qp, int lo, int hi, int q) {
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (qp[mid] <= q) lo = mid; else hi = mid;
    }
    return lo;
}

// One staging unit: tokens 4g..4g+3 of the tile x columns 16kc..16kc+15.
// rw[i][j] = bytes of token 4g+i at columns 16kc+4j..16kc+4j+3 (zero past M
// or K).
__device__ __forceinline__ void load_unit(const LaunchArgs& a, int K, long long m0, int g, int kc,
                                          uint32_t (&rw)[4][4]) {
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
}

// Write one unit k-major: word g of rows 16kc..16kc+15 (tokens 4g..4g+3).
template <int MT>
__device__ __forceinline__ void store_unit(uint32_t* xt, int g, int kc, const uint32_t (&rw)[4][4]) {
    constexpr int RW = MT / 4;  // words per k-row
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint32_t t0, t1, t2, t3;
        transpose4(rw[0][j], rw[1][j], rw[2][j], rw[3][j], t0, t1, t2, t3);
        uint32_t* dst = xt + static_cast<size_t>(16 * kc + 4 * j) * RW + g;
        dst[0] = t0;
        dst[RW] = t1;
        dst[2 * RW] = t2;
        dst[3 * RW] = t3;
    }
}

// Stage activation rows m0..m0+MT-1, all K columns, into xt as k-major rows
// of MT bytes (word g of row k = tokens 4g..4g+3 at column k).  Each thread
// keeps kStageBatch units' loads in flight before transposing them.
template <int MT>
__device__ __forceinline__ void stage_tile(uint32_t* xt, const LaunchArgs& a, int K, int kpad, long long m0) {
    constexpr int G = MT / 4;
    constexpr int kStageBatch = 2;
    const int total = G * (kpad >> 4);
    for (int base = threadIdx.x; base < total; base += kStageBatch * kThreads) {
        uint32_t rw[kStageBatch][4][4];
#pragma unroll
        for (int b = 0; b < kStageBatch; ++b) {
            const int id = base + b * kThreads;
            if (id < total) load_unit(a, K, m0, id % G, id / G, rw[b]);
        }
#pragma unroll
        for (int b = 0; b < kStageBatch; ++b) {
            const int id = base + b * kThreads;
            if (id < total) store_unit<MT>(xt, id % G, id / G, rw[b]);
        }
    }
}

// cp.async (16 bytes, L2 only) into shared memory, and its group fences.
__device__ __forceinline__ void cp_async16(uint32_t smem_dst, const void* gmem_src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(smem_dst), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// Shared-memory loads with 32-bit shared-window addresses.
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ int4 lds128(uint32_t addr) {
    int4 v;
    asm volatile("ld.shared.v4.s32 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}
__device__ __forceinline__ uint2 lds64(uint32_t addr) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];\n" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

// mbarrier + bulk-copy (TMA) helpers.  Waits are bounded: a wait that
// gives up reports false and the caller records kStatusTimeout.
constexpr unsigned kWaitLimit = 1u << 20;

__device__ __forceinline__ void mbar_init(uint32_t bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, unsigned bytes) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n"
                 ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, unsigned parity) {
    for (unsigned i = 0; i < kWaitLimit; ++i) {
        unsigned done;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                     " selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(done) : "r"(bar), "r"(parity) : "memory");
        if (done) return true;
    }
    return false;
}
// Global -> shared bulk copy completing on an mbarrier (16-byte aligned, size % 16 == 0).
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, unsigned bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// Order this thread's earlier generic-proxy shared-memory accesses before
// later asynchronous-proxy (bulk copy) writes.
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }

// One quad for one lane's 8 tokens: 4 x 8 bytes from the k-major tile at the
// quad's columns, two 4x4 byte transposes, 32 dp4a (8 tokens x 4 channels).
template <int MT>
__device__ __forceinline__ void quad8(uint32_t xlane, const int4& kk, const int4& ww, int (&acc)[32]) {
    const uint2 x0 = lds64(xlane + kk.x * MT), x1 = lds64(xlane + kk.y * MT);
    const uint2 x2 = lds64(xlane + kk.z * MT), x3 = lds64(xlane + kk.w * MT);
    uint32_t t[8];
    transpose4(x0.x, x1.x, x2.x, x3.x, t[0], t[1], t[2], t[3]);
    transpose4(x0.y, x1.y, x2.y, x3.y, t[4], t[5], t[6], t[7]);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        acc[4 * i + 0] = __dp4a(static_cast<int>(t[i]), ww.x, acc[4 * i + 0]);
        acc[4 * i + 1] = __dp4a(static_cast<int>(t[i]), ww.y, acc[4 * i + 1]);
        acc[4 * i + 2] = __dp4a(static_cast<int>(t[i]), ww.z, acc[4 * i + 2]);
        acc[4 * i + 3] = __dp4a(static_cast<int>(t[i]), ww.w, acc[4 * i + 3]);
    }
}

// Sum the G lane groups' partial accumulators of one block-row and scatter
// the result: afterwards group g holds tokens [g*8/G, (g+1)*8/G) of its
// lanes' 8 (red[j*4 + c] = token g*8/G + j, channel c).
template <int G>
__device__ __forceinline__ void reduce_groups(int lane, const int (&acc)[32], int (&red)[32 / G]) {
    constexpr unsigned kFull = 0xffffffffu;
    const bool up = (lane & 16) != 0;
    if (G == 1) {
#pragma unroll
        for (int j = 0; j < 32 / G; ++j) red[j] = acc[j];
    } else if (G == 2) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int send = up ? acc[j] : acc[16 + j];
            const int keep = up ? acc[16 + j] : acc[j];
            red[j % (32 / G)] = keep + __shfl_xor_sync(kFull, send, 16);
        }
    } else {
        int k1[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int send = up ? acc[j] : acc[16 + j];
            const int keep = up ? acc[16 + j] : acc[j];
            k1[j] = keep + __shfl_xor_sync(kFull, send, 16);
        }
        const bool up2 = (lane & 8) != 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int send = up2 ? k1[j] : k1[8 + j];
            const int keep = up2 ? k1[8 + j] : k1[j];
            red[j % (32 / G)] = keep + __shfl_xor_sync(kFull, send, 8);
        }
    }
}

template <int MT, int KIND, bool TMA>
__global__ void __launch_bounds__(kThreads, 1)
bsgemm_kernel(DeviceWeights w, LaunchArgs a, const __grid_constant__ Schedule sched) {
    constexpr int LW = MT / 8;          // lanes spanning the token tile (8 tokens per lane)
    constexpr int G = 32 / LW;          // lane groups per warp; they interleave a block-row's quads
    constexpr int TPG = 8 / G;          // tokens per lane after the groups' sums are combined
    constexpr int SW = slot_words(MT);  // MT tokens x 4 channels
    constexpr int RC = ring_chunk(MT);  // records per ring chunk
    constexpr int S = RC / G;           // steps (G quads each) per ring chunk
    constexpr int kRec = 32;            // bytes per quad record
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_qp[kRowWin + 1];          // quad offsets of the current block-row window
    __shared__ __align__(8) unsigned long long s_bar;  // completion of the token tile's bulk copy
    __shared__ int s_cnt[kSlots];                      // warps that have added into each slot

    const int K = w.K;
    const int kpad = (K + 15) & ~15;
    uint32_t* xt = reinterpret_cast<uint32_t*>(smem);
    int* slots = reinterpret_cast<int*>(smem + static_cast<size_t>(kpad) * MT);
    unsigned char* ring = reinterpret_cast<unsigned char*>(slots + kSlots * SW);
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int g = lane / LW, li = lane % LW;
    const long long nbr = w.nbr;

    const uint32_t bar = smem_addr(&s_bar);
    if (TMA && tid == 0) mbar_init(bar, 1);
    // slots and their counters start at zero; whoever finishes a slot resets it
    for (int i = tid; i < kSlots * SW; i += kThreads) slots[i] = 0;
    if (tid < kSlots) s_cnt[tid] = 0;
    __syncthreads();
    unsigned phase = 0;
    long long u = sched.u[blockIdx.x];
    const long long u_end = sched.u[blockIdx.x + 1];
    unsigned char* ringw = ring + warp * (kRingSlots * RC * kRec);
    const uint32_t ring_s = smem_addr(ringw);
    const uint32_t xlane = smem_addr(xt) + 8 * li;  // this lane's 8 tokens in every k-row
    const int i0 = g * TPG;

    long long staged = -1;  // token tile currently in xt
    while (u < u_end) {
        // next window: one token tile, at most kRowWin consecutive block-rows
        const long long t = u / nbr;
        const int r_lo = static_cast<int>(u - t * nbr);
        const int r_hi = static_cast<int>(min(min(nbr, r_lo + (u_end - u)), static_cast<long long>(r_lo + kRowWin)));
        u += r_hi - r_lo;
        const long long m0 = t * MT;
        const long long m_lane = m0 + 8 * li + i0;  // first token this lane finishes
        // quad offset of block-row r (r_lo <= r <= r_hi), from the window
        auto qp = [&](int r) { return s_qp[r - r_lo]; };
        auto row_of_q = [&](int q) { return r_lo + row_of(s_qp, 0, r_hi - r_lo, q); };

        for (int i = tid; i <= r_hi - r_lo; i += kThreads) s_qp[i] = __ldg(w.qptr + r_lo + i);
        const bool stage = (t != staged);
        if (TMA && stage && tid == 0) {
            // one bulk copy of the token tile (already k-major in a.xb)
            const unsigned bytes = static_cast<unsigned>(kpad) * MT;
            const int8_t* src = a.xb + static_cast<size_t>(t) * kpad * MT;
            fence_proxy_async();
            mbar_arrive_expect_tx(bar, bytes);
            for (unsigned off = 0; off < bytes; off += 65536u)
                bulk_g2s(smem_addr(xt) + off, src + off, min(65536u, bytes - off), bar);
        }
        __syncthreads();  // the block-row window is visible
        if (!TMA && stage) {  // gather the tile with per-thread loads
            stage_tile<MT>(xt, a, K, kpad, m0);
            __syncthreads();
            staged = t;
        }

        const int qa = qp(r_lo), qb = qp(r_hi);
        // Every block-row holds a multiple of G quads, so the tile's quads form
        // nst steps of G; warps take an even split of the steps.
        const int nst = (qb - qa) / G;
        auto wstep = [&](int wi) { return static_cast<int>(static_cast<long long>(wi) * nst / kWarps); };
        const int ws0 = wstep(warp), ws1 = wstep(warp + 1);
        const int wq0 = qa + ws0 * G, wq1 = qa + ws1 * G;

        // Stream the warp's records [wq0, wq1) through the ring: chunk c =
        // records wq0 + RC*c ..; one 16-byte copy per lane (RC*2 lanes).  The
        // first chunks load while the token tile does.
        const unsigned char* gsrc = reinterpret_cast<const unsigned char*>(w.quads) + static_cast<size_t>(wq0) * kRec;
        const int nchunks = (wq1 - wq0 + RC - 1) / RC;
        auto issue = [&](int c) {
            if (c < nchunks && lane < RC * 2)
                cp_async16(ring_s + (c % kRingSlots) * (RC * kRec) + 16 * lane,
                           gsrc + static_cast<size_t>(c) * (RC * kRec) + 16 * lane);
            cp_async_commit();
        };
#pragma unroll
        for (int c = 0; c < kRingSlots; ++c) issue(c);

        // Block-rows with no stored block: acc = 0.
        for (int r = r_lo + warp; r < r_hi; r += kWarps) {
            if (qp(r) == qp(r + 1)) {
                int red[TPG * 4];
#pragma unroll
                for (int j = 0; j < TPG * 4; ++j) red[j] = 0;
                store_rows<KIND, TPG>(w, a, m_lane, r, red, load_s4(w.scale, r), load_s4(w.bias, r));
            }
        }

        if (TMA && stage) {
            const bool ok = mbar_wait(bar, phase & 1u);
            ++phase;
            if (__syncthreads_or(!ok)) {
                if (tid == 0) {
                    atomicOr(w.status, kStatusTimeout);
                    mbar_wait(bar, (phase - 1) & 1u);  // give the copy one more bounded chance to land
                }
                cp_async_wait<0>();
                __syncthreads();
                return;
            }
            staged = t;
        }

        if (wq0 < wq1) {
            cp_async_wait<kRingSlots - 1>();  // chunk 0 has landed
            __syncwarp();
            int cur = 0;
            int r = row_of_q(wq0);
            int p = 0;  // step index relative to ws0
            const int p_all = ws1 - ws0;
            while (p < p_all) {
                const int rs = qp(r), re_row = qp(r + 1);
                const int p_end = min(p_all, (re_row - wq0) / G);
                float4 sc = make_float4(0.f, 0.f, 0.f, 0.f), bi = sc;
                if (KIND != 0) {  // needed at the row's end; load it now
                    sc = load_s4(w.scale, r);
                    bi = load_s4(w.bias, r);
                }
                int acc[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) acc[i] = 0;
                while (p < p_end) {
                    const int cq = p / S;
                    if (cq != cur) {  // entering the next chunk (cq == cur + 1)
                        cur = cq;
                        __syncwarp();  // everyone is done with chunk cur - 1, whose slot is refilled
                        issue(cur + kRingSlots - 1);
                        cp_async_wait<kRingSlots - 1>();  // chunk cur has landed
                        __syncwarp();
                    }
                    const int seg_end = min(p_end, (cur + 1) * S);
                    uint32_t rec = ring_s + (cur % kRingSlots) * (RC * kRec) + ((p - cur * S) * G + g) * kRec;
                    for (; p + 1 < seg_end; p += 2, rec += 2 * G * kRec) {
                        const int4 k0 = lds128(rec), w0 = lds128(rec + 16);
                        const int4 k1 = lds128(rec + G * kRec), w1 = lds128(rec + G * kRec + 16);
                        quad8<MT>(xlane, k0, w0, acc);
                        quad8<MT>(xlane, k1, w1, acc);
                    }
                    if (p < seg_end) {
                        const int4 k0 = lds128(rec), w0 = lds128(rec + 16);
                        quad8<MT>(xlane, k0, w0, acc);
                        ++p;
                    }
                }
                int red[TPG * 4];
                reduce_groups<G>(lane, acc, red);
                if (rs >= wq0 && re_row <= wq1) {
                    store_rows<KIND, TPG>(w, a, m_lane, r, red, sc, bi);
                } else {
                    // Shared with other warps: sum into the slot of the first warp
                    // split inside the block-row; the last warp to add finishes it.
                    const int s0 = (rs - qa) / G, s1 = (re_row - qa) / G;  // the row's steps
                    const int b = static_cast<int>((static_cast<long long>(s0 + 1) * kWarps + nst - 1) / nst);
                    int* sl = slots + (b - 1) * SW + li;
#pragma unroll
                    for (int j = 0; j < TPG * 4; ++j) atomicAdd(sl + (4 * i0 + j) * LW, red[j]);
                    __syncwarp();
                    int arrived = 0;
                    if (lane == 0) {
                        __threadfence_block();
                        arrived = atomicAdd(&s_cnt[b - 1], 1) + 1;
                    }
                    arrived = __shfl_sync(0xffffffffu, arrived, 0);
                    int parts = 0;  // warps whose step range meets the row's
                    for (int wi = 0; wi < kWarps; ++wi) {
                        const int a0 = wstep(wi), a1 = wstep(wi + 1);
                        parts += (a0 < a1 && a0 < s1 && a1 > s0) ? 1 : 0;
                    }
                    if (arrived == parts) {
                        __threadfence_block();
#pragma unroll
                        for (int j = 0; j < TPG * 4; ++j) red[j] = atomicExch(sl + (4 * i0 + j) * LW, 0);
                        store_rows<KIND, TPG>(w, a, m_lane, r, red, sc, bi);
                        if (lane == 0) s_cnt[b - 1] = 0;
                    }
                }
                ++r;
                while (r < r_hi && qp(r + 1) == qp(r)) ++r;  // skip block-rows without quads
            }
        }
        cp_async_wait<0>();
        __syncthreads();  // the tile, window, ring and slots may be reused
    }
}

// Token-tile relayout: xb[t][k][j] = x[t*MT + j][k] for k < kpad (zero when
// t*MT + j >= M or k >= K).  A persistent CTA walks items (tile t, block of
// KC columns): MT tokens x KC columns (16 KB) through shared memory --
// 16-byte row loads, a 4x4 byte transpose per thread, 16-byte stores of the
// k-major block, which is contiguous in xb.  The next item's loads are in
// flight (in registers) while the current item is transposed and stored.
template <int MT>
__global__ void __launch_bounds__(256)
pretile_kernel(const int8_t* __restrict__ x, int M, int K, int kpad, int8_t* __restrict__ xb, long long items,
               int ncb) {
    constexpr int KC = 16384 / MT;     // columns per item (256 or 128)
    constexpr int C16 = KC / 16;       // 16-byte chunks per raw row
    constexpr int RW = KC / 4 + 4;     // raw row stride in words (rows shift by 4 banks)
    constexpr int OS = MT / 4 + 1;     // transposed row stride in words
    constexpr int NL = (MT * C16) / 256;  // row loads per thread and item
    __shared__ __align__(16) uint32_t raw[MT * RW];
    __shared__ uint32_t tr[KC * OS];
    const bool vec16 = ((K & 15) == 0) && ((reinterpret_cast<uintptr_t>(x) & 15) == 0);
    auto load_item = [&](long long it, uint4 (&v)[NL]) {
        const long long m0 = (it / ncb) * MT;
        const int k0 = static_cast<int>(it % ncb) * KC;
#pragma unroll
        for (int i = 0; i < NL; ++i) {
            const int c = i * 256 + threadIdx.x;
            const int rho = c / C16, c16 = c % C16;
            const long long m = m0 + rho;
            const int k = k0 + 16 * c16;
            v[i] = make_uint4(0u, 0u, 0u, 0u);
            if (m < M && k < K) {
                const int8_t* src = x + static_cast<size_t>(m) * K + k;
                if (vec16) {
                    v[i] = __ldg(reinterpret_cast<const uint4*>(src));
                } else {
                    uint32_t wv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (k + e < K) wv[e >> 2] |= static_cast<uint32_t>(static_cast<uint8_t>(src[e])) << (8 * (e & 3));
                    v[i] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                }
            }
        }
    };
    uint4 v[NL];
    long long it = blockIdx.x;
    if (it < items) load_item(it, v);
    for (; it < items; it += gridDim.x) {
        const long long t = it / ncb;
        const int k0 = static_cast<int>(it % ncb) * KC;
        const int kc = min(KC, kpad - k0);  // a multiple of 16
#pragma unroll
        for (int i = 0; i < NL; ++i) {
            const int c = i * 256 + threadIdx.x;
            *reinterpret_cast<uint4*>(raw + (c / C16) * RW + 4 * (c % C16)) = v[i];
        }
        __syncthreads();  // raw is complete; every thread is past the previous item's stores
        if (it + gridDim.x < items) load_item(it + gridDim.x, v);
        for (int i = threadIdx.x; i < (MT / 4) * (KC / 4); i += 256) {
            const int j = i % (KC / 4), g = i / (KC / 4);
            uint32_t t0, t1, t2, t3;
            transpose4(raw[(4 * g + 0) * RW + j], raw[(4 * g + 1) * RW + j], raw[(4 * g + 2) * RW + j],
                       raw[(4 * g + 3) * RW + j], t0, t1, t2, t3);
            tr[(4 * j + 0) * OS + g] = t0;
            tr[(4 * j + 1) * OS + g] = t1;
            tr[(4 * j + 2) * OS + g] = t2;
            tr[(4 * j + 3) * OS + g] = t3;
        }
        __syncthreads();  // tr is complete; raw may be refilled
        int8_t* dst = xb + (static_cast<size_t>(t) * kpad + k0) * MT;
        for (int i = threadIdx.x; i < kc * (MT / 16); i += 256) {
            const int row = i / (MT / 16), c = i % (MT / 16);
            const uint32_t* srow = tr + row * OS + 4 * c;
            *reinterpret_cast<uint4*>(dst + static_cast<size_t>(row) * MT + 16 * c) =
                make_uint4(srow[0], srow[1], srow[2], srow[3]);
        }
    }
}

template <int MT, bool TMA>
const void* kernel_for(int kind) {
    switch (kind) {
    case 0: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 0, TMA>);
    case 1: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 1, TMA>);
    case 2: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 2, TMA>);
    case 3: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 3, TMA>);
    default: return reinterpret_cast<const void*>(&bsgemm_kernel<MT, 4, TMA>);
    }
}

const void* kernel_ptr(int MT, int kind, bool tma) {
    if (MT == 128) return tma ? kernel_for<128, true>(kind) : kernel_for<128, false>(kind);
    return tma ? kernel_for<64, true>(kind) : kernel_for<64, false>(kind);
}

}  // namespace

size_t smem_bytes(int MT, int K) {
    const size_t kpad = (static_cast<size_t>(K) + 15) & ~static_cast<size_t>(15);
    return kpad * MT + static_cast<size_t>(kSlots) * slot_words(MT) * 4 + ring_bytes(MT);
}

int tile_for_k(int K) {
    if (K < 1) return 0;
    if (smem_bytes(128, K) + kStaticSmem <= static_cast<size_t>(kSmemOptin)) return 128;
    if (smem_bytes(64, K) + kStaticSmem <= static_cast<size_t>(kSmemOptin)) return 64;
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
        for (int tma = 0; tma < 2; ++tma) {
            cudaError_t e = cudaFuncSetAttribute(kernel_ptr(MT, kind, tma != 0),
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemOptin - kStaticSmem);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, kernel_ptr(MT, 0, true), kThreads, smem);
}

cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, const Schedule& sched, int MT, int grid,
                   cudaStream_t s) {
    const size_t smem = smem_bytes(MT, w.K);
#define BSG_LAUNCH(MTV, KV)                                                                   \
    do {                                                                                      \
        if (a.xb) bsgemm_kernel<MTV, KV, true><<<grid, kThreads, smem, s>>>(w, a, sched);     \
        else bsgemm_kernel<MTV, KV, false><<<grid, kThreads, smem, s>>>(w, a, sched);         \
    } while (0)
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

size_t tiled_bytes(int MT, int K, long long M) {
    const size_t kpad = (static_cast<size_t>(K) + 15) & ~static_cast<size_t>(15);
    return static_cast<size_t>((M + MT - 1) / MT) * kpad * MT;
}

cudaError_t launch_pretile(const int8_t* x, int M, int K, int MT, int8_t* xb, int sms, cudaStream_t s) {
    const int kpad = (K + 15) & ~15;
    const int ncb = (kpad + 16384 / MT - 1) / (16384 / MT);
    const long long items = (static_cast<long long>(M) + MT - 1) / MT * ncb;
    const long long cap = 4LL * (sms > 0 ? sms : 1);  // 4 resident CTAs per SM (35 KB of shared memory each)
    const unsigned grid = static_cast<unsigned>(items < cap ? items : cap);
    if (MT == 128) pretile_kernel<128><<<grid, 256, 0, s>>>(x, M, K, kpad, xb, items, ncb);
    else pretile_kernel<64><<<grid, 256, 0, s>>>(x, M, K, kpad, xb, items, ncb);
    return cudaGetLastError();
}

}  // namespace bsg

// Token-tile scratch of bsgemm_run_static: one fixed array per device, so
// that entry point allocates nothing.  Every byte a run reads from it is
// written by the relayout kernel of the same run (tokens past M and columns
// past K as zeros), so nothing in it has to start at zero.
static __device__ __align__(256) int8_t g_static_tiles[BSGEMM_STATIC_SCRATCH_BYTES];

namespace bsg {

cudaError_t static_scratch(int device, int8_t** ptr) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static int8_t* addr[kMaxDevices] = {};
    if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[device]) {
        // Resolved once per device, with that device current (the caller
        // checks): the address of this module's copy in its context.
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_static_tiles);
        if (e != cudaSuccess) return e;
        addr[device] = static_cast<int8_t*>(p);
    }
    *ptr = addr[device];
    return cudaSuccess;
}

}  // namespace bsg
