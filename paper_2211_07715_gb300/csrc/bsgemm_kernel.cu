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
// * Block-rows are sorted by length and taken 4 at a time into row groups
//   (16 output channels).  Unit of work: (token tile t, row group) -- 64
//   tokens x 16 channels.  Units are ordered tile-major and split into one
//   contiguous, cost-balanced range per CTA of a persistent grid (CTAs =
//   SMs x resident CTAs).
// * The CTA stages its token tile of the activations for ALL of K in shared
//   memory once, swizzled k-major; every row group of the tile then gathers
//   from it.  This is the re-organisation of the input by the mask that
//   Algorithm 1 does with vpermt2d/vpshufb, done once per tile instead of
//   once per block.  The fast path copies 64 x 64-byte boxes of x [M][K] by
//   tensor copies and each warp transposes its boxes in place; K-major x^T
//   lands in the layout as it is; other shapes use tiles the relayout
//   kernel wrote (one bulk copy) or per-thread gathers.
// * One step of a warp takes one quad (4 stored columns) of each of the
//   group's 4 block-rows: two transposed shared-memory gathers (ldmatrix
//   .m16n16 .b8) give lane l (q = l % 4, g = l / 4) 8 dot-4 operands -- tokens
//   g + 8 i x the 4 columns of block-row q's quad -- with no byte permutes,
//   and the lane issues 32 dp4a against the quad's 4 channel words:
//   Algorithm 1's broadcast weight block A, re-organised input block B and
//   vpdpbusd, 8 tokens at a time.  Each lane thus owns whole outputs of its
//   block-row: no cross-lane sum.  The columns of each half-step are chosen
//   at create time to fall in distinct shared-memory bank groups of the
//   swizzled tile, so a gather reads in one pass per 8 rows.
// * A CTA's steps are split evenly between its 8 warps.  Each warp reads
//   its contiguous range of 128-byte step records straight from global
//   memory (L1/L2) into a 12-deep register ring.  A row group that
//   straddles a split between warps is summed in a shared-memory slot
//   (int32 atomics) and finished after the window's barrier.
// * GB300 runs int8 dot products on dp4a at the rate of its int8 MMA paths
//   (tcgen05 has no int8 kind on sm_103a), and a 4-channel block cannot fill
//   an MMA tile, so the contraction stays on dp4a.
// * The epilogue runs in registers: int32 -> fp32 (RNE), one fma with scale
//   and bias, optional GELU by a fixed fp32 op sequence (A&S 7.1.28 erf),
//   optional requantise (fp32 multiply, round half to even, saturate), or
//   the residual add before LayerNorm (the LayerNorm itself is a row-wise
//   kernel at the end of this file).
#include <cstdint>
#include <cstring>
#include <mutex>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "bsgemm.h"
#include "bsgemm_device.cuh"
#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kSmemOptin = 232448;  // sm_103 opt-in shared memory per block
constexpr int kSlots = kWarps - 1;  // one per split point between warp ranges
static_assert(kRing == 3 * kBlock, "a ring round is three blocks of steps");
// Cost of a row group's end (epilogue, stores) in steps, for splitting a
// window's work evenly between warps.
#ifndef BSG_GROUP_END_COST
#define BSG_GROUP_END_COST 14
#endif
constexpr int kGroupEndCost = BSG_GROUP_END_COST;
// Bytes per bulk copy of a token tile into shared memory (a multiple of 16).
#ifndef BSG_TMA_PIECE
#define BSG_TMA_PIECE 65536
#endif
constexpr unsigned kTmaPiece = BSG_TMA_PIECE;
// Fewest tensor copies of a token tile when x is copied as a 3-D view
// (each copy then brings box_d of its 64-column boxes).
#ifndef BSG_MIN_COPIES
#define BSG_MIN_COPIES 8
#endif
constexpr int kMinCopies = BSG_MIN_COPIES;

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


// Byte offset of chunk 0 of activation column k in a swizzled token tile
// (rows 2i, 2i+1 share 128-byte line i; chunk c of row k in 16-byte slot
// (4 (k & 1) + c) XOR (i & 3)); chunk c is at row_off(k) XOR 16 c.
__device__ __forceinline__ uint32_t row_off(int k) {
    const uint32_t line = static_cast<uint32_t>(k) >> 1;
    return (line << 7) | ((((static_cast<uint32_t>(k) & 1u) << 2) ^ (line & 3u)) << 4);
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

// Write one unit into the swizzled tile: word (tokens 4g..4g+3) of rows
// 16kc..16kc+15; the word lies in chunk g / 4 at byte 4 (g % 4).
__device__ __forceinline__ void store_unit(unsigned char* xt, int g, int kc, const uint32_t (&rw)[4][4]) {
    const uint32_t cx = static_cast<uint32_t>(g >> 2) << 4, wb = 4u * static_cast<uint32_t>(g & 3);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint32_t t[4];
        transpose4(rw[0][j], rw[1][j], rw[2][j], rw[3][j], t[0], t[1], t[2], t[3]);
#pragma unroll
        for (int e = 0; e < 4; ++e)
            *reinterpret_cast<uint32_t*>(xt + ((row_off(16 * kc + 4 * j + e) ^ cx) + wb)) = t[e];
    }
}

// Stage activation rows m0..m0+63, all kpad columns, into the swizzled tile
// with per-thread loads.  Each thread keeps kStageBatch units' loads in
// flight before transposing them.
#ifndef BSG_STAGE_BATCH
#define BSG_STAGE_BATCH 4
#endif
__device__ __forceinline__ void stage_tile(unsigned char* xt, const LaunchArgs& a, int K, int kpad, long long m0) {
    constexpr int G = kTile / 4;
    constexpr int kStageBatch = BSG_STAGE_BATCH;
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
            if (id < total) store_unit(xt, id % G, id / G, rw[b]);
        }
    }
}


// Staging from the activations themselves (no relayout kernel): a tensor
// copy brings box b of the token tile -- 64 tokens x columns 64b..64b+63,
// row-major, 64 bytes a token -- into the tile's bytes [4096 b, 4096 b +
// 4096), with the 64-byte swizzle: token r's 16-byte chunk c at 64 r + 16
// (c ^ ((r >> 1) & 3)).  Those are the bytes the box's columns take in the
// swizzled k-major tile, so one warp turns the box around in place: eight
// transposed matrix loads (16 tokens x 16 columns each; lane l addresses
// token row l of the two matrices) put the whole box in registers, and 32
// word stores write lane (g, q)'s words -- 4 tokens of one column -- to
// their column rows.  Both the loads (8 tokens of a phase on 8 distinct
// 16-byte slots) and the stores (8 columns x 4 words on 32 banks) are free
// of bank conflicts.
__device__ __forceinline__ void transpose_box(uint32_t tb, int b, int lane) {
    const uint32_t box = tb + 4096u * static_cast<uint32_t>(b);
    uint32_t v[8][4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint32_t r = 32u * h + static_cast<uint32_t>(lane);
            ldsm_x2_trans_b8(box + 64u * r + 16u * (static_cast<uint32_t>(c) ^ ((r >> 1) & 3u)), v[4 * h + c][0],
                             v[4 * h + c][1], v[4 * h + c][2], v[4 * h + c][3]);
        }
    }
    __syncwarp();
    const int g = lane >> 2;
    const uint32_t wq4 = 4u * static_cast<uint32_t>(lane & 3);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int k = 64 * b + 16 * c + g;
            const uint32_t o0 = row_off(k), o1 = row_off(k + 8);
            const uint32_t j0 = 32u * h, j1 = 32u * h + 16u;  // chunks 2h, 2h + 1 (16 tokens each)
            st_shared_u32(tb + (o0 ^ j0) + wq4, v[4 * h + c][0]);
            st_shared_u32(tb + (o1 ^ j0) + wq4, v[4 * h + c][1]);
            st_shared_u32(tb + (o0 ^ j1) + wq4, v[4 * h + c][2]);
            st_shared_u32(tb + (o1 ^ j1) + wq4, v[4 * h + c][3]);
        }
    }
}

// One step for one lane: the step's 16 columns x the tile's 64 tokens come
// in by two transposed gathers (tokens 0-31, then 32-63); lane l (g = l / 4,
// q = l % 4) receives x[g + 8 i][k_{4q} .. k_{4q+3}] as word t[i], i < 8, and
// issues 32 dp4a against quad q's 4 channel words.  `off` is the step's
// column offset for row l % 16, lb = 16 (l / 16) selects the chunk (16
// tokens) of matrix l / 16.  tb is 128-byte aligned, so XOR with 16 c moves
// to chunk c of the same row.
__device__ __forceinline__ void gather16(uint32_t tb, uint32_t lb, int off, uint32_t (&t)[8]) {
    const uint32_t a0 = tb + (static_cast<uint32_t>(off) ^ lb);
    ldsm_x2_trans_b8(a0, t[0], t[1], t[2], t[3]);
    ldsm_x2_trans_b8(a0 ^ 32u, t[4], t[5], t[6], t[7]);
}
__device__ __forceinline__ void dot16(const uint32_t (&t)[8], const int4& w, int (&acc)[32]) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        acc[4 * i + 0] = __dp4a(static_cast<int>(t[i]), w.x, acc[4 * i + 0]);
        acc[4 * i + 1] = __dp4a(static_cast<int>(t[i]), w.y, acc[4 * i + 1]);
        acc[4 * i + 2] = __dp4a(static_cast<int>(t[i]), w.z, acc[4 * i + 2]);
        acc[4 * i + 3] = __dp4a(static_cast<int>(t[i]), w.w, acc[4 * i + 3]);
    }
}

// This lane's view of the step records: ro points at the column offset of
// row (lane % 16) of a step, rw at quad q's 4 channel words of the same
// step; step s + i is at ro + 32 i, rw + 8 i.
struct RecPtr {
    const int* ro;
    const int4* rw;
    __device__ __forceinline__ RecPtr(const int4* recs, long long s, int lane, int q)
        : ro(reinterpret_cast<const int*>(recs + s * 8) + (lane & 15)), rw(recs + s * 8 + 4 + q) {}
    __device__ __forceinline__ void load(int i, int& off, int4& w, uint64_t pol) const {
        off = ldg_hint(ro + 32 * i, pol);
        w = ldg_hint(rw + 8 * i, pol);
    }
    __device__ __forceinline__ void advance(int steps) {
        ro += 32 * steps;
        rw += 8 * steps;
    }
};

// Epilogue of one lane for one row group: its block-row r (channels
// 4r..4r+3; r < 0 for none) at tokens m_g + 8 i, i < 8, from acc[4 i + c].
template <int KIND>
__device__ __forceinline__ void store_lane(const LaunchArgs& a, int N, long long m_g, int r, const int (&acc)[32],
                                           float4 sc, float4 bi) {
    if (r < 0) return;
    if (N & 3) {
        store_lane_narrow<KIND, 8>(a, N, m_g, r, acc, sc, bi);
        return;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) store_token<KIND>(a, N, m_g + 8 * i, r, acc + 4 * i, sc, bi);
}

// Block-row q of a row group whose 4 block-rows are packed as 16-bit
// fields (0xffff: none).
__device__ __forceinline__ int block_row16(unsigned long long gr, int q) {
    const int v = static_cast<int>((gr >> (16 * q)) & 0xffffu);
    return v == 0xffff ? -1 : v;
}
__device__ __forceinline__ unsigned long long pack_rows16(int4 gr) {
    auto f = [](int r) { return static_cast<unsigned long long>(r < 0 ? 0xffff : r); };
    return f(gr.x) | f(gr.y) << 16 | f(gr.z) << 32 | f(gr.w) << 48;
}

// Block shapes of the stored weight.  A step's gather gives lane (g, q)
// the dot-4 words of tokens g + 8 i (i < 8) for the 4 columns of quad q;
// what a quad holds differs:
//   kShape4x1: 4 stored 4 x 1 blocks of block-row q (4 columns, 4 output
//     channels each): 32 dp4a against the quad's 4 channel words, 32
//     accumulators a lane (8 tokens x 4 channels);
//   kShape1x4: one 1 x 4 block (one output row x 4 consecutive columns) of
//     the group's row q: 8 dp4a against its one weight word, 8 accumulators
//     a lane (8 tokens x 1 row).
constexpr int kShape4x1 = 0;
constexpr int kShape1x4 = 1;

template <int SHAPE>
struct BlockShape {
    static constexpr int kAcc = 32;
    __device__ static __forceinline__ void dot(const uint32_t (&t)[8], const int4& w, int (&acc)[kAcc]) {
        dot16(t, w, acc);
    }
    // scale and bias of block-row r's 4 channels (r < 0: an unused float4)
    __device__ static __forceinline__ float4 load_sb(const float* p, int r, uint64_t pol) {
        return ldg_hint(reinterpret_cast<const float4*>(p) + max(r, 0), pol);
    }
    template <int KIND>
    __device__ static __forceinline__ void store(const LaunchArgs& a, int N, long long m_g, int r,
                                                 const int (&acc)[kAcc], float4 sc, float4 bi) {
        store_lane<KIND>(a, N, m_g, r, acc, sc, bi);
    }
};

template <>
struct BlockShape<kShape1x4> {
    static constexpr int kAcc = 8;
    __device__ static __forceinline__ void dot(const uint32_t (&t)[8], const int4& w, int (&acc)[kAcc]) {
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = __dp4a(static_cast<int>(t[i]), w.x, acc[i]);
    }
    // scale and bias of row n in .x
    __device__ static __forceinline__ float4 load_sb(const float* p, int n, uint64_t pol) {
        return make_float4(__int_as_float(ldg_hint(reinterpret_cast<const int*>(p) + max(n, 0), pol)), 0.f, 0.f, 0.f);
    }
    // Epilogue of row n at tokens m_g + 8 i: one value a token (no residual kind).
    template <int KIND>
    __device__ static __forceinline__ void store(const LaunchArgs& a, int N, long long m_g, int n,
                                                 const int (&acc)[kAcc], float4 sc, float4 bi) {
        if (n < 0) return;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const long long m = m_g + 8 * i;
            if (m >= a.M) continue;
            const size_t o = static_cast<size_t>(m) * N + n;
            if (KIND == 0) {
                static_cast<int32_t*>(a.out)[o] = acc[i];
            } else if (KIND == 1 || KIND == 2) {
                static_cast<float*>(a.out)[o] = epilogue_value<KIND>(acc[i], sc.x, bi.x);
            } else if (KIND == 3 || KIND == 4) {
                const int q = __float2int_rn(__fmul_rn(epilogue_value<KIND>(acc[i], sc.x, bi.x), a.inv_out_scale));
                static_cast<int8_t*>(a.out)[o] = static_cast<int8_t>(q > 127 ? 127 : (q < -128 ? -128 : q));
            }
        }
    }
};

// MODE: how a window's token tile reaches shared memory.
constexpr int kStageGather = 0;  // per-thread loads from x [M][K], transposed in registers
constexpr int kStageTiles = 1;   // one bulk copy of a tile the relayout kernel wrote
constexpr int kStageTensor = 2;  // tensor copies of x's boxes, transposed in place (transpose_box)
constexpr int kStageKMajor = 3;  // tensor copies of x^T [K][M] boxes, already in the tile's layout

template <int KIND, int MODE, int SHAPE>
__global__ void __launch_bounds__(kThreads, 1)
bsgemm_kernel(DeviceWeights w, LaunchArgs a, const __grid_constant__ Schedule sched,
              const __grid_constant__ CUtensorMap xmap) {
    constexpr bool TMA = MODE == kStageTiles;
    constexpr bool KMAJOR = MODE == kStageKMajor;
    constexpr bool TENSOR = MODE == kStageTensor || KMAJOR;
    using BS = BlockShape<SHAPE>;
    constexpr int NA = BS::kAcc;    // accumulators a lane
    constexpr int SW = 32 * NA;     // slot words: a warp's accumulators
    static_assert(kGroupWin < kThreads, "one thread loads each group of a window");
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int s_gp[kGroupWin + 1];                          // step offsets of the current group window
    __shared__ unsigned long long s_grow[kGroupWin];             // their block-rows (block_row16)
    __shared__ __align__(8) unsigned long long s_bar[kMaxBoxes];  // completion of the tile's copies
    __shared__ int s_wst[kWarps + 1];                            // first step of each warp in the window (relative)

    const int K = w.K, N = w.N;
    const int kpad = (K + 15) & ~15;
    const int nbox = (K + 63) >> 6;  // 64-column boxes of a tile
    const uint32_t sbase = smem_addr(smem);
    const uint32_t tb = (sbase + 511u) & ~511u;  // the token tile, 512-byte aligned (the boxes' 64-byte swizzle)
    unsigned char* tile = smem + (tb - sbase);
    int* slots = reinterpret_cast<int*>(tile + static_cast<size_t>(nbox) * 64 * kTile);
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int q = lane & 3, g = lane >> 2;  // block-row q of each group; tokens g + 8 i
    const uint32_t lb = 16u * static_cast<uint32_t>(lane >> 4);
    const long long ng = w.ngroups;
    const unsigned wlim = a.wait_limit ? a.wait_limit : kWaitLimit;
    const uint64_t pol_w = l2_policy_evict_last(), pol_x = l2_policy_evict_first();

    // the tensor map's descriptor comes into the TMA unit's cache while the
    // CTA sets up, ahead of the first tensor copy
    if (TENSOR && tid == 0) asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(&xmap)) : "memory");
    griddep_launch_dependents();
    const uint32_t bar = smem_addr(&s_bar[0]);  // box b's barrier at bar + 8 b (TMA: box 0 only)
    // A tensor copy brings box_d consecutive 64-column boxes (one barrier
    // each copy); this warp issues copies [op0, op1) and turns their boxes
    // around.
    const int box_d = TENSOR ? a.box_d : 1;  // > 1 exactly when xmap is the 3-D view of x
    const int nops = nbox / box_d;
    if ((TMA || TENSOR) && tid == 0) mbar_init_n(bar, TENSOR ? nops : 1);
    const int op0 = warp * nops / kWarps, op1 = (warp + 1) * nops / kWarps;
    __syncthreads();
    unsigned phase = 0;
    long long u = sched.u[blockIdx.x];
    const long long u_end = sched.u[blockIdx.x + 1];

    long long staged = -1;  // token tile currently in shared memory
    bool waited = false;    // the previous grid has completed and its writes are visible
    auto wait_prev = [&]() {  // before this thread's global writes
        if (!waited) {
            griddep_wait();
            waited = true;
        }
    };
    while (u < u_end) {
        // next window: one token tile, at most kGroupWin consecutive row groups
        const long long t = u / ng;
        const int g_lo = static_cast<int>(u - t * ng);
        const int g_hi = static_cast<int>(min(min(ng, g_lo + (u_end - u)), static_cast<long long>(g_lo + kGroupWin)));
        u += g_hi - g_lo;
        const long long m0 = t * kTile;
        auto gp = [&](int gi) { return s_gp[gi - g_lo]; };

        const bool stage = (t != staged);
        // the token tile (already swizzled in a.xb) in kTmaPiece-byte bulk
        // copies, issued by the lanes of warp 0 (one completion barrier)
        auto copy_tile = [&]() {
            if (a.skip_copy) return;  // test hook: the waits below give up
            if (TENSOR && stage && lane < op1 - op0) {  // lane i of each warp: the warp's copy op0 + i
                const int o = op0 + lane;
                if (staged >= 0) fence_proxy_async();  // the previous tile's reads come first
                mbar_arrive_expect_tx(bar + 8u * o, 64u * kTile * box_d);
                if (KMAJOR)  // rows 64o..64o+63 of x^T at tokens t*64.., landing as the tile's rows
                    tensor_g2s_hint(tb + 4096u * o, &xmap, static_cast<int>(t * kTile), 64 * o, bar + 8u * o, pol_x);
                else if (box_d > 1)  // x viewed as [K/64][M][64]: boxes o*box_d.. of tokens t*64..
                    tensor_g2s_3d_hint(tb + 4096u * box_d * o, &xmap, 0, static_cast<int>(t * kTile), o * box_d,
                                       bar + 8u * o, pol_x);
                else
                    tensor_g2s_hint(tb + 4096u * o, &xmap, 64 * o, static_cast<int>(t * kTile), bar + 8u * o, pol_x);
            }
            if (TMA && stage && warp == 0) {
                const unsigned bytes = static_cast<unsigned>(kpad) * kTile;
                const int8_t* src = a.xb + static_cast<size_t>(t) * kpad * kTile;
                if (staged >= 0) fence_proxy_async();
                if (lane == 0) mbar_arrive_expect_tx(bar, bytes);
                __syncwarp();
                for (unsigned off = static_cast<unsigned>(lane) * kTmaPiece; off < bytes; off += 32u * kTmaPiece)
                    bulk_g2s(tb + off, src + off, min(static_cast<unsigned>(kTmaPiece), bytes - off), bar);
            }
        };
        // The tile's copies go out first: after the first window the previous
        // grid is done, and with act_ready (x complete before the previous
        // kernel started) the first window's copies may start at once too;
        // the window's set-up and the previous kernel's end overlap them.
        const bool issued = waited || (TENSOR && a.act_ready);
        if (issued) copy_tile();
        // The window's step offsets and block-rows (the weights stay in L2:
        // these loads hit it even while the tile's bytes stream in).
        int gp_v = 0;
        unsigned long long gr_v = ~0ull;
        if (tid <= g_hi - g_lo) {
            gp_v = ldg_hint(w.gptr + g_lo + tid, pol_w);
            if (tid < g_hi - g_lo) gr_v = pack_rows16(ldg_hint(w.grow + g_lo + tid, pol_w));
        }
        if (staged < 0) {  // the split-group slots start at zero; whoever finishes a slot resets it
            for (int i = tid; i < kSlots * SW / 4; i += kThreads) reinterpret_cast<int4*>(slots)[i] = make_int4(0, 0, 0, 0);
        }
        if (tid <= g_hi - g_lo) s_gp[tid] = gp_v;     // g_hi - g_lo + 1 <= kGroupWin + 1 entries
        if (tid < g_hi - g_lo) s_grow[tid] = gr_v;    // g_hi - g_lo <= kGroupWin entries
        __syncthreads();  // the group window is visible
        const int sa = gp(g_lo);
        if (tid <= kWarps) {
            // Warps take an even split of the window's cost: a step costs 1,
            // a group's end kGroupEndCost (charged after its last step).
            // Group j of the window starts at cost s_gp[j] - sa + j * kGroupEndCost;
            // warp tid starts at the step where the cost reaches tid / kWarps
            // of the total, or at the next group if that falls on a group's end.
            const int ngw = g_hi - g_lo;
            const long long total = static_cast<long long>(s_gp[ngw] - sa) + static_cast<long long>(ngw) * kGroupEndCost;
            const long long target = total * tid / kWarps;
            int lo = 0, hi = ngw;  // the last group j with its start cost <= target
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (static_cast<long long>(s_gp[mid] - sa) + static_cast<long long>(mid) * kGroupEndCost <= target) lo = mid;
                else hi = mid;
            }
            const long long into = target - (static_cast<long long>(s_gp[lo] - sa) + static_cast<long long>(lo) * kGroupEndCost);
            const int len = s_gp[lo + 1] - s_gp[lo];  // a multiple of kBlock
            const int in_grp = static_cast<int>(into < len ? into : len) / kBlock * kBlock;
            s_wst[tid] = (tid == kWarps) ? s_gp[ngw] - sa : s_gp[lo] - sa + in_grp;
        }
        __syncthreads();  // the warps' step ranges are visible

        const int ws0 = s_wst[warp], ws1 = s_wst[warp + 1];

        // Groups split between warps are finished after the window's last
        // barrier: warp w takes boundary w + 1 if it is the first boundary
        // inside its group (slot w then holds the group's sum).  Its block-row,
        // scale and bias load now.
        int fin_r = -1;
        float4 fin_sc = make_float4(0.f, 0.f, 0.f, 0.f), fin_bi = fin_sc;
        bool fin = false;
        if (warp < kSlots) {
            const int bnd = s_wst[warp + 1];
            const int j = row_of(s_gp, 0, g_hi - g_lo, sa + min(bnd, s_wst[kWarps] - 1));
            const int gs = s_gp[j] - sa;
            fin = bnd > gs && bnd < s_gp[j + 1] - sa && s_wst[warp] <= gs;
            if (fin) {
                fin_r = block_row16(s_grow[j], q);
                if (KIND != 0) {  // needed after the window; no wait here
                    fin_sc = BS::load_sb(w.scale, fin_r, pol_w);
                    fin_bi = BS::load_sb(w.bias, fin_r, pol_w);
                }
            }
        }

        // The warp's first kRing step records load while the tile does; the
        // record of a step is loaded kRing steps before its use (the record
        // array has kStepPad spare steps for the loads past the last one).
        RecPtr rec(w.recs, sa + ws0, lane, q);  // step of ring slot 0
        int off[kRing];
        int4 wq[kRing];
#pragma unroll
        for (int i = 0; i < kRing; ++i) {
            off[i] = 0;
            wq[i] = make_int4(0, 0, 0, 0);
            if (ws0 < ws1) rec.load(i, off[i], wq[i], pol_w);
        }

        // Everything above reads only the weights: in the first window it
        // overlaps the end of the previous kernel.  The activations wait for
        // that kernel's completion -- unless act_ready says they were complete
        // before it began: then only this thread's first global write waits
        // (wait_prev), and the steps overlap that kernel's end.
        if (!waited && !(TENSOR && a.act_ready)) {
            griddep_wait();
            waited = true;
            if (!issued) copy_tile();
        }
        if (MODE == kStageGather && stage) {  // gather the tile with per-thread loads
            stage_tile(tile, a, K, kpad, m0);
            __syncthreads();
            staged = t;
        }

        // Row groups without any stored block: acc = 0.
        for (int gi = g_lo + warp; gi < g_hi; gi += kWarps) {
            if (gp(gi) == gp(gi + 1)) {
                const int r = block_row16(s_grow[gi - g_lo], q);
                int zero[NA];
#pragma unroll
                for (int i = 0; i < NA; ++i) zero[i] = 0;
                wait_prev();
                if (r >= 0)
                    BS::template store<KIND>(a, N, m0 + g, r, zero, BS::load_sb(w.scale, r, pol_w),
                                             BS::load_sb(w.bias, r, pol_w));
            }
        }

        if (TENSOR && stage) {
            // the warp turns its boxes around as they land
            bool ok = true;
            if (KMAJOR) {  // nothing to turn around: every thread sees every box land
                for (int o = 0; o < nops && ok; ++o) ok = __all_sync(0xffffffffu, mbar_wait(bar + 8u * o, phase & 1u, wlim));
            } else {
                for (int o = op0; o < op1 && ok; ++o) {
                    ok = __all_sync(0xffffffffu, mbar_wait(bar + 8u * o, phase & 1u, wlim));
                    for (int j = 0; j < box_d && ok; ++j) transpose_box(tb, o * box_d + j, lane);
                }
            }
            ++phase;
            if (__syncthreads_or(!ok)) {
                if (tid == 0) {
                    wait_prev();
                    atomicOr(w.status, kStatusTimeout);
                    for (int o = 0; o < nops; ++o) mbar_wait(bar + 8u * o, (phase - 1) & 1u, wlim);  // one more chance
                }
                __syncthreads();
                return;
            }
            staged = t;
        }
        if (TMA && stage) {
            const bool ok = mbar_wait(bar, phase & 1u, wlim);
            ++phase;
            if (__syncthreads_or(!ok)) {
                if (tid == 0) {
                    wait_prev();
                    atomicOr(w.status, kStatusTimeout);
                    mbar_wait(bar, (phase - 1) & 1u, wlim);  // give the copy one more bounded chance to land
                }
                __syncthreads();
                return;
            }
            staged = t;
        }

        // one step: the gathers, then the block shape's dot products
        auto bsg_step = [&](int off_i, const int4& w_i, int (&acc_r)[NA]) {
            uint32_t t[8];
            gather16(tb, lb, off_i, t);
            BS::dot(t, w_i, acc_r);
        };
        if (ws0 < ws1) {
            int gi = g_lo + row_of(s_gp, 0, g_hi - g_lo, sa + ws0);
            int p = ws0;  // step index relative to sa
            int blk = 0;  // ring block (slots 4 blk .. 4 blk + 3) holding step p
            while (p < ws1) {
                const int gs = gp(gi), ge = gp(gi + 1);
                const int p_end = min(ws1, ge - sa);
                const int r = block_row16(s_grow[gi - g_lo], q);
                float4 sc = make_float4(0.f, 0.f, 0.f, 0.f), bi = sc;
                if (KIND != 0) {  // used at the group's end: the loads fly during its steps
                    sc = BS::load_sb(w.scale, r, pol_w);
                    bi = BS::load_sb(w.bias, r, pol_w);
                }
                int acc[NA];
#pragma unroll
                for (int i = 0; i < NA; ++i) acc[i] = 0;
                // Steps p .. p_end - 1.  Ring slot i holds step (ring base + i);
                // after its step it loads step (base + kRing + i), and after
                // slot kRing - 1 the base moves on by kRing.  Groups hold a
                // multiple of kBlock steps and warp ranges start at such a
                // multiple, so a group starts and ends at a block boundary:
                // whole rounds run as one straight block of kRing steps (the
                // compiler overlaps one step's gathers with the previous
                // step's dp4a), and a round that a group enters or leaves in
                // the middle runs block by block (kBlock straight steps each).
                while (p < p_end) {
                    if (blk == 0 && p + kRing <= p_end) {
#pragma unroll
                        for (int i = 0; i < kRing; ++i) {
                            bsg_step(off[i], wq[i], acc);
                            rec.load(kRing + i, off[i], wq[i], pol_w);
                        }
                        rec.advance(kRing);
                        p += kRing;
                        continue;
                    }
#define BSG_RING_BLOCK(j)                                                   \
    _Pragma("unroll") for (int i = kBlock * (j); i < kBlock * ((j) + 1); ++i) { \
        bsg_step(off[i], wq[i], acc);                                  \
        rec.load(kRing + i, off[i], wq[i], pol_w);                           \
    }
                    if (blk == 0) {
                        BSG_RING_BLOCK(0)
                        blk = 1;
                    } else if (blk == 1) {
                        BSG_RING_BLOCK(1)
                        blk = 2;
                    } else {
                        BSG_RING_BLOCK(2)
                        rec.advance(kRing);
                        blk = 0;
                    }
#undef BSG_RING_BLOCK
                    p += kBlock;
                }
                if (gs >= sa + ws0 && ge <= sa + ws1) {
                    wait_prev();
                    BS::template store<KIND>(a, N, m0 + g, r, acc, sc, bi);
                } else {
                    // Shared with other warps: add into the slot of the first warp
                    // boundary inside the group (the first b with s_wst[b] > the
                    // group's first step); the group is finished after the window's
                    // barrier.  Slot layout [j][lane]: every warp's lane l holds
                    // the same (token, block-row, channel) in acc[j].
                    int b = 1;
                    while (s_wst[b] <= gs - sa) ++b;
                    int* sl = slots + (b - 1) * SW + lane;
#pragma unroll
                    for (int j = 0; j < NA; ++j) atomicAdd(sl + 32 * j, acc[j]);
                }
                ++gi;
                while (gi < g_hi && gp(gi + 1) == gp(gi)) ++gi;  // skip groups without steps
            }
        }
        __syncthreads();  // every part of every split group is in its slot

        if (fin) {  // the split group of boundary warp + 1 (see above)
            int* sl = slots + warp * SW + lane;
            int acc[NA];
#pragma unroll
            for (int j = 0; j < NA; ++j) {
                acc[j] = sl[32 * j];
                sl[32 * j] = 0;
            }
            wait_prev();
            BS::template store<KIND>(a, N, m0 + g, fin_r, acc, fin_sc, fin_bi);
        }
        if (u < u_end) __syncthreads();  // the window's offsets, the slots' reset and the tile may be reused
    }
}

// Token-tile relayout: x [M][K] -> swizzled tiles (tile t = tokens
// 64t..64t+63, all kpad columns; zero past M or K).  One warp takes one
// unit -- 64 tokens x 32 columns -- at a time, with no block-wide barrier:
//   * lane (g, h) = (lane / 2, lane % 2) loads tokens 4g..4g+3 x columns
//     16h..16h+15 (four 16-byte loads; per load the warp reads 32
//     contiguous bytes of each of 16 rows);
//   * four 4x4 byte transposes turn them into words (4 tokens of one
//     column), written to the warp's staging buffer in shared memory: 32
//     column rows x 16 words, rows with bit 4 set stored at the partner
//     row (bit 0 flipped) so that the two column halves of a store use
//     different banks;
//   * the warp copies the 32 rows out as 16-byte chunks (16 tokens of one
//     column) to their slots of the swizzled tile: 8 lanes fill one
//     128-byte line.
// The next unit's loads are in flight while a unit is transposed.
__global__ void __launch_bounds__(256)
pretile_kernel(const int8_t* __restrict__ x, int M, int K, int kpad, int8_t* __restrict__ xb, long long units,
               int ncb) {
    constexpr int kW = 8;                        // warps per CTA
    __shared__ __align__(16) uint32_t stage[kW][32 * 16];
    griddep_launch_dependents();
    griddep_wait();  // x may be the previous kernel's output
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 1, h = lane & 1;
    uint32_t* st = stage[warp];
    const bool vec16 = ((K & 15) == 0) && ((reinterpret_cast<uintptr_t>(x) & 15) == 0);
    const long long nw = static_cast<long long>(gridDim.x) * kW;

    // rw[i][j] = bytes of token 4g+i at columns k0+16h+4j .. +3 of unit u (zero past M or K)
    auto load_unit = [&](long long u, uint32_t (&rw)[4][4]) {
        const long long t = u / ncb;
        const int k = static_cast<int>(u % ncb) * 32 + 16 * h;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const long long m = t * kTile + 4 * g + i;
            rw[i][0] = rw[i][1] = rw[i][2] = rw[i][3] = 0u;
            if (m < M && k < K) {
                const int8_t* src = x + static_cast<size_t>(m) * K + k;
                if (vec16) {
                    const uint4 v = __ldg(reinterpret_cast<const uint4*>(src));
                    rw[i][0] = v.x; rw[i][1] = v.y; rw[i][2] = v.z; rw[i][3] = v.w;
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (k + e < K) rw[i][e >> 2] |= static_cast<uint32_t>(static_cast<uint8_t>(src[e])) << (8 * (e & 3));
                }
            }
        }
    };

    long long u = static_cast<long long>(blockIdx.x) * kW + warp;
    uint32_t rw[4][4];
    if (u < units) load_unit(u, rw);
    for (; u < units; u += nw) {
        const long long t = u / ncb;
        const int k0 = static_cast<int>(u % ncb) * 32;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            uint32_t w4[4];
            transpose4(rw[0][j], rw[1][j], rw[2][j], rw[3][j], w4[0], w4[1], w4[2], w4[3]);
#pragma unroll
            for (int e = 0; e < 4; ++e) st[(16 * h + 4 * j + (e ^ h)) * 16 + g] = w4[e];
        }
        if (u + nw < units) load_unit(u + nw, rw);  // the next unit's loads fly while this one is stored
        __syncwarp();
        int8_t* dst = xb + static_cast<size_t>(t) * kpad * kTile;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
            const int ch = lane + 32 * qq;
            const int row = ch >> 2, c = ch & 3;
            const int k = k0 + row;
            if (k < kpad) {
                const uint4 v = *reinterpret_cast<const uint4*>(st + (row ^ (row >> 4)) * 16 + 4 * c);
                *reinterpret_cast<uint4*>(dst + (row_off(k) ^ (static_cast<uint32_t>(c) << 4))) = v;
            }
        }
        __syncwarp();
    }
}

template <int MODE, int SHAPE>
const void* kernel_for(int kind) {
    switch (kind) {
    case 0: return reinterpret_cast<const void*>(&bsgemm_kernel<0, MODE, SHAPE>);
    case 1: return reinterpret_cast<const void*>(&bsgemm_kernel<1, MODE, SHAPE>);
    case 2: return reinterpret_cast<const void*>(&bsgemm_kernel<2, MODE, SHAPE>);
    case 3: return reinterpret_cast<const void*>(&bsgemm_kernel<3, MODE, SHAPE>);
    case 4: return reinterpret_cast<const void*>(&bsgemm_kernel<4, MODE, SHAPE>);
    default: return SHAPE == kShape4x1 ? reinterpret_cast<const void*>(&bsgemm_kernel<5, MODE, kShape4x1>) : nullptr;
    }
}
template <int SHAPE>
const void* kernel_for_mode(int kind, int mode) {
    switch (mode) {
    case kStageKMajor: return kernel_for<kStageKMajor, SHAPE>(kind);
    case kStageTensor: return kernel_for<kStageTensor, SHAPE>(kind);
    case kStageTiles: return kernel_for<kStageTiles, SHAPE>(kind);
    default: return kernel_for<kStageGather, SHAPE>(kind);
    }
}
// The layer kernel for an epilogue kind, staging mode and block shape (NULL
// for the residual kind with 1 x 4 blocks, which is not built).
const void* kernel_for(int kind, int mode, int shape) {
    return shape == kShape1x4 ? kernel_for_mode<kShape1x4>(kind, mode) : kernel_for_mode<kShape4x1>(kind, mode);
}

// cuTensorMapEncodeTiled from the driver, looked up once.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

}  // namespace

bool tensor_staging(int K, const void* x) {
    return K % 16 == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0 && (K + 63) / 64 <= kMaxBoxes &&
           tensor_map_encoder() != nullptr;
}

size_t smem_bytes(int K) {
    const size_t tpad = (static_cast<size_t>(K) + 63) & ~static_cast<size_t>(63);
    // 512 bytes of slack to align the tile, the tile (whole 64-column boxes),
    // the split-group slots
    return 512 + tpad * kTile + static_cast<size_t>(kSlots) * kTile * 16 * sizeof(int);
}

int max_k() {
    int k = 16;
    while (smem_bytes(k + 16) + kStaticSmem <= static_cast<size_t>(kSmemOptin)) k += 16;
    return k;
}

cudaError_t prepare_kernels(int K, int* ctas_per_sm) {
    const int smem = static_cast<int>(smem_bytes(K));
    for (int shape = 0; shape < 2; ++shape) {
        for (int kind = 0; kind < 6; ++kind) {
            for (int mode = 0; mode < 4; ++mode) {
                const void* k = kernel_for(kind, mode, shape);
                if (!k) continue;
                cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                     kSmemOptin - kStaticSmem);
                if (e != cudaSuccess) return e;
            }
        }
    }
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas_per_sm, kernel_for(0, kStageTensor, kShape4x1), kThreads,
                                                         smem);
}

cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a_in, const Schedule& sched, int grid, cudaStream_t s) {
    LaunchArgs a = a_in;
    a.box_d = 1;
    const size_t smem = smem_bytes(w.K);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // a.tensor: a tensor map over x [M][K] (int8, 64 x 64 boxes, 64-byte
    // swizzle, zeros outside M x K); otherwise an unused all-zero map
    CUtensorMap xmap;
    std::memset(&xmap, 0, sizeof(xmap));
    if (a.kmajor) {
        // x^T [K][M] (row stride a.ld bytes): 64 tokens x 64 rows a box; its
        // 64-byte swizzle is the tile's layout (tile_row_offset)
        PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
        if (!encode || (w.K + 63) / 64 > kMaxBoxes) return cudaErrorNotSupported;
        const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(a.M), static_cast<cuuint64_t>(w.K)};
        const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(a.ld)};
        const cuuint32_t box[2] = {static_cast<cuuint32_t>(kTile), 64u};
        const cuuint32_t estride[2] = {1u, 1u};
        if (encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t*>(a.x), gdim, gstride, box, estride,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    } else if (a.tensor) {
        PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
        const int nbox = (w.K + 63) / 64;
        if (!encode || nbox > kMaxBoxes) return cudaErrorNotSupported;
        // box_d: the largest divisor of nbox that leaves at least kMinCopies
        // copies (1: the 2-D boxes below)
        int d = 1;
        for (int c = 2; c <= nbox / kMinCopies; ++c)
            if (nbox % c == 0) d = c;
        if (w.K % 64 == 0 && d > 1) {  // box_d > 1 <=> the 3-D map (and copy)
            // x viewed as [K/64 blocks][M tokens][64 columns] (the block
            // stride is 64 bytes), boxes of box_d blocks x 64 tokens x 64
            // columns: the 64-byte rows land as the 2-D boxes below would, box
            // after box.  The tensor-copy unit takes and completes copies one
            // by one, so 8 large copies (one a warp) finish a tile sooner
            // than 48 small ones.
            a.box_d = d;
            const cuuint64_t gdim[3] = {64u, static_cast<cuuint64_t>(a.M), static_cast<cuuint64_t>(nbox)};
            const cuuint64_t gstride[2] = {static_cast<cuuint64_t>(w.K), 64u};
            const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(kTile), static_cast<cuuint32_t>(a.box_d)};
            const cuuint32_t estride[3] = {1u, 1u, 1u};
            if (encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<int8_t*>(a.x), gdim, gstride, box, estride,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                       CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        } else {
            const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(w.K), static_cast<cuuint64_t>(a.M)};
            const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(w.K)};
            const cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(kTile)};
            const cuuint32_t estride[2] = {1u, 1u};
            if (encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t*>(a.x), gdim, gstride, box, estride,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                       CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        }
    }
    cudaError_t e = cudaSuccess;
#define BSG_LAUNCH(KV, SH)                                                                               \
    do {                                                                                                 \
        if (a.kmajor)                                                                                    \
            e = cudaLaunchKernelEx(&cfg, bsgemm_kernel<KV, kStageKMajor, SH>, w, a, sched, xmap);        \
        else if (a.tensor)                                                                               \
            e = cudaLaunchKernelEx(&cfg, bsgemm_kernel<KV, kStageTensor, SH>, w, a, sched, xmap);        \
        else if (a.xb)                                                                                   \
            e = cudaLaunchKernelEx(&cfg, bsgemm_kernel<KV, kStageTiles, SH>, w, a, sched, xmap);         \
        else                                                                                             \
            e = cudaLaunchKernelEx(&cfg, bsgemm_kernel<KV, kStageGather, SH>, w, a, sched, xmap);        \
    } while (0)
#define BSG_LAUNCH_KIND(KV)                       \
    do {                                          \
        if (a.shape == kShape1x4)                 \
            BSG_LAUNCH(KV, kShape1x4);            \
        else                                      \
            BSG_LAUNCH(KV, kShape4x1);            \
    } while (0)
    switch (a.kind) {
    case 0: BSG_LAUNCH_KIND(0); break;
    case 1: BSG_LAUNCH_KIND(1); break;
    case 2: BSG_LAUNCH_KIND(2); break;
    case 3: BSG_LAUNCH_KIND(3); break;
    case 4: BSG_LAUNCH_KIND(4); break;
    default:
        if (a.shape == kShape1x4) return cudaErrorNotSupported;
        BSG_LAUNCH(5, kShape4x1);
        break;
    }
#undef BSG_LAUNCH_KIND
#undef BSG_LAUNCH
    return e != cudaSuccess ? e : cudaGetLastError();
}

// LayerNorm of each row of z [M][N] fp32 (the post-operator the optimized
// INT8 graph fuses after the output projection and FFN2, Sec. 3 "Graph
// optimization"): one warp a row, fp32 throughout (GB300's fp64 rate is a
// small fraction of its fp32 rate).  The mean is the row's first value c
// plus the mean of (z - c) -- summing deviations from a value of the row
// keeps the rounding small when the mean is large against the spread --
// then the variance from the centred squares; out = fmaf((z - mean) *
// rstd, gamma, beta), fp32 or requantised to int8 (kind 3: fp32 multiply
// by 1 / out_scale, round half even, saturate).  With N % 4 == 0 and
// 16-byte aligned arrays the row moves as float4 (and 4-byte int8 words),
// and for N <= 1024 it is read once into registers for all three passes.
// Launched with programmatic dependent launch: z is read after the
// previous kernel completes.
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ void ln_store(int kind, void* out, long long idx, float v, float inv) {
    if (kind == 3) {
        const int q = __float2int_rn(__fmul_rn(v, inv));
        static_cast<int8_t*>(out)[idx] = static_cast<int8_t>(q > 127 ? 127 : (q < -128 ? -128 : q));
    } else {
        static_cast<float*>(out)[idx] = v;
    }
}

constexpr int kLnVec = 8;  // float4s a lane keeps in registers: rows of N <= 1024 take one read

__global__ void __launch_bounds__(256)
layernorm_kernel(const float* __restrict__ z, int M, int N, const float* __restrict__ gamma,
                 const float* __restrict__ beta, float eps, int kind, float inv_out_scale, void* __restrict__ out) {
    griddep_launch_dependents();
    const int lane = threadIdx.x & 31;
    const long long m = static_cast<long long>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (m >= M) return;
    griddep_wait();  // z is the previous kernel's output
    const float* row = z + m * N;
    const bool vec = (N & 3) == 0 && (reinterpret_cast<uintptr_t>(z) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(gamma) & 15) == 0 && (reinterpret_cast<uintptr_t>(beta) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(out) & 15) == 0;
    if (vec && N <= 128 * kLnVec) {
        // the row in registers (lane l: float4s l, l + 32, ...), read once;
        // the same operations in the same order as the loops below
        float4 v[kLnVec];
#pragma unroll
        for (int i = 0; i < kLnVec; ++i) {
            const int n = 4 * lane + 128 * i;
            v[i] = n < N ? __ldg(reinterpret_cast<const float4*>(row + n)) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        const float c = __shfl_sync(0xffffffffu, v[0].x, 0);
        float s1 = 0.0f;
#pragma unroll
        for (int i = 0; i < kLnVec; ++i)
            if (4 * lane + 128 * i < N) s1 += ((v[i].x - c) + (v[i].y - c)) + ((v[i].z - c) + (v[i].w - c));
        const float mean = c + warp_sum(s1) / N;
        float s2 = 0.0f;
#pragma unroll
        for (int i = 0; i < kLnVec; ++i) {
            if (4 * lane + 128 * i < N) {
                const float a = v[i].x - mean, b = v[i].y - mean, d = v[i].z - mean, e = v[i].w - mean;
                s2 += (a * a + b * b) + (d * d + e * e);
            }
        }
        const float rstd = rsqrtf(warp_sum(s2) / N + eps);
        const long long base = m * N;
#pragma unroll
        for (int i = 0; i < kLnVec; ++i) {
            const int n = 4 * lane + 128 * i;
            if (n >= N) continue;
            const float4 g = __ldg(reinterpret_cast<const float4*>(gamma + n));
            const float4 b = __ldg(reinterpret_cast<const float4*>(beta + n));
            const float y0 = __fmaf_rn((v[i].x - mean) * rstd, g.x, b.x), y1 = __fmaf_rn((v[i].y - mean) * rstd, g.y, b.y);
            const float y2 = __fmaf_rn((v[i].z - mean) * rstd, g.z, b.z), y3 = __fmaf_rn((v[i].w - mean) * rstd, g.w, b.w);
            if (kind == 3)
                *reinterpret_cast<uint32_t*>(static_cast<int8_t*>(out) + base + n) = requant4_s8(y0, y1, y2, y3, inv_out_scale);
            else
                *reinterpret_cast<float4*>(static_cast<float*>(out) + base + n) = make_float4(y0, y1, y2, y3);
        }
        return;
    }
    const float c = __ldg(row);
    float s1 = 0.0f;
    if (vec) {
        for (int n = 4 * lane; n < N; n += 128) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(row + n));
            s1 += ((v.x - c) + (v.y - c)) + ((v.z - c) + (v.w - c));
        }
    } else {
        for (int n = lane; n < N; n += 32) s1 += __ldg(row + n) - c;
    }
    const float mean = c + warp_sum(s1) / N;
    float s2 = 0.0f;
    if (vec) {
        for (int n = 4 * lane; n < N; n += 128) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(row + n));
            const float a = v.x - mean, b = v.y - mean, d = v.z - mean, e = v.w - mean;
            s2 += (a * a + b * b) + (d * d + e * e);
        }
    } else {
        for (int n = lane; n < N; n += 32) {
            const float a = __ldg(row + n) - mean;
            s2 += a * a;
        }
    }
    const float rstd = rsqrtf(warp_sum(s2) / N + eps);
    const long long base = m * N;
    if (vec) {
        for (int n = 4 * lane; n < N; n += 128) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(row + n));
            const float4 g = __ldg(reinterpret_cast<const float4*>(gamma + n));
            const float4 b = __ldg(reinterpret_cast<const float4*>(beta + n));
            const float y0 = __fmaf_rn((v.x - mean) * rstd, g.x, b.x), y1 = __fmaf_rn((v.y - mean) * rstd, g.y, b.y);
            const float y2 = __fmaf_rn((v.z - mean) * rstd, g.z, b.z), y3 = __fmaf_rn((v.w - mean) * rstd, g.w, b.w);
            if (kind == 3) {
                *reinterpret_cast<uint32_t*>(static_cast<int8_t*>(out) + base + n) =
                    requant4_s8(y0, y1, y2, y3, inv_out_scale);
            } else {
                *reinterpret_cast<float4*>(static_cast<float*>(out) + base + n) = make_float4(y0, y1, y2, y3);
            }
        }
    } else {
        for (int n = lane; n < N; n += 32)
            ln_store(kind, out, base + n, __fmaf_rn((__ldg(row + n) - mean) * rstd, __ldg(gamma + n), __ldg(beta + n)),
                     inv_out_scale);
    }
}

cudaError_t launch_layernorm(const float* z, int M, int N, const float* gamma, const float* beta, float eps, int kind,
                             float inv_out_scale, void* out, cudaStream_t s) {
    const int rows_per_block = 8;
    const unsigned grid = static_cast<unsigned>((static_cast<long long>(M) + rows_per_block - 1) / rows_per_block);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(32 * rows_per_block);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // its set-up overlaps the previous kernel's end
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, layernorm_kernel, z, M, N, gamma, beta, eps, kind, inv_out_scale, out);
    return e != cudaSuccess ? e : cudaGetLastError();
}

size_t tiled_bytes(int K, long long M) {
    const size_t kpad = (static_cast<size_t>(K) + 15) & ~static_cast<size_t>(15);
    return static_cast<size_t>((M + kTile - 1) / kTile) * kpad * kTile;
}

cudaError_t launch_pretile(const int8_t* x, int M, int K, int8_t* xb, int sms, cudaStream_t s) {
    const int kpad = (K + 15) & ~15;
    const int ncb = (kpad + 31) / 32;  // units of 32 columns per token tile
    const long long units = (static_cast<long long>(M) + kTile - 1) / kTile * ncb;
    const long long cap = 8LL * (sms > 0 ? sms : 1);  // 8 resident CTAs of 8 warps per SM
    const long long want = (units + 7) / 8;
    const unsigned grid = static_cast<unsigned>(want < cap ? want : cap);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, pretile_kernel, x, M, K, kpad, xb, units, ncb);
    return e != cudaSuccess ? e : cudaGetLastError();
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
