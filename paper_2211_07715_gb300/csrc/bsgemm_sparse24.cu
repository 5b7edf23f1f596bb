// Weights with 2:4 structured sparsity along K on the sparse tensor cores.
//
// A 2:4 weight (two values in every group of 4 consecutive input columns of
// a row; Sec. 1 cites the pattern as the one sparse tensor cores take) is a
// dense contraction of its stored half, so here it runs on the
// fifth-generation tensor cores' sparse MMA (`tcgen05.mma.sp ... kind::f16`):
// out^T = W x^T with the weight as the sparse A operand (M = 128 output
// channels a tile, its stored values as f16 plus 2-bit positions) and the
// token tile as the dense B operand (N = 128 tokens).  int8 values are exact
// in f16 and their products (|v x| <= 127 * 128) exact in fp32; every
// partial sum of at most 1024 products stays below 2^24, so each chunk of
// 2048 input columns (1024 stored values a row) accumulates exactly in its
// own fp32 accumulator in tensor memory, and the chunks are added in int32
// by the epilogue: the int32 result of the definition, bit for bit.
//
// Per CTA (128 channels x 128 tokens, all of K in stages of 128 columns):
//   * the create step lays out every (channel tile, stage) of the weight as
//     the 16 KB shared-memory image of its stored values (128 rows of 64 f16,
//     the 128-byte swizzle) and the stage's 4 x 128 metadata words (one
//     tensor-memory column per MMA); one thread of the MMA warp brings the
//     images in by bulk copies, three stages ahead (a ring of four);
//   * the 8 converter warps (two threads a token row, one per 64 columns)
//     copy the stage's int8 activations with cp.async two stages ahead (a
//     ring of three int8 tiles), widen them to f16 into
//     the B image (two 128-row x 64-column sub-tiles, 128-byte swizzle), and
//     store the stage's metadata into tensor memory (warps 0-3: lane r =
//     weight row r);
//   * one thread of the MMA warp issues the stage's 4 MMAs (K = 32 each)
//     into the chunk's accumulator (tensor-memory columns 0-127 and
//     128-255) and commits them to the stage's "empty" barrier; two stages
//     are in flight; each MMA's metadata column sits on a 32-column boundary
//     (columns 256 + 32 j);
//   * the epilogue (the converter warps again; lane m = channel m of the
//     tile, warps w and w + 4 the two halves of the tokens): the chunks'
//     accumulators read from tensor memory 32 tokens at a time, converted to int32 exactly, added, and the fused epilogue
//     (dequantise + bias, GELU, requantise) stored as out[token][channel].
// Every wait is bounded; a wait that gives up sets the handle's status word.
//
// The same kernel with DENSE set runs any int8 weight, stored in full, on
// the dense MMA (`tcgen05.mma ... kind::f16`, K = 16): every block-sparse
// weight taken as dense over K, the tensor-core form of Algorithm 1's
// contraction that skips no zero block.  A stage's weight image is then
// 32 KB (128 rows x 128 f16 as two 64-column sub-tiles, the B image's
// layout; a ring of three, loaded two stages ahead), its 8 MMAs read no
// metadata, and a chunk of exactly-accumulated columns is 1024 (8 stages:
// at most 1024 products below 2^14 in magnitude each), four chunks for K =
// 4096 filling the 512 tensor-memory columns.

#include <cstdint>
#include <cuda_runtime.h>

#include "bsgemm.h"
#include "bsgemm_device.cuh"
#include "bsgemm_internal.h"
#include "bsgemm_tcgen05.cuh"

namespace bsg {
namespace {

constexpr int kTcThreads = 288;            // 8 converter / epilogue warps + 1 MMA warp
constexpr uint32_t kXImg = 128 * 128;      // a stage's int8 token tile (128 tokens x 128 columns)
constexpr uint32_t kBImg = 2 * 128 * 128;  // its f16 form: two 128 x 64 sub-tiles
constexpr int kXRing = 3;                  // int8 token tiles in flight (copied two stages ahead)
// bytes of a stage's weight image; weight images in flight (the sparse
// form loads three stages ahead, the dense form two); stages of one exact
// fp32 accumulator chunk
__host__ __device__ constexpr uint32_t a_img_bytes(bool dense) { return dense ? kBImg : kTc24AImage; }
__host__ __device__ constexpr int a_ring(bool dense) { return dense ? 3 : 4; }
__host__ __device__ constexpr int chunk_stages(bool dense) { return dense ? 8 : 16; }
// shared memory: the weight-image ring, the two f16 token images, the int8 ring
__host__ __device__ constexpr uint32_t b_off(bool dense) { return a_ring(dense) * a_img_bytes(dense); }
__host__ __device__ constexpr uint32_t x_off(bool dense) { return b_off(dense) + 2 * kBImg; }
__host__ __device__ constexpr uint32_t smem_bytes(bool dense) { return x_off(dense) + kXRing * kXImg; }
static_assert(smem_bytes(true) + 1024 <= 227 * 1024 && smem_bytes(false) + 1024 <= 227 * 1024, "shared memory");
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColMeta = 256;         // metadata of MMA i of stage buffer b at column 256 + 32 (4 b + i)

// Instruction descriptors: f16 A and B, fp32 accumulator, both K-major,
// N = 128, M = 128; the sparse MMA's with the sparsity flag (bit 2).
constexpr uint32_t kIdesc = f16_idesc(128, 128, false);
constexpr uint32_t kIdescSp = kIdesc | (1u << 2);

__device__ __forceinline__ void mma_sp(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t meta, uint32_t acc) {
    asm volatile("{\n .reg .pred p;\n setp.ne.u32 p, %5, 0;\n"
                 " tcgen05.mma.sp.cta_group::1.kind::f16 [%0], %1, %2, [%3], %4, p;\n}\n"
                 ::"r"(d), "l"(adesc), "l"(bdesc), "r"(meta), "r"(kIdescSp), "r"(acc) : "memory");
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }
__device__ __forceinline__ void arrive(uint32_t bar) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(bar) : "memory");
}
// Two int8 values (bytes sel of u = w ^ 0x80808080) as an exact f16 pair:
// 0x64uu is the f16 1024 + uu, minus 1152 = the value.
__device__ __forceinline__ uint32_t s8x2_f16x2(uint32_t u, uint32_t sel) {
    const uint32_t b = __byte_perm(u, 0x64646464u, sel);
    uint32_t r;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(b), "r"(0x64806480u));
    return r;
}

template <int KIND, bool DENSE>
__global__ void __launch_bounds__(kTcThreads, 1)
sparse24_kernel(const int8_t* __restrict__ x, int M, int N, int K, const unsigned char* __restrict__ aimg,
                const uint32_t* __restrict__ meta, const float* __restrict__ scale, const float* __restrict__ bias,
                void* __restrict__ out, float inv_out_scale, int act_ready, unsigned wait_limit, int* status) {
    constexpr uint32_t kAImg = a_img_bytes(DENSE);
    constexpr int kARing = a_ring(DENSE), kChunk = chunk_stages(DENSE);
    extern __shared__ unsigned char smem_raw[];
    unsigned char* sm =
        reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    __shared__ __align__(8) unsigned long long s_bar[9];  // a_full[4], b_full[2], empty[2], done
    __shared__ uint32_t s_tmem;
    const int tid = threadIdx.x, warp = tid >> 5;
    const bool mma_warp = warp == 8;
    const int ct = blockIdx.x;                    // channel tile
    const long long t0 = static_cast<long long>(blockIdx.y) * 128;  // first token
    const int nst = K / 128;                      // stages
    const uint32_t bar = smem_addr(&s_bar[0]);
    const uint32_t a_full = bar, b_full = bar + 32, empty = bar + 48, done = bar + 64;
    auto a_base = [&](int s) { return sm + static_cast<uint32_t>(s % kARing) * kAImg; };
    auto b_base = [&](int s) { return sm + b_off(DENSE) + static_cast<uint32_t>(s & 1) * kBImg; };
    auto x_base = [&](int s) { return sm + x_off(DENSE) + static_cast<uint32_t>(s % kXRing) * kXImg; };

    griddep_launch_dependents();
    if (tid == kTcThreads - 32) {
        for (int i = 0; i < kARing; ++i) mbar_init(a_full + 8u * i, 1);
        mbar_init(b_full, 256);
        mbar_init(b_full + 8, 256);
        mbar_init(empty, 1);
        mbar_init(empty + 8, 1);
        mbar_init(done, 1);
    }
    if (mma_warp) tmem_alloc(smem_addr(&s_tmem), kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;
    bool ok = true;

    if (mma_warp) {
        if (tid == kTcThreads - 32) {
            // the weight images of the first kARing stages, then stage s +
            // kARing - 1's once stage s - 1's MMAs (issued before stage s's)
            // have read its ring slot
            auto load_a = [&](int s) {
                const uint32_t slot = static_cast<uint32_t>(s % kARing);
                mbar_arrive_expect_tx(a_full + 8u * slot, kAImg);
#pragma unroll
                for (uint32_t o = 0; o < kAImg; o += 16384u)  // copies of 16 KB
                    bulk_g2s(smem_addr(a_base(s)) + o, aimg + (static_cast<size_t>(ct) * nst + s) * kAImg + o, 16384u,
                             a_full + 8u * slot);
            };
            for (int s = 0; s < kARing && s < nst; ++s) load_a(s);
            for (int s = 0; s < nst; ++s) {
                const uint32_t b = static_cast<uint32_t>(s & 1), ph = static_cast<uint32_t>(s >> 1) & 1u;
                ok &= mbar_wait(a_full + 8u * static_cast<uint32_t>(s % kARing), static_cast<uint32_t>(s / kARing) & 1u,
                                wait_limit);
                ok &= mbar_wait(b_full + 8u * b, ph, wait_limit);
                tc_fence_after();
                const uint32_t as = smem_addr(a_base(s)), bs = smem_addr(b_base(s));
                const uint32_t d = tm + 128u * static_cast<uint32_t>(s / kChunk);  // the chunk's accumulator
                if (DENSE) {
                    // MMA i: columns 16 i .. 16 i + 15 of the stage, in sub-tile i / 4 of both images
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const uint32_t off = 16384u * static_cast<uint32_t>(i >> 2) + 32u * static_cast<uint32_t>(i & 3);
                        mma_f16_ss(d, sw128_desc(as + off, 16, 1024), sw128_desc(bs + off, 16, 1024), kIdesc,
                                   (s % kChunk != 0 || i > 0) ? 1u : 0u);
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        mma_sp(d, sw128_desc(as + 32u * i, 16, 1024),
                               sw128_desc(bs + 16384u * (i >> 1) + 64u * (i & 1), 16, 1024),
                               tm + kColMeta + 32u * (4u * b + static_cast<uint32_t>(i)), (s % kChunk != 0 || i > 0) ? 1u : 0u);
                }
                tc_commit(empty + 8u * b);
                if (s >= 1 && s + kARing - 1 < nst) {
                    ok &= mbar_wait(empty + 8u * (b ^ 1u), static_cast<uint32_t>((s - 1) >> 1) & 1u, wait_limit);
                    tc_fence_after();
                    load_a(s + kARing - 1);
                }
            }
            tc_commit(done);
        }
        __syncwarp();
    } else {
        // converter warps: thread tid takes token row r = tid % 128 of the tile
        // and its columns 64 h .. 64 h + 63 of each stage, h = tid / 128 (f16
        // sub-tile h of the B image)
        const int r = tid & 127, h = tid >> 7;
        if (!act_ready) griddep_wait();
        const long long tok = t0 + r;
        const int8_t* xrow = x + (tok < M ? tok : 0) * static_cast<long long>(K) + 64 * h;
        const uint32_t src_bytes = tok < M ? 16u : 0u;
        // 4 copies of 16 bytes: chunk c (= 4 h + cc) of row r at r * 128 + (c ^
        // (r % 8)) * 16 (conflict-free reads by 8 consecutive threads)
        auto copy_x = [&](int s) {
            const uint32_t xs = smem_addr(x_base(s)) + 128u * static_cast<uint32_t>(r);
#pragma unroll
            for (int cc = 0; cc < 4; ++cc)
                cp_async16(xs + ((static_cast<uint32_t>(4 * h + cc) ^ (r & 7)) << 4), xrow + 128 * s + 16 * cc, src_bytes);
            cp_async_commit();
        };
        copy_x(0);
        if (nst > 1) copy_x(1);
        // the metadata words of this lane (warps 0-3: lane r = weight row r), a stage ahead
        auto load_meta = [&](int s) {
            return !DENSE && h == 0 ? __ldg(reinterpret_cast<const uint4*>(meta + ((static_cast<size_t>(ct) * nst + s) * 128 + r) * 4))
                          : make_uint4(0u, 0u, 0u, 0u);
        };
        uint4 mv = load_meta(0);
        for (int s = 0; s < nst; ++s) {
            const uint32_t b = static_cast<uint32_t>(s & 1);
            // stage s's copies landed (groups are committed in stage order; the
            // ring slot of stage s + 2 was last read by this thread for stage s - 1)
            if (s + 2 < nst) {
                copy_x(s + 2);
                cp_async_wait<2>();
            } else if (s + 1 < nst) {
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            if (s >= 2) {  // stage s - 2's MMAs have read this buffer's B image and metadata
                ok &= mbar_wait(empty + 8u * b, static_cast<uint32_t>((s - 2) >> 1) & 1u, wait_limit);
                tc_fence_after();
            }
            const unsigned char* xs = x_base(s) + 128u * static_cast<uint32_t>(r);
            unsigned char* row = b_base(s) + 16384u * static_cast<uint32_t>(h) + 128u * static_cast<uint32_t>(r);
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
                const int c = 4 * h + cc;
                const int4 v = *reinterpret_cast<const int4*>(xs + ((static_cast<uint32_t>(c) ^ (r & 7)) << 4));
                const uint32_t w[4] = {static_cast<uint32_t>(v.x) ^ 0x80808080u, static_cast<uint32_t>(v.y) ^ 0x80808080u,
                                       static_cast<uint32_t>(v.z) ^ 0x80808080u, static_cast<uint32_t>(v.w) ^ 0x80808080u};
                uint32_t o[8];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    o[2 * q] = s8x2_f16x2(w[q], 0x4140u);
                    o[2 * q + 1] = s8x2_f16x2(w[q], 0x4342u);
                }
                // columns 16 c .. + 15 = f16 chunks 2 cc, 2 cc + 1 of the row of sub-tile h, swizzled
                const uint32_t c0 = static_cast<uint32_t>(2 * cc), c1 = c0 + 1;
                *reinterpret_cast<uint4*>(row + ((c0 ^ (r & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
                *reinterpret_cast<uint4*>(row + ((c1 ^ (r & 7)) << 4)) = make_uint4(o[4], o[5], o[6], o[7]);
            }
            fence_proxy_async();  // the B image, for the tensor cores
            if (!DENSE && h == 0) {
                // the stage's metadata: word r of each of its 4 MMAs into lane r, one
                // column each (32-column aligned)
                const uint32_t mw[4] = {mv.x, mv.y, mv.z, mv.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};\n"
                                 ::"r"(tm + (static_cast<uint32_t>(32 * warp) << 16) + kColMeta + 32u * (4u * b + i)),
                                   "r"(mw[i])
                                 : "memory");
                tmem_wait_st();
            }
            tc_fence_before();
            arrive(b_full + 8u * b);
            if (s + 1 < nst) mv = load_meta(s + 1);
        }

        // epilogue: lane r = channel ch of the tile, tokens 64 h .. 64 h + 63
        ok &= mbar_wait(done, 0, wait_limit);
        __syncwarp();
        tc_fence_after();
        const int ch = ct * 128 + r;
        const float sc = scale[ch], bi = bias[ch];
        const int nchunks = (nst + kChunk - 1) / kChunk;
        griddep_wait();  // outputs after the preceding kernel
        for (int n0 = 64 * h; n0 < 64 * h + 64; n0 += 32) {
            int acc[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) acc[j] = 0;
            for (int c = 0; c < nchunks; ++c) {
                uint32_t v[32];
                tmem_ld32(tm + (static_cast<uint32_t>(32 * (warp & 3)) << 16) + 128u * static_cast<uint32_t>(c) +
                              static_cast<uint32_t>(n0), v);
                tmem_wait_ld(v);
#pragma unroll
                for (int j = 0; j < 32; ++j) acc[j] += __float2int_rn(__uint_as_float(v[j]));  // an exact integer
            }
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const long long t = t0 + n0 + j;
                if (t >= M) break;
                const size_t o = static_cast<size_t>(t) * N + ch;
                if (KIND == 0) {
                    static_cast<int32_t*>(out)[o] = acc[j];
                } else if (KIND == 1 || KIND == 2) {
                    static_cast<float*>(out)[o] = epilogue_value<KIND>(acc[j], sc, bi);
                } else {
                    const int qv = __float2int_rn(__fmul_rn(epilogue_value<KIND>(acc[j], sc, bi), inv_out_scale));
                    static_cast<int8_t*>(out)[o] = static_cast<int8_t>(qv > 127 ? 127 : (qv < -128 ? -128 : qv));
                }
            }
        }
    }
    if (!ok) {
        griddep_wait();
        atomicOr(status, kStatusTimeout);
    }
    tc_fence_before();
    __syncthreads();
    if (mma_warp) tmem_dealloc(tm, kTmemCols);
}

}  // namespace

cudaError_t launch_tc_linear(const int8_t* x, int M, int N, int K, const unsigned char* aimg, const uint32_t* meta,
                             bool dense, const float* scale, const float* bias, void* out, int kind,
                             float inv_out_scale, bool act_ready, int* status, cudaStream_t s) {
    const void* fn = nullptr;
    switch (kind + (dense ? 8 : 0)) {
    case 0: fn = reinterpret_cast<const void*>(&sparse24_kernel<0, false>); break;
    case 1: fn = reinterpret_cast<const void*>(&sparse24_kernel<1, false>); break;
    case 2: fn = reinterpret_cast<const void*>(&sparse24_kernel<2, false>); break;
    case 3: fn = reinterpret_cast<const void*>(&sparse24_kernel<3, false>); break;
    case 4: fn = reinterpret_cast<const void*>(&sparse24_kernel<4, false>); break;
    case 8: fn = reinterpret_cast<const void*>(&sparse24_kernel<0, true>); break;
    case 9: fn = reinterpret_cast<const void*>(&sparse24_kernel<1, true>); break;
    case 10: fn = reinterpret_cast<const void*>(&sparse24_kernel<2, true>); break;
    case 11: fn = reinterpret_cast<const void*>(&sparse24_kernel<3, true>); break;
    case 12: fn = reinterpret_cast<const void*>(&sparse24_kernel<4, true>); break;
    default: return cudaErrorNotSupported;
    }
    if (K % 128 != 0 || K > 4096 || N % 128 != 0 || (!dense && meta == nullptr)) return cudaErrorInvalidValue;
    const int smem = static_cast<int>(smem_bytes(dense) + 1024);
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(N / 128), static_cast<unsigned>((M + 127) / 128));
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = static_cast<size_t>(smem);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const unsigned wl = kWaitLimit;
    const int ar = act_ready ? 1 : 0;
    void* args[] = {const_cast<int8_t**>(&x), &M, &N, &K, const_cast<unsigned char**>(&aimg), const_cast<uint32_t**>(&meta),
                    const_cast<float**>(&scale), const_cast<float**>(&bias), &out, &inv_out_scale,
                    const_cast<int*>(&ar), const_cast<unsigned*>(&wl), &status};
    e = cudaLaunchKernelExC(&cfg, fn, args);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace bsg
