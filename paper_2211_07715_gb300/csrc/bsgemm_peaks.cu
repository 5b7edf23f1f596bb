// Peak rates of GB300's int8 dot-product units, measured on the device the
// layer kernel runs on.  They are the denominators of the layer's roofline:
// the layer is an int8 contraction (Sec. 3, Algorithm 1's vpdpbusd dot-4),
// and on this GPU it runs on dp4a.  Two probes:
//   * dp4a: every thread runs 8 independent accumulation chains of
//     __dp4a (4 int8 multiply-adds into int32 each), 32 warps per SM;
//   * mma.sync m16n8k32 s8 x s8 -> s32 (the legacy warp-level tensor-core
//     instruction): every warp keeps 4 independent accumulator tiles.
// Operands change every iteration so that nothing can be folded away; the
// results are combined into one word that is written only if it has an
// impossible value (so the work stays live without stores in the loop).
#include <cstdint>
#include <cuda_runtime.h>

#include "bsgemm.h"

namespace {

constexpr int kPeakThreads = 256;
constexpr int kPeakBlocksPerSm = 4;

__global__ void __launch_bounds__(kPeakThreads)
dp4a_peak_kernel(int iters, int seed, int* sink) {
    uint32_t a = static_cast<uint32_t>(seed) + threadIdx.x * 2654435761u;
    const int b = seed * 3 + 1;
    int acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = j;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int r = 0; r < 16; ++r) {
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] = __dp4a(static_cast<int>(a ^ static_cast<uint32_t>(j)), b + r, acc[j]);
        }
        a = a * 1664525u + 1013904223u;
    }
    int s = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) s ^= acc[j];
    if (s == 0x7fffffff && seed == 12345) sink[blockIdx.x] = s;
}

__global__ void __launch_bounds__(kPeakThreads)
mma_s8_peak_kernel(int iters, int seed, int* sink) {
    uint32_t a[4], b[2];
#pragma unroll
    for (int j = 0; j < 4; ++j) a[j] = static_cast<uint32_t>(seed) * (j + 1) + threadIdx.x;
    b[0] = static_cast<uint32_t>(seed) ^ 0x5a5a5a5au;
    b[1] = static_cast<uint32_t>(seed) + 77u;
    int d[4][4];
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int j = 0; j < 4; ++j) d[t][j] = t + j;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                asm volatile(
                    "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
                    "{%0, %1, %2, %3};\n"
                    : "+r"(d[t][0]), "+r"(d[t][1]), "+r"(d[t][2]), "+r"(d[t][3])
                    : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3] + static_cast<uint32_t>(t)), "r"(b[0]), "r"(b[1]));
            }
        }
        a[0] = a[0] * 1664525u + 1013904223u;
    }
    int s = 0;
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int j = 0; j < 4; ++j) s ^= d[t][j];
    if (s == 0x7fffffff && seed == 12345) sink[blockIdx.x] = s;
}

}  // namespace

extern "C" int bsgemm_int8_peak(int unit, int iters, double* tops) {
    if ((unit != 0 && unit != 1) || iters < 1 || !tops) return BSGEMM_ERR_INVALID;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return BSGEMM_ERR_CUDA;
    const int blocks = sms * kPeakBlocksPerSm;
    int* sink = nullptr;
    if (cudaMalloc(&sink, sizeof(int) * blocks) != cudaSuccess) return BSGEMM_ERR_CUDA;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    cudaError_t e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    float best_ms = 0.0f;
    for (int rep = 0; rep < 4 && e == cudaSuccess; ++rep) {  // the first launch warms up; the best of the rest
        e = cudaEventRecord(e0, 0);
        if (unit == 0)
            dp4a_peak_kernel<<<blocks, kPeakThreads>>>(iters, 7 + rep, sink);
        else
            mma_s8_peak_kernel<<<blocks, kPeakThreads>>>(iters, 7 + rep, sink);
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e == cudaSuccess) e = cudaEventRecord(e1, 0);
        if (e == cudaSuccess) e = cudaEventSynchronize(e1);
        float ms = 0.0f;
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
        if (e == cudaSuccess && rep > 0 && (best_ms == 0.0f || ms < best_ms)) best_ms = ms;
    }
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    cudaFree(sink);
    if (e != cudaSuccess || best_ms <= 0.0f) return BSGEMM_ERR_CUDA;
    const double threads = static_cast<double>(blocks) * kPeakThreads;
    // dp4a: 128 per thread per iteration, 8 ops each; mma: 16 per warp per
    // iteration, 16 x 8 x 32 multiply-adds = 8192 ops each
    const double ops = unit == 0 ? threads * iters * 128.0 * 8.0 : threads / 32.0 * iters * 16.0 * 8192.0;
    *tops = ops / (best_ms * 1e-3) / 1e12;
    return BSGEMM_OK;
}
