// Create-side block pruning (App. A.1): score every 4x1 block of a dense
// fp32 weight by the mean magnitude of its four values and keep the blocks
// outside the `npruned` lowest scores.  Equal scores are ordered by the
// block's index r * K + k, the lower index pruned first.
//
// GPU form: the scores are non-negative doubles, whose IEEE bit patterns
// sort like the values, so the block at rank `npruned` (the lowest kept
// block) is found by an 8-pass radix select over the 64-bit keys (one byte
// per pass: a histogram of the keys that match the bytes chosen so far,
// then a 256-entry scan that picks the next byte).  Blocks below that key
// are pruned, blocks above it kept, and among the blocks equal to it the
// first `rank` in index order are pruned (an ordered count over chunks).
//
// All of it is one cooperative kernel (every CTA resident): phases are
// separated by grid barriers whose waits are bounded, and every CTA repeats
// the 256-entry scans itself, so no phase needs a kernel of its own.
#include <cstdint>
#include <mutex>

#include "bsgemm.h"
#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kPruneThreads = 512;
constexpr int kBatch = 8;  // elements a thread loads before using any (loads in flight)
constexpr unsigned kBarrierLimit = 1u << 22;  // spins of a grid barrier before it gives up

// Scratch of one call (zeroed by the host before the launch).
struct PruneScratch {
    unsigned long long hist[8][256];  // pass p's histogram of key byte p
    unsigned int barrier;             // arrivals at the grid barriers (monotonic)
    int bad;                          // 1: a weight is not finite; 2: a grid barrier gave up
};

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid barrier number `n` (0, 1, ...): every CTA arrives once; returns false
// (in every thread of the CTA) if the wait gave up.
__device__ bool grid_barrier(PruneScratch* st, unsigned n, unsigned limit) {
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        atomicAdd(&st->barrier, 1u);
        const unsigned target = (n + 1) * gridDim.x;
        unsigned i = 0;
        while (ld_acquire(&st->barrier) < target && i < limit) ++i;
        s_ok = i < limit;
        if (!s_ok) atomicOr(&st->bad, 2);
        __threadfence();
    }
    __syncthreads();
    return s_ok != 0;
}

// Select byte `pass` of the wanted key from the histogram: the bin where the
// running count passes `rank`.  Every CTA does it; thread 0's result is
// broadcast through shared memory.
__device__ void select_byte(const unsigned long long* hist, int pass, unsigned long long& prefix,
                            unsigned long long& rank) {
    __shared__ unsigned long long c[256];
    __shared__ unsigned long long s_prefix, s_rank;
    const int t = threadIdx.x;
    if (t < 256) c[t] = __ldcg(hist + t);
    __syncthreads();
    for (int off = 1; off < 256; off <<= 1) {
        unsigned long long v = 0;
        if (t < 256 && t >= off) v = c[t - off];
        __syncthreads();
        if (t < 256) c[t] += v;
        __syncthreads();
    }
    if (t < 256) {
        const unsigned long long before = t ? c[t - 1] : 0ull;
        if (before <= rank && rank < c[t]) {
            s_prefix = prefix | (static_cast<unsigned long long>(t) << (56 - 8 * pass));
            s_rank = rank - before;
        }
    }
    __syncthreads();
    prefix = s_prefix;
    rank = s_rank;
}

__global__ void __launch_bounds__(kPruneThreads)
prune_kernel(const float* __restrict__ W, int nbr, int K, unsigned long long npruned,
             unsigned long long* __restrict__ key, unsigned int* __restrict__ cnt, PruneScratch* st,
             uint8_t* __restrict__ keep, unsigned barrier_limit, int leave_cta) {
    __shared__ unsigned int h[256];
    __shared__ unsigned int ws[kPruneThreads / 32];
    __shared__ unsigned long long s_base;
    const long long total = static_cast<long long>(nbr) * K;
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    const long long tid0 = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    __syncthreads();

    // Scores: key[r K + k] = bits of (((|w0| + |w1|) + |w2|) + |w3|) / 4 in
    // double, w_i = W[4r + i][k], in that order; and pass 0's histogram.
    bool bad = false;
    for (long long id0 = tid0; id0 < total; id0 += kBatch * stride) {
        float a[kBatch][4];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const long long id = id0 + u * stride;
            if (id < total) {
                const long long r = id / K;
                const float* p = W + 4 * r * K + (id - r * K);
#pragma unroll
                for (int i = 0; i < 4; ++i) a[u][i] = __ldg(p + i * static_cast<long long>(K));
            }
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const long long id = id0 + u * stride;
            if (id < total) {
                bad |= !(isfinite(a[u][0]) && isfinite(a[u][1]) && isfinite(a[u][2]) && isfinite(a[u][3]));
                double s = fabs(static_cast<double>(a[u][0]));
                s = __dadd_rn(s, fabs(static_cast<double>(a[u][1])));
                s = __dadd_rn(s, fabs(static_cast<double>(a[u][2])));
                s = __dadd_rn(s, fabs(static_cast<double>(a[u][3])));
                const unsigned long long v = static_cast<unsigned long long>(__double_as_longlong(__dmul_rn(s, 0.25)));
                key[id] = v;
                atomicAdd(&h[v >> 56], 1u);
            }
        }
    }
    if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(&st->bad, 1);
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(&st->hist[0][i], static_cast<unsigned long long>(h[i]));
    unsigned nb = 0;
    if (static_cast<int>(blockIdx.x) == leave_cta) return;  // test hook: the others' first barrier gives up
    if (!grid_barrier(st, nb++, barrier_limit)) return;

    // Radix select of the key at rank npruned (0 < npruned < total).
    unsigned long long prefix = 0, rank = npruned;
    for (int pass = 1; pass < 8; ++pass) {
        select_byte(st->hist[pass - 1], pass - 1, prefix, rank);
        for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
        __syncthreads();
        const int shift = 56 - 8 * pass;
        const unsigned long long hi = prefix >> (shift + 8);
        for (long long id0 = tid0; id0 < total; id0 += kBatch * stride) {
            unsigned long long v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const long long id = id0 + u * stride;
                v[u] = id < total ? __ldcg(key + id) : ~0ull;
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (id0 + u * stride < total && (v[u] >> (shift + 8)) == hi) atomicAdd(&h[(v[u] >> shift) & 255u], 1u);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < 256; i += blockDim.x)
            if (h[i]) atomicAdd(&st->hist[pass][i], static_cast<unsigned long long>(h[i]));
        if (!grid_barrier(st, nb++, barrier_limit)) return;
    }
    select_byte(st->hist[7], 7, prefix, rank);
    const unsigned long long T = prefix, need = rank;

    // Keys equal to T: the first `need` in index order are pruned.  CTA c
    // owns the contiguous chunk [c * chunk, (c + 1) * chunk) of ids.
    const long long chunk = (total + gridDim.x - 1) / gridDim.x;
    const long long lo = blockIdx.x * chunk;
    const long long hi_id = lo + chunk < total ? lo + chunk : total;
    unsigned n = 0;
    for (long long id0 = lo + threadIdx.x; id0 < hi_id; id0 += kBatch * blockDim.x) {
        unsigned long long v[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const long long id = id0 + u * static_cast<long long>(blockDim.x);
            v[u] = id < hi_id ? __ldcg(key + id) : ~T;
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) n += v[u] == T;
    }
    for (int o = 16; o; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    if (lane == 0) ws[warp] = n;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned s = 0;
        for (int w = 0; w < kPruneThreads / 32; ++w) s += ws[w];
        cnt[blockIdx.x] = s;
    }
    if (!grid_barrier(st, nb++, barrier_limit)) return;

    // equal keys in the chunks before this one
    unsigned long long b = 0;
    for (int c = threadIdx.x; c < static_cast<int>(blockIdx.x); c += blockDim.x) b += __ldcg(cnt + c);
    for (int o = 16; o; o >>= 1) b += __shfl_xor_sync(0xffffffffu, b, o);
    if (threadIdx.x == 0) s_base = 0;
    __syncthreads();
    if (lane == 0 && b) atomicAdd(&s_base, b);
    __syncthreads();
    unsigned long long run = s_base;
    for (long long s0 = lo; s0 < hi_id; s0 += kBatch * static_cast<long long>(blockDim.x)) {
        unsigned long long v[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const long long id = s0 + u * static_cast<long long>(blockDim.x) + threadIdx.x;
            v[u] = id < hi_id ? __ldcg(key + id) : 0ull;
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {  // rounds in index order; in a round, ids in thread order
            const long long id = s0 + u * static_cast<long long>(blockDim.x) + threadIdx.x;
            const bool eq = id < hi_id && v[u] == T;
            const unsigned bal = __ballot_sync(0xffffffffu, eq);
            const unsigned before_lane = __popc(bal & ((1u << lane) - 1u));
            __syncthreads();  // ws of the previous round is read
            if (lane == 0) ws[warp] = __popc(bal);
            __syncthreads();
            unsigned before_warp = 0, all = 0;
            for (int w = 0; w < kPruneThreads / 32; ++w) {
                before_warp += w < warp ? ws[w] : 0u;
                all += ws[w];
            }
            if (id < hi_id) keep[id] = v[u] > T || (eq && run + before_warp + before_lane >= need);
            run += all;
        }
    }
}

__global__ void prune_fill_kernel(const float* __restrict__ W, int nbr, int K, uint8_t* __restrict__ keep, uint8_t v,
                                  PruneScratch* st) {
    const long long total = static_cast<long long>(nbr) * K;
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    bool bad = false;
    for (long long id = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; id < total; id += stride) {
        const long long r = id / K;
        const long long k = id - r * K;
        const float* p = W + 4 * r * K + k;
        for (int i = 0; i < 4; ++i) bad |= !isfinite(p[static_cast<long long>(i) * K]);
        keep[id] = v;
    }
    if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(&st->bad, 1);
}

}  // namespace

namespace {

// Scratch kept per device between calls (grown on demand): the keys, the
// per-CTA tie counts, the phase state, and a pinned host word for the
// status.  Calls on one device are serialised by the mutex (pruning is a
// create-time step).
struct PruneCache {
    std::mutex mu;
    void* dev = nullptr;
    size_t bytes = 0;
    int* host_bad = nullptr;
};
PruneCache g_prune_cache[64];

}  // namespace

cudaError_t block_prune(const float* W, int N, int K, long long npruned, uint8_t* keep, int sms, cudaStream_t s,
                        bool* bad) {
    *bad = false;
    const int nbr = N / 4;
    const long long total = static_cast<long long>(nbr) * K;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    // one CTA per SM: every CTA is resident, and a grid barrier waits for
    // as few arrivals as the GPU has SMs
    const long long want = (total + kPruneThreads - 1) / kPruneThreads;
    const long long cap = sms > 0 ? sms : 1;
    const int grid = static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);

    PruneCache& c = g_prune_cache[dev];
    std::lock_guard<std::mutex> lock(c.mu);
    const size_t off_cnt = (sizeof(PruneScratch) + 255) & ~static_cast<size_t>(255);
    const size_t off_key = off_cnt + ((sizeof(unsigned int) * grid + 255) & ~static_cast<size_t>(255));
    const size_t need = off_key + sizeof(unsigned long long) * static_cast<size_t>(total);
    if (!c.host_bad) {
        e = cudaMallocHost(reinterpret_cast<void**>(&c.host_bad), sizeof(int));
        if (e != cudaSuccess) return e;
    }
    if (c.bytes < need) {
        if (c.dev) cudaFree(c.dev);
        c.dev = nullptr;
        c.bytes = 0;
        e = cudaMalloc(&c.dev, need);
        if (e != cudaSuccess) return e;
        c.bytes = need;
    }
    char* base = static_cast<char*>(c.dev);
    PruneScratch* st = reinterpret_cast<PruneScratch*>(base);
    unsigned int* cnt = reinterpret_cast<unsigned int*>(base + off_cnt);
    unsigned long long* key = reinterpret_cast<unsigned long long*>(base + off_key);
    *c.host_bad = 0;
    e = cudaMemsetAsync(st, 0, sizeof(PruneScratch), s);
    if (e == cudaSuccess) {
        if (npruned == 0 || npruned == total) {
            prune_fill_kernel<<<grid, kPruneThreads, 0, s>>>(W, nbr, K, keep, npruned == 0 ? 1 : 0, st);
            e = cudaGetLastError();
        } else {
            unsigned long long np = static_cast<unsigned long long>(npruned);
            // test hook: CTA 0 leaves before the first grid barrier, the others give up after a few polls
            const bool stall = (test_hooks() & BSGEMM_TEST_STALL_PRUNE_CTA) != 0;
            unsigned limit = stall ? 4096u : kBarrierLimit;
            int leave = stall ? 0 : -1;
            void* args[] = {const_cast<float**>(&W), const_cast<int*>(&nbr), &K, &np, &key, &cnt, &st, &keep,
                            &limit, &leave};
            e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(prune_kernel), dim3(grid),
                                            dim3(kPruneThreads), args, 0, s);
        }
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(c.host_bad, &st->bad, sizeof(int), cudaMemcpyDeviceToHost, s);
    const cudaError_t e2 = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = e2;
    const int bad_h = e == cudaSuccess ? *c.host_bad : 0;
    if (e == cudaSuccess && (bad_h & 2)) e = cudaErrorLaunchTimeout;  // a grid barrier gave up
    *bad = (bad_h & 1) != 0;
    return e;
}

}  // namespace bsg
