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
#include <cstdint>

#include "bsgemm_internal.h"

namespace bsg {
namespace {

constexpr int kPruneThreads = 256;

struct PruneState {
    unsigned long long prefix;  // key bytes chosen so far (the selected key after 8 passes)
    unsigned long long rank;    // rank of the wanted key among the keys matching `prefix`
    unsigned long long hist[256];
    int bad;                    // a weight was not finite
};

__global__ void prune_init_kernel(PruneState* st, unsigned long long rank) {
    const int t = threadIdx.x;
    st->hist[t] = 0;
    if (t == 0) {
        st->prefix = 0;
        st->rank = rank;
        st->bad = 0;
    }
}

// key[r * K + k] = bits of (((|w0| + |w1|) + |w2|) + |w3|) / 4 in double,
// w_i = W[4r + i][k]; the adds are exact-order IEEE double adds.
__global__ void prune_score_kernel(const float* __restrict__ W, int nbr, int K, unsigned long long* __restrict__ key,
                                   PruneState* st) {
    const long long total = static_cast<long long>(nbr) * K;
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    bool bad = false;
    for (long long id = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; id < total; id += stride) {
        const long long r = id / K;
        const long long k = id - r * K;
        const float* p = W + 4 * r * K + k;
        const float a0 = p[0], a1 = p[K], a2 = p[2 * static_cast<long long>(K)], a3 = p[3 * static_cast<long long>(K)];
        bad |= !(isfinite(a0) && isfinite(a1) && isfinite(a2) && isfinite(a3));
        double s = fabs(static_cast<double>(a0));
        s = __dadd_rn(s, fabs(static_cast<double>(a1)));
        s = __dadd_rn(s, fabs(static_cast<double>(a2)));
        s = __dadd_rn(s, fabs(static_cast<double>(a3)));
        key[id] = static_cast<unsigned long long>(__double_as_longlong(__dmul_rn(s, 0.25)));
    }
    if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(&st->bad, 1);
}

// Histogram of byte `pass` (0 = most significant) of the keys whose higher
// bytes equal those chosen so far.
__global__ void prune_hist_kernel(const unsigned long long* __restrict__ key, long long total, PruneState* st,
                                  int pass) {
    __shared__ unsigned int h[256];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    __syncthreads();
    const int shift = 56 - 8 * pass;
    const unsigned long long hi = pass == 0 ? 0ull : st->prefix >> (shift + 8);
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    for (long long id = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; id < total; id += stride) {
        const unsigned long long v = key[id];
        if (pass == 0 || (v >> (shift + 8)) == hi) atomicAdd(&h[(v >> shift) & 255u], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(&st->hist[i], static_cast<unsigned long long>(h[i]));
}

// Pick byte `pass` of the wanted key: the bin where the running count
// passes `rank`; one CTA of 256 threads.  Clears the histogram.
__global__ void prune_select_kernel(PruneState* st, int pass) {
    __shared__ unsigned long long c[256];
    const int t = threadIdx.x;
    c[t] = st->hist[t];
    __syncthreads();
    for (int off = 1; off < 256; off <<= 1) {
        const unsigned long long v = t >= off ? c[t - off] : 0ull;
        __syncthreads();
        c[t] += v;
        __syncthreads();
    }
    const unsigned long long rank = st->rank;
    const unsigned long long before = t ? c[t - 1] : 0ull;
    __syncthreads();  // every thread has read st->rank
    if (before <= rank && rank < c[t]) {
        st->prefix |= static_cast<unsigned long long>(t) << (56 - 8 * pass);
        st->rank = rank - before;
    }
    st->hist[t] = 0;
}

// Blocks with key equal to the selected one, per chunk of ids.
__global__ void prune_count_kernel(const unsigned long long* __restrict__ key, long long total, long long chunk,
                                   const PruneState* st, unsigned int* __restrict__ cnt) {
    const unsigned long long T = st->prefix;
    const long long lo = blockIdx.x * chunk;
    const long long hi = lo + chunk < total ? lo + chunk : total;
    unsigned int n = 0;
    for (long long id = lo + threadIdx.x; id < hi; id += blockDim.x) n += key[id] == T;
    for (int o = 16; o; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    __shared__ unsigned int ws[kPruneThreads / 32];
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = n;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned int s = 0;
        for (int w = 0; w < kPruneThreads / 32; ++w) s += ws[w];
        cnt[blockIdx.x] = s;
    }
}

// keep[id] = key > T, or key == T and at least `rank` equal keys come
// before it in id order.
__global__ void prune_mark_kernel(const unsigned long long* __restrict__ key, long long total, long long chunk,
                                  const PruneState* st, const unsigned int* __restrict__ cnt,
                                  uint8_t* __restrict__ keep) {
    __shared__ unsigned long long base_s;
    __shared__ unsigned int ws[kPruneThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned long long T = st->prefix;
    const unsigned long long need = st->rank;
    // equal keys in the chunks before this one
    unsigned long long b = 0;
    for (int c = threadIdx.x; c < static_cast<int>(blockIdx.x); c += blockDim.x) b += cnt[c];
    for (int o = 16; o; o >>= 1) b += __shfl_xor_sync(0xffffffffu, b, o);
    if (threadIdx.x == 0) base_s = 0;
    __syncthreads();
    if (lane == 0 && b) atomicAdd(&base_s, b);
    __syncthreads();
    unsigned long long run = base_s;
    const long long lo = blockIdx.x * chunk;
    const long long hi = lo + chunk < total ? lo + chunk : total;
    for (long long start = lo; start < hi; start += blockDim.x) {
        const long long id = start + threadIdx.x;
        const unsigned long long v = id < hi ? key[id] : 0ull;
        const bool eq = id < hi && v == T;
        const unsigned int bal = __ballot_sync(0xffffffffu, eq);
        const unsigned int before_lane = __popc(bal & ((1u << lane) - 1u));
        if (lane == 0) ws[warp] = __popc(bal);
        __syncthreads();
        unsigned int before_warp = 0, all = 0;
        for (int w = 0; w < kPruneThreads / 32; ++w) {
            before_warp += w < warp ? ws[w] : 0u;
            all += ws[w];
        }
        if (id < hi) keep[id] = v > T || (eq && run + before_warp + before_lane >= need);
        run += all;
        __syncthreads();  // ws is rewritten by the next round
    }
}

__global__ void prune_fill_kernel(uint8_t* __restrict__ keep, long long total, uint8_t v) {
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    for (long long id = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; id < total; id += stride)
        keep[id] = v;
}

}  // namespace

cudaError_t block_prune(const float* W, int N, int K, long long npruned, uint8_t* keep, int sms, cudaStream_t s,
                        bool* bad) {
    *bad = false;
    const int nbr = N / 4;
    const long long total = static_cast<long long>(nbr) * K;
    long long want = (total + kPruneThreads - 1) / kPruneThreads;
    const int grid = static_cast<int>(want < 4LL * sms ? (want > 0 ? want : 1) : 4LL * sms);
    // chunks of the ordered tie count: one per CTA, at most `grid`
    const long long chunk = (total + grid - 1) / grid;
    const int nchunks = static_cast<int>((total + chunk - 1) / chunk);

    unsigned long long* key = nullptr;
    PruneState* st = nullptr;
    unsigned int* cnt = nullptr;
    cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&key), sizeof(unsigned long long) * total, s);
    if (e == cudaSuccess) e = cudaMallocAsync(reinterpret_cast<void**>(&st), sizeof(PruneState), s);
    if (e == cudaSuccess) e = cudaMallocAsync(reinterpret_cast<void**>(&cnt), sizeof(unsigned int) * nchunks, s);
    if (e == cudaSuccess) {
        prune_init_kernel<<<1, 256, 0, s>>>(st, static_cast<unsigned long long>(npruned));
        prune_score_kernel<<<grid, kPruneThreads, 0, s>>>(W, nbr, K, key, st);
        if (npruned == 0 || npruned == total) {
            prune_fill_kernel<<<grid, kPruneThreads, 0, s>>>(keep, total, npruned == 0 ? 1 : 0);
        } else {
            for (int pass = 0; pass < 8; ++pass) {
                prune_hist_kernel<<<grid, kPruneThreads, 0, s>>>(key, total, st, pass);
                prune_select_kernel<<<1, 256, 0, s>>>(st, pass);
            }
            prune_count_kernel<<<nchunks, kPruneThreads, 0, s>>>(key, total, chunk, st, cnt);
            prune_mark_kernel<<<nchunks, kPruneThreads, 0, s>>>(key, total, chunk, st, cnt, keep);
        }
        e = cudaGetLastError();
    }
    int bad_h = 0;
    if (e == cudaSuccess && st) e = cudaMemcpyAsync(&bad_h, &st->bad, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (key) cudaFreeAsync(key, s);
    if (st) cudaFreeAsync(st, s);
    if (cnt) cudaFreeAsync(cnt, s);
    const cudaError_t e2 = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = e2;
    *bad = bad_h != 0;
    return e;
}

}  // namespace bsg
