// Host side of the C ABI declared in include/bsgemm.h: argument checks, the
// create-time repack of the block-compressed weight into steps (16 stored
// blocks of one block-row = 4 quads, the dot-4 unit of Algorithm 1), device
// upload, and the launch of the kernel in bsgemm_kernel.cu.
#include "bsgemm.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "bsgemm_internal.h"

struct bsgemm_ctx {
    int device = -1;
    int num_sms = 0;
    int ctas_per_sm = 0;
    int64_t nnzb = 0;
    void* arena = nullptr;
    size_t arena_bytes = 0;
    std::vector<int32_t> cost;  // host copy of the schedule's prefix cost [nbr + 1]
    bsg::DeviceWeights w{};
    std::mutex sched_mu;        // guards the cached schedule of the last token count
    long long sched_m = -1;
    int sched_grid = 0;
    bsg::Schedule sched{};
};

namespace {

thread_local std::string g_error;
thread_local int g_status = BSGEMM_OK;

int fail(int code, const std::string& msg) {
    g_error = msg;
    g_status = code;
    return code;
}

void clear_error() {
    g_error.clear();
    g_status = BSGEMM_OK;
}

std::string cuda_msg(const char* what, cudaError_t e) {
    return std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

const int kZeroStatus = 0;

// Check the block-compressed arrays; returns an empty string if valid.
std::string check_bsr(int N, int K, const int32_t* indptr, const int32_t* colidx) {
    const int nbr = N / BSGEMM_BLOCK;
    if (indptr[0] != 0) return "indptr[0] must be 0";
    for (int r = 0; r < nbr; ++r) {
        if (indptr[r + 1] < indptr[r]) return "indptr must be non-decreasing (block-row " + std::to_string(r) + ")";
        for (int j = indptr[r]; j < indptr[r + 1]; ++j) {
            const int k = colidx[j];
            if (k < 0 || k >= K)
                return "colidx[" + std::to_string(j) + "] = " + std::to_string(k) + " is outside [0, K)";
            if (j > indptr[r] && colidx[j - 1] >= k)
                return "columns must strictly increase within block-row " + std::to_string(r);
        }
    }
    return "";
}

// Schedule costs, in steps (16 stored blocks of one block-row for 64
// tokens: 32 dp4a per lane): every block-row adds kRowCost for its
// cross-lane sum and epilogue, every token tile in a CTA's range adds
// kTileCost for its copy into shared memory and the start-up around it.
constexpr long long kRowCost = 2;
constexpr long long kTileCost = 250;

// End of the greedy range that starts at unit u under the cost bound C: it
// takes whole units while the cost (units' cost + tc per token tile
// touched) stays within C, and at least one unit.
long long fill_range(const std::vector<int32_t>& cost, long long nbr, long long ntiles, long long tc, long long C,
                     long long u) {
    long long t = u / nbr, r = u - t * nbr, left = C;
    bool first = true;
    while (t < ntiles) {
        left -= tc;
        const long long rest = cost[nbr] - cost[r];
        if (left >= rest) {  // the rest of this tile fits
            left -= rest;
            ++t;
            r = 0;
            first = false;
            continue;
        }
        // the largest e with cost[e] - cost[r] <= left
        long long e = std::upper_bound(cost.begin() + r, cost.begin() + nbr + 1, cost[r] + (left > 0 ? left : 0)) -
                      cost.begin() - 1;
        if (e <= r && first) e = r + 1;  // at least one unit
        return t * nbr + (e > r ? e : r);
    }
    return ntiles * nbr;
}

// Contiguous unit ranges (tile-major units t * nbr + r), one per CTA, with
// the largest range cost as small as bisection on the bound finds it;
// returns the number of ranges (<= cap, each non-empty).
int make_schedule(const std::vector<int32_t>& cost, long long nbr, long long ntiles, int cap, long long tc,
                  bsg::Schedule& sched) {
    const long long end = ntiles * nbr;
    auto ranges = [&](long long C) {
        int n = 0;
        for (long long u = 0; u < end; u = fill_range(cost, nbr, ntiles, tc, C, u))
            if (++n > cap) break;
        return n;
    };
    long long hi = ntiles * (cost[nbr] + tc), lo = 0;
    while (hi - lo > 1) {
        const long long mid = lo + (hi - lo) / 2;
        if (ranges(mid) <= cap) hi = mid; else lo = mid;
    }
    int n = 0;
    sched.u[0] = 0;
    for (long long u = 0; u < end;) {
        u = fill_range(cost, nbr, ntiles, tc, hi, u);
        sched.u[++n] = u;
    }
    return n;
}

}  // namespace

extern "C" {

const char* bsgemm_last_error(void) { return g_error.c_str(); }

int bsgemm_last_status(void) { return g_status; }

int bsgemm_max_k(void) { return bsg::max_k(); }

bsgemm_t bsgemm_create(int N, int K, int block, const int32_t* indices, const int8_t* values, const float* scales,
                       const float* bias) {
    clear_error();
    if (block != BSGEMM_BLOCK) {
        fail(BSGEMM_ERR_UNSUPPORTED, "block must be 4 (4 output rows x 1 input column)");
        return nullptr;
    }
    if (N < BSGEMM_BLOCK || K < 1) {
        fail(BSGEMM_ERR_INVALID, "need N >= 4 and K >= 1");
        return nullptr;
    }
    if (N % BSGEMM_BLOCK != 0) {
        fail(BSGEMM_ERR_UNSUPPORTED, "N must be a multiple of 4 (padding is not implemented)");
        return nullptr;
    }
    if (K > bsg::max_k()) {
        fail(BSGEMM_ERR_UNSUPPORTED, "K = " + std::to_string(K) + " exceeds bsgemm_max_k() = " +
                                         std::to_string(bsg::max_k()));
        return nullptr;
    }
    if (!indices || !scales) {
        fail(BSGEMM_ERR_INVALID, "indices and scales must not be NULL");
        return nullptr;
    }
    const int nbr = N / BSGEMM_BLOCK;
    const int32_t* indptr = indices;
    const int64_t nnzb = indptr[nbr];
    if (indptr[0] != 0 || nnzb < 0 || nnzb > static_cast<int64_t>(nbr) * K) {
        fail(BSGEMM_ERR_INVALID, "indptr[0] must be 0 and 0 <= indptr[N/4] <= (N/4) * K");
        return nullptr;
    }
    if (nnzb > 0 && !values) {
        fail(BSGEMM_ERR_INVALID, "values must not be NULL when blocks are stored");
        return nullptr;
    }
    const int32_t* colidx = indices + nbr + 1;
    std::string bad = check_bsr(N, K, indptr, colidx);
    if (!bad.empty()) {
        fail(BSGEMM_ERR_INVALID, bad);
        return nullptr;
    }
    for (int n = 0; n < N; ++n) {
        if (!std::isfinite(scales[n]) || (bias && !std::isfinite(bias[n]))) {
            fail(BSGEMM_ERR_INVALID, "scales and bias must be finite (channel " + std::to_string(n) + ")");
            return nullptr;
        }
    }

    // Repack into steps.  Per block-row the stored columns are ordered so
    // that each half-step (8 consecutive columns, one pass of the kernel's
    // shared-memory gather) takes its columns from distinct bank groups of
    // the swizzled token tile where it can: every half-step draws one
    // column from each of the 8 bank-key buckets with the most columns left,
    // then (if fewer than 8 buckets are left) again from the fullest; the
    // last step is padded with zero-weight entries on unused keys (columns
    // 0..7 cover all 8 keys and are rows of every tile, which has
    // round_up(K, 16) >= 16 rows).
    std::vector<int32_t> sptr(nbr + 1, 0);
    std::vector<int32_t> cost(nbr + 1, 0);
    for (int r = 0; r < nbr; ++r) {
        const int nz = indptr[r + 1] - indptr[r];
        sptr[r + 1] = sptr[r] + (nz + 15) / 16;
        cost[r + 1] = static_cast<int32_t>(cost[r] + (nz + 15) / 16 + (nz > 0 ? kRowCost : 0));
    }
    const int S = sptr[nbr];
    std::vector<int32_t> recs(static_cast<size_t>(S + bsg::kStepPad) * 32, 0);
    int pad_col[8];
    for (int k = 0; k < 8; ++k) pad_col[bsg::bank_key(k)] = k;
    {
        std::vector<int> bucket[8];
        std::vector<int> order;  // stored-block index j, or -1 - key for a padding entry
        for (int r = 0; r < nbr; ++r) {
            const int j0 = indptr[r], j1 = indptr[r + 1];
            if (j1 == j0) continue;
            for (auto& b : bucket) b.clear();
            for (int j = j1 - 1; j >= j0; --j) bucket[bsg::bank_key(colidx[j])].push_back(j);  // popped in column order
            const int entries = (sptr[r + 1] - sptr[r]) * 16;
            order.clear();
            int left = j1 - j0;
            while (static_cast<int>(order.size()) < entries) {
                int keys[8] = {0, 1, 2, 3, 4, 5, 6, 7};
                std::stable_sort(keys, keys + 8, [&](int x, int y) { return bucket[x].size() > bucket[y].size(); });
                bool used[8] = {false, false, false, false, false, false, false, false};
                int taken = 0;
                for (int i = 0; i < 8 && taken < 8; ++i) {
                    if (bucket[keys[i]].empty()) continue;
                    order.push_back(bucket[keys[i]].back());
                    bucket[keys[i]].pop_back();
                    used[keys[i]] = true;
                    ++taken;
                    --left;
                }
                while (taken < 8 && left > 0) {  // fewer than 8 keys left: repeat the fullest
                    int best = 0;
                    for (int x = 1; x < 8; ++x)
                        if (bucket[x].size() > bucket[best].size()) best = x;
                    order.push_back(bucket[best].back());
                    bucket[best].pop_back();
                    used[best] = true;
                    ++taken;
                    --left;
                }
                for (int x = 0; x < 8 && taken < 8; ++x) {  // padding on keys this half-step does not use
                    if (used[x]) continue;
                    order.push_back(-1 - x);
                    used[x] = true;
                    ++taken;
                }
            }
            for (int s = 0; s < sptr[r + 1] - sptr[r]; ++s) {
                int32_t* rec = &recs[static_cast<size_t>(sptr[r] + s) * 32];
                uint32_t wwords[4][4] = {};
                for (int e = 0; e < 16; ++e) {
                    const int o = order[16 * s + e];
                    if (o >= 0) {
                        rec[e] = static_cast<int32_t>(bsg::tile_row_offset(colidx[o]));
                        for (int c = 0; c < 4; ++c)
                            wwords[e / 4][c] |= static_cast<uint32_t>(static_cast<uint8_t>(values[static_cast<size_t>(o) * 4 + c]))
                                                << (8 * (e % 4));
                    } else {
                        rec[e] = static_cast<int32_t>(bsg::tile_row_offset(pad_col[-1 - o]));
                    }
                }
                for (int qd = 0; qd < 4; ++qd)
                    for (int c = 0; c < 4; ++c) rec[16 + 4 * qd + c] = static_cast<int32_t>(wwords[qd][c]);
            }
        }
    }
    std::vector<float> bias_v(N, 0.0f);
    if (bias) std::memcpy(bias_v.data(), bias, sizeof(float) * N);

    auto* h = new bsgemm_ctx();
    cudaError_t e = cudaGetDevice(&h->device);
    if (e != cudaSuccess) {
        fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetDevice", e));
        delete h;
        return nullptr;
    }
    int optin = 0;
    e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
    if (e != cudaSuccess) {
        fail(BSGEMM_ERR_CUDA, cuda_msg("cudaDeviceGetAttribute", e));
        delete h;
        return nullptr;
    }
    if (bsg::smem_bytes(K) + bsg::kStaticSmem > static_cast<size_t>(optin)) {
        fail(BSGEMM_ERR_UNSUPPORTED, "this device has too little shared memory per block for K = " + std::to_string(K));
        delete h;
        return nullptr;
    }
    e = bsg::prepare_kernels(K, &h->ctas_per_sm);
    if (e != cudaSuccess || h->ctas_per_sm < 1) {
        fail(BSGEMM_ERR_CUDA, e != cudaSuccess ? cuda_msg("kernel setup", e) : "kernel cannot be resident on an SM");
        delete h;
        return nullptr;
    }

    const size_t off_sptr = 0;
    const size_t off_recs = align_up(off_sptr + sizeof(int32_t) * (nbr + 1), 256);
    const size_t off_scale = align_up(off_recs + sizeof(int32_t) * recs.size(), 256);
    const size_t off_bias = align_up(off_scale + sizeof(float) * N, 256);
    const size_t off_status = align_up(off_bias + sizeof(float) * N, 256);
    h->arena_bytes = align_up(off_status + sizeof(int), 256);
    e = cudaMalloc(&h->arena, h->arena_bytes);
    if (e != cudaSuccess) {
        fail(BSGEMM_ERR_CUDA, cuda_msg("cudaMalloc", e));
        delete h;
        return nullptr;
    }
    char* base = static_cast<char*>(h->arena);
    struct Piece { size_t off; const void* src; size_t bytes; } pieces[] = {
        {off_sptr, sptr.data(), sizeof(int32_t) * sptr.size()},
        {off_recs, recs.data(), sizeof(int32_t) * recs.size()},
        {off_scale, scales, sizeof(float) * N},
        {off_bias, bias_v.data(), sizeof(float) * N},
        {off_status, &kZeroStatus, sizeof(int)},
    };
    for (const Piece& p : pieces) {
        e = cudaMemcpy(base + p.off, p.src, p.bytes, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) {
            fail(BSGEMM_ERR_CUDA, cuda_msg("cudaMemcpy", e));
            cudaFree(h->arena);
            delete h;
            return nullptr;
        }
    }
    h->nnzb = nnzb;
    h->cost = cost;
    h->w.sptr = reinterpret_cast<const int32_t*>(base + off_sptr);
    h->w.recs = reinterpret_cast<const int4*>(base + off_recs);
    h->w.scale = reinterpret_cast<const float*>(base + off_scale);
    h->w.bias = reinterpret_cast<const float*>(base + off_bias);
    h->w.status = reinterpret_cast<int*>(base + off_status);
    h->w.N = N;
    h->w.K = K;
    h->w.nbr = nbr;
    h->w.S = S;
    return h;
}

// mode: 0 = gather from act (no scratch), 1 = relayout act into workspace
// then stage tiles, 2 = stage tiles already in workspace (act unused).
static int run_common(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                      size_t workspace_bytes, int mode, void* stream) {
    const bool use_ws = mode != 0;
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    if (M < 0) return fail(BSGEMM_ERR_INVALID, "M must be >= 0");
    if (epi.kind < BSGEMM_OUT_I32 || epi.kind > BSGEMM_OUT_I8_GELU)
        return fail(BSGEMM_ERR_INVALID, "unknown epilogue kind " + std::to_string(epi.kind));
    float inv = 0.0f;
    if (epi.kind == BSGEMM_OUT_I8 || epi.kind == BSGEMM_OUT_I8_GELU) {
        if (!(epi.out_scale > 0.0f) || !std::isfinite(epi.out_scale))
            return fail(BSGEMM_ERR_INVALID, "out_scale must be finite and > 0 for int8 outputs");
        inv = 1.0f / epi.out_scale;
        if (!std::isfinite(inv)) return fail(BSGEMM_ERR_INVALID, "1 / out_scale overflows fp32");
    }
    if (M == 0) return BSGEMM_OK;
    if ((mode != 2 && !act) || !out) return fail(BSGEMM_ERR_INVALID, "act and out must not be NULL");
    if (reinterpret_cast<uintptr_t>(out) % 16 != 0) return fail(BSGEMM_ERR_INVALID, "out must be 16-byte aligned");
    if (use_ws) {
        const size_t need = bsg::tiled_bytes(h->w.K, M);
        if (!workspace || workspace_bytes < need)
            return fail(BSGEMM_ERR_INVALID, "workspace must hold bsgemm_workspace_bytes(h, M) = " +
                                                std::to_string(need) + " bytes");
        if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
            return fail(BSGEMM_ERR_INVALID, "workspace must be 16-byte aligned");
    }
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetDevice", e));
    if (dev != h->device)
        return fail(BSGEMM_ERR_INVALID, "current device " + std::to_string(dev) + " is not the handle's device " +
                                            std::to_string(h->device));
    const cudaStream_t s = static_cast<cudaStream_t>(stream);

    bsg::LaunchArgs a{};
    a.x = act;
    a.xb = use_ws ? static_cast<const int8_t*>(workspace) : nullptr;
    a.out = out;
    a.M = M;
    a.kind = epi.kind;
    a.inv_out_scale = inv;
    a.x_vec16 = (reinterpret_cast<uintptr_t>(act) % 16 == 0) && (h->w.K % 16 == 0);
    const long long ntiles = (static_cast<long long>(M) + bsg::kTile - 1) / bsg::kTile;
    const long long nbr = h->w.nbr;
    long long cap = static_cast<long long>(h->num_sms) * h->ctas_per_sm;
    if (cap > bsg::kMaxGrid) cap = bsg::kMaxGrid;
    bsg::Schedule sched;
    int grid = 0;
    {
        std::lock_guard<std::mutex> lock(h->sched_mu);
        if (h->sched_m != M) {
            h->sched_grid = make_schedule(h->cost, nbr, ntiles, static_cast<int>(cap), kTileCost, h->sched);
            h->sched_m = M;
        }
        grid = h->sched_grid;
        std::memcpy(sched.u, h->sched.u, sizeof(long long) * (grid + 1));
    }
    if (mode == 1) {
        e = bsg::launch_pretile(act, M, h->w.K, static_cast<int8_t*>(workspace), h->num_sms, s);
        if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("relayout launch", e));
    }
    e = bsg::launch(h->w, a, sched, grid, s);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("kernel launch", e));
    return BSGEMM_OK;
}

int bsgemm_run(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* stream) {
    return run_common(h, act, M, out, epi, nullptr, 0, 0, stream);
}

int bsgemm_run_ws(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                  size_t workspace_bytes, void* stream) {
    return run_common(h, act, M, out, epi, workspace, workspace_bytes, 1, stream);
}

int bsgemm_run_tiled(bsgemm_t h, const void* tiles, size_t tiles_bytes, int M, void* out, bsgemm_epilogue epi,
                     void* stream) {
    return run_common(h, nullptr, M, out, epi, const_cast<void*>(tiles), tiles_bytes, 2, stream);
}

int bsgemm_run_static(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* stream) {
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    if (M > 0) {
        const size_t need = bsg::tiled_bytes(h->w.K, M);
        if (need > BSGEMM_STATIC_SCRATCH_BYTES) {
            const size_t per_tile = bsg::tiled_bytes(h->w.K, bsg::kTile);
            const long long m_max = static_cast<long long>(BSGEMM_STATIC_SCRATCH_BYTES / per_tile) * bsg::kTile;
            return fail(BSGEMM_ERR_INVALID, "M = " + std::to_string(M) + " needs " + std::to_string(need) +
                                                " bytes of token tiles; the static scratch holds " +
                                                std::to_string(static_cast<size_t>(BSGEMM_STATIC_SCRATCH_BYTES)) +
                                                " (M <= " + std::to_string(m_max) + " at K = " +
                                                std::to_string(h->w.K) + "): use bsgemm_run_ws");
        }
    }
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetDevice", e));
    if (dev != h->device)
        return fail(BSGEMM_ERR_INVALID, "current device " + std::to_string(dev) + " is not the handle's device " +
                                            std::to_string(h->device));
    int8_t* scratch = nullptr;
    e = bsg::static_scratch(dev, &scratch);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetSymbolAddress (static scratch)", e));
    return run_common(h, act, M, out, epi, scratch, BSGEMM_STATIC_SCRATCH_BYTES, 1, stream);
}

int bsgemm_tile_activations(bsgemm_t h, const int8_t* act, int M, void* tiles, size_t tiles_bytes, void* stream) {
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    if (M < 0) return fail(BSGEMM_ERR_INVALID, "M must be >= 0");
    if (M == 0) return BSGEMM_OK;
    if (!act) return fail(BSGEMM_ERR_INVALID, "act must not be NULL");
    const size_t need = bsg::tiled_bytes(h->w.K, M);
    if (!tiles || tiles_bytes < need)
        return fail(BSGEMM_ERR_INVALID, "tiles must hold bsgemm_workspace_bytes(h, M) = " + std::to_string(need) +
                                            " bytes");
    if (reinterpret_cast<uintptr_t>(tiles) % 16 != 0) return fail(BSGEMM_ERR_INVALID, "tiles must be 16-byte aligned");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetDevice", e));
    if (dev != h->device) return fail(BSGEMM_ERR_INVALID, "current device is not the handle's device");
    e = bsg::launch_pretile(act, M, h->w.K, static_cast<int8_t*>(tiles), h->num_sms, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("relayout launch", e));
    return BSGEMM_OK;
}

size_t bsgemm_workspace_bytes(bsgemm_t h, int M) {
    if (!h || M <= 0) return 0;
    return bsg::tiled_bytes(h->w.K, M);
}

int bsgemm_device_status(bsgemm_t h, int clear) {
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    int v = 0;
    cudaError_t e = cudaMemcpy(&v, h->w.status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && clear && v != 0) e = cudaMemcpy(h->w.status, &kZeroStatus, sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("reading the device status", e));
    return v;
}

void bsgemm_destroy(bsgemm_t h) {
    if (!h) return;
    if (h->arena) cudaFree(h->arena);
    delete h;
}

int bsgemm_info(bsgemm_t h, int64_t* out, int n) {
    clear_error();
    if (!h || (!out && n > 0)) return fail(BSGEMM_ERR_INVALID, "NULL handle or output");
    const int64_t v[7] = {h->w.N, h->w.K, h->nnzb, 4 * static_cast<int64_t>(h->w.S), bsg::kTile,
                          static_cast<int64_t>(h->num_sms) * h->ctas_per_sm, static_cast<int64_t>(h->arena_bytes)};
    for (int i = 0; i < n && i < 7; ++i) out[i] = v[i];
    return 7;
}

}  // extern "C"
