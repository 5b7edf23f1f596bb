// Host side of the C ABI declared in include/bsgemm.h: argument checks, the
// create-time repack of the block-compressed weight into steps (16 stored
// blocks of one block-row = 4 quads, the dot-4 unit of Algorithm 1), device
// upload, and the launch of the kernel in bsgemm_kernel.cu.
#include "bsgemm.h"

#include <algorithm>
#include <atomic>
#include <cfloat>
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "bsgemm_internal.h"

constexpr int kShape4x1 = 0;  // 4 consecutive output rows x 1 input column
constexpr int kShape1x4 = 1;  // 1 output row x 4 consecutive input columns

struct bsgemm_ctx {
    int device = -1;
    int shape = kShape4x1;      // block shape of the stored weight
    int num_sms = 0;
    int ctas_per_sm = 0;
    int64_t nnzb = 0;
    void* arena = nullptr;
    size_t arena_bytes = 0;
    std::vector<int32_t> cost;  // schedule prefix cost of the row groups [ngroups + 1]
    bsg::DeviceWeights w{};
    // Handles of bsgemm_create_2to4 / bsgemm_create_tc with N and K
    // multiples of 128: the tensor cores' operands (launch_tc_linear), in
    // their own allocation; NULL otherwise.  tc_dense: the dense MMA's image.
    void* tc_arena = nullptr;
    const unsigned char* tc_aimg = nullptr;
    const uint32_t* tc_meta = nullptr;
    bool tc_dense = false;
    size_t tc_bytes = 0;
    std::mutex sched_mu;        // guards the cached schedule of the last token count
    long long sched_m = -1;
    int sched_grid = 0;
    bsg::Schedule sched{};
};

namespace {

std::atomic<uint32_t> g_test_hooks{0};  // bsgemm_set_test_hooks
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

// IEEE binary16 bits of an int8 value (exact: |v| <= 128 needs at most 8
// significant bits).
uint16_t f16_of_int(int8_t v8) {
    int v = v8;
    if (v == 0) return 0;
    const uint16_t sign = v < 0 ? 0x8000u : 0u;
    unsigned a = static_cast<unsigned>(v < 0 ? -v : v);
    int ex = 0;
    while ((a >> ex) > 1) ++ex;                      // a = 1.f x 2^ex
    const unsigned mant = (a << (10 - ex)) & 0x3FFu;  // 10 fraction bits
    return static_cast<uint16_t>(sign | ((ex + 15) << 10) | mant);
}

const int kZeroStatus = 0;

// Check the block-compressed arrays; returns an empty string if valid.
std::string check_bsr(int N, int K, const int32_t* indptr, const int32_t* colidx) {
    const int nbr = (N + BSGEMM_BLOCK - 1) / BSGEMM_BLOCK;
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

// Schedule costs, in steps (one quad of each of a row group's 4 block-rows
// for 64 tokens: 32 dp4a per lane), from per-CTA clock traces of the
// kernel on GB300 (FFN1/FFN2/QKV/attention-output shapes, M = 3072-4096):
// a CTA spends about 19 cycles per step and 17 steps' worth per row group
// (its epilogue); a CTA that touches a second token tile runs 1.6K-5K
// cycles longer than the first tile's cost predicts (the tile's copy into
// shared memory, its transpose, the warps' set-up and finishing spread),
// which puts a tile at 450 + 300 K / 3072 steps (tuned on the four shapes).
#ifndef BSG_GROUP_COST
#define BSG_GROUP_COST 17
#endif
constexpr long long kGroupCost = BSG_GROUP_COST;
#ifndef BSG_TILE_COST_A
#define BSG_TILE_COST_A 450
#endif
#ifndef BSG_TILE_COST_B
#define BSG_TILE_COST_B 300
#endif
long long tile_cost(int K) { return BSG_TILE_COST_A + BSG_TILE_COST_B * static_cast<long long>(K) / 3072; }

// End of the greedy range that starts at unit u under the cost bound C: it
// takes whole units while the cost (units' cost + tc per token tile
// touched) stays within C, and at least one unit.
long long fill_range(const std::vector<int32_t>& cost, long long upt, long long ntiles, long long tc, long long C,
                     long long u) {
    long long t = u / upt, r = u - t * upt, left = C;
    bool first = true;
    while (t < ntiles) {
        left -= tc;
        const long long rest = cost[upt] - cost[r];
        if (left >= rest) {  // the rest of this tile fits
            left -= rest;
            ++t;
            r = 0;
            first = false;
            continue;
        }
        // the largest e with cost[e] - cost[r] <= left
        long long e = std::upper_bound(cost.begin() + r, cost.begin() + upt + 1, cost[r] + (left > 0 ? left : 0)) -
                      cost.begin() - 1;
        if (e <= r && first) e = r + 1;  // at least one unit
        return t * upt + (e > r ? e : r);
    }
    return ntiles * upt;
}

// Contiguous unit ranges (tile-major units t * upt + r, upt = row groups
// per token tile), one per CTA, with the largest range cost as small as
// bisection on the bound finds it; returns the number of ranges (<= cap,
// each non-empty).
int make_schedule(const std::vector<int32_t>& cost, long long upt, long long ntiles, int cap, long long tc,
                  bsg::Schedule& sched) {
    const long long end = ntiles * upt;
    auto ranges = [&](long long C) {
        int n = 0;
        for (long long u = 0; u < end; u = fill_range(cost, upt, ntiles, tc, C, u))
            if (++n > cap) break;
        return n;
    };
    long long hi = ntiles * (cost[upt] + tc), lo = 0;
    while (hi - lo > 1) {
        const long long mid = lo + (hi - lo) / 2;
        if (ranges(mid) <= cap) hi = mid; else lo = mid;
    }
    int n = 0;
    sched.u[0] = 0;
    for (long long u = 0; u < end;) {
        u = fill_range(cost, upt, ntiles, tc, hi, u);
        sched.u[++n] = u;
    }
    return n;
}

// Column order of every step of every row group (create time).  Each half
// of a step (8 columns: one quad of block-row 2h, one of block-row 2h + 1,
// one pass of the kernel's shared-memory gather) takes its columns from
// distinct bank groups of the swizzled token tile where it can: pick by
// pick, the block-row whose fullest bucket of an unused bank key is largest
// takes a column from it; a block-row whose remaining columns all sit on
// used keys takes one anyway (a conflict, never an extra step); a block-row
// with no columns left is padded with a zero-weight entry on an unused key
// (columns 0..7 cover all 8 keys and are rows of every tile).  ent[16 s + e] = the stored-block index j of entry e of step s, or
// -1 - (pad column).
void order_steps(const int32_t* indptr, const int32_t* colidx, int ngroups, const std::vector<int32_t>& grow,
                 const std::vector<int32_t>& gptr, int (*bank_key)(int), std::vector<int32_t>& ent) {
    ent.assign(static_cast<size_t>(gptr[ngroups]) * 16, 0);
    int pad_col[8];
    for (int k = 0; k < 8; ++k) pad_col[bank_key(k)] = k;
    std::vector<int> bucket[4][8];  // stored-block indices j of each block-row, by bank key
    int left[4];
    for (int gi = 0; gi < ngroups; ++gi) {
        for (int q = 0; q < 4; ++q) {
            for (auto& bk : bucket[q]) bk.clear();
            left[q] = 0;
            const int r = grow[4 * gi + q];
            if (r < 0) continue;
            for (int j = indptr[r + 1] - 1; j >= indptr[r]; --j) bucket[q][bank_key(colidx[j])].push_back(j);
            left[q] = indptr[r + 1] - indptr[r];
        }
        for (int s = gptr[gi]; s < gptr[gi + 1]; ++s) {
            int32_t* es = &ent[static_cast<size_t>(s) * 16];
            for (int h = 0; h < 2; ++h) {
                bool used[8] = {false, false, false, false, false, false, false, false};
                int placed[2] = {0, 0};
                for (int n = 0; n < 8; ++n) {
                    // candidate of each of the two block-rows still short of 4 entries:
                    // the size of its fullest bucket on an unused key (-1: none)
                    int best_x = -1, best_key = -1, best_size = -2;
                    for (int x = 0; x < 2; ++x) {
                        const int q = 2 * h + x;
                        if (placed[x] == 4) continue;
                        int key = -1, size = -1;
                        for (int kk = 0; kk < 8; ++kk)
                            if (!used[kk] && static_cast<int>(bucket[q][kk].size()) > size && !bucket[q][kk].empty()) {
                                key = kk;
                                size = static_cast<int>(bucket[q][kk].size());
                            }
                        if (size > best_size || (size == best_size && left[q] > left[2 * h + best_x])) {
                            best_x = x;
                            best_key = key;
                            best_size = size;
                        }
                    }
                    const int q = 2 * h + best_x;
                    const int e = 4 * q + placed[best_x];
                    int j = -1, key = best_key;
                    if (key < 0 && left[q] > 0) {  // its columns sit on used keys only: take a conflict
                        for (int kk = 0; kk < 8; ++kk)
                            if (key < 0 || bucket[q][kk].size() > bucket[q][key].size()) key = kk;
                    }
                    if (key >= 0 && left[q] > 0) {
                        j = bucket[q][key].back();
                        bucket[q][key].pop_back();
                        --left[q];
                    } else {  // padding on an unused key (any key if all are used)
                        key = 0;
                        for (int kk = 7; kk >= 0; --kk)
                            if (!used[kk]) key = kk;
                    }
                    used[key] = true;
                    ++placed[best_x];
                    es[e] = j >= 0 ? j : -1 - pad_col[key];
                }
            }
        }
    }
}

// One step's 16 entries: off[e] = the tile offset of its column (row_off of
// the layout), w[q][c] byte e % 4 = W[4 r_q + c][column of entry 4q + e % 4]
// (0 for padding).
void step_entries(const int32_t* es, const int32_t* colidx, const int8_t* values, uint32_t (*row_off)(int),
                  int32_t* off, uint32_t (&w)[4][4]) {
    for (int e = 0; e < 16; ++e) {
        const int j = es[e];
        const int q = e / 4;
        if (j >= 0) {
            off[e] = static_cast<int32_t>(row_off(colidx[j]));
            for (int c = 0; c < 4; ++c)
                w[q][c] |= static_cast<uint32_t>(static_cast<uint8_t>(values[static_cast<size_t>(j) * 4 + c]))
                           << (8 * (e % 4));
        } else {
            off[e] = static_cast<int32_t>(row_off(-1 - j));
        }
    }
}

// A weight repacked into row groups and step records (either block shape).
struct Repacked {
    int shape = kShape4x1;
    int N = 0, K = 0;
    int64_t nnzb = 0;
    int ngroups = 0, S = 0;
    std::vector<int32_t> grow, gptr, cost, recs;
};

// Device upload of a repacked weight into one arena; the kernels are set up
// for K on the current device.  Returns NULL (with the error recorded) on
// failure.
bsgemm_t upload(const Repacked& rp, const float* scales, const float* bias) {
    const int N = rp.N, K = rp.K, ngroups = rp.ngroups;
    // scales and biases padded with zeros to a multiple of 4 channels (the
    // 4 x 1 kernel reads 4 channels at a time and stores only channels < N)
    const int npad = (N + 3) / 4 * 4;
    std::vector<float> scale_v(npad, 0.0f), bias_v(npad, 0.0f);
    std::memcpy(scale_v.data(), scales, sizeof(float) * N);
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

    const size_t off_gptr = 0;
    const size_t off_grow = align_up(off_gptr + sizeof(int32_t) * (ngroups + 1), 256);
    const size_t off_recs = align_up(off_grow + sizeof(int32_t) * rp.grow.size(), 256);
    const size_t off_scale = align_up(off_recs + sizeof(int32_t) * rp.recs.size(), 256);
    const size_t off_bias = align_up(off_scale + sizeof(float) * npad, 256);
    const size_t off_status = align_up(off_bias + sizeof(float) * npad, 256);
    h->arena_bytes = align_up(off_status + sizeof(int), 256);
    e = cudaMalloc(&h->arena, h->arena_bytes);
    if (e != cudaSuccess) {
        fail(BSGEMM_ERR_CUDA, cuda_msg("cudaMalloc", e));
        delete h;
        return nullptr;
    }
    char* base = static_cast<char*>(h->arena);
    struct Piece { size_t off; const void* src; size_t bytes; } pieces[] = {
        {off_gptr, rp.gptr.data(), sizeof(int32_t) * rp.gptr.size()},
        {off_grow, rp.grow.data(), sizeof(int32_t) * rp.grow.size()},
        {off_recs, rp.recs.data(), sizeof(int32_t) * rp.recs.size()},
        {off_scale, scale_v.data(), sizeof(float) * npad},
        {off_bias, bias_v.data(), sizeof(float) * npad},
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
    h->nnzb = rp.nnzb;
    h->cost = rp.cost;
    h->shape = rp.shape;
    h->w.gptr = reinterpret_cast<const int32_t*>(base + off_gptr);
    h->w.grow = reinterpret_cast<const int4*>(base + off_grow);
    h->w.recs = reinterpret_cast<const int4*>(base + off_recs);
    h->w.scale = reinterpret_cast<const float*>(base + off_scale);
    h->w.bias = reinterpret_cast<const float*>(base + off_bias);
    h->w.status = reinterpret_cast<int*>(base + off_status);
    h->w.N = N;
    h->w.K = K;
    h->w.ngroups = ngroups;
    h->w.S = rp.S;
    return h;
}

}  // namespace

unsigned bsg::test_hooks() { return g_test_hooks.load(); }

// Upload the tensor cores' operands of handle h into their own allocation;
// on failure destroys h and returns NULL.
static bsgemm_t attach_tc(bsgemm_t h, const std::vector<uint16_t>& aimg, const std::vector<uint32_t>& meta,
                          bool dense) {
    const size_t abytes = aimg.size() * sizeof(uint16_t), mbytes = meta.size() * sizeof(uint32_t);
    void* arena = nullptr;
    cudaError_t e = cudaMalloc(&arena, abytes + mbytes);
    if (e == cudaSuccess) e = cudaMemcpy(arena, aimg.data(), abytes, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && mbytes)
        e = cudaMemcpy(static_cast<char*>(arena) + abytes, meta.data(), mbytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        if (arena) cudaFree(arena);
        bsgemm_destroy(h);
        fail(BSGEMM_ERR_CUDA, cuda_msg("tensor-core operands", e));
        return nullptr;
    }
    h->tc_arena = arena;
    h->tc_aimg = static_cast<const unsigned char*>(arena);
    h->tc_meta = mbytes ? reinterpret_cast<const uint32_t*>(static_cast<const char*>(arena) + abytes) : nullptr;
    h->tc_dense = dense;
    h->tc_bytes = abytes + mbytes;
    return h;
}

extern "C" {

uint32_t bsgemm_set_test_hooks(uint32_t bits) { return g_test_hooks.exchange(bits); }

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
    if (N < 1 || K < 1) {
        fail(BSGEMM_ERR_INVALID, "need N >= 1 and K >= 1");
        return nullptr;
    }
    if (N > BSGEMM_MAX_N) {  // block-row indices are 16-bit fields in the kernel's group window
        fail(BSGEMM_ERR_UNSUPPORTED, "N = " + std::to_string(N) + " exceeds " + std::to_string(BSGEMM_MAX_N));
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
    const int nbr = (N + BSGEMM_BLOCK - 1) / BSGEMM_BLOCK;  // the last block-row may hold fewer than 4 rows
    const int npad = BSGEMM_BLOCK * nbr;
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

    // Repack into row groups and steps.  Block-rows sorted by stored-block
    // count (longest first, ties by index) are taken 4 at a time, so a
    // group's block-rows need about the same number of quads; the columns
    // of each step are ordered by order_steps.
    const int ngroups = (nbr + 3) / 4;
    std::vector<int> rows_sorted(nbr);
    for (int r = 0; r < nbr; ++r) rows_sorted[r] = r;
    std::stable_sort(rows_sorted.begin(), rows_sorted.end(),
                     [&](int x, int y) { return indptr[x + 1] - indptr[x] > indptr[y + 1] - indptr[y]; });
    std::vector<int32_t> grow(static_cast<size_t>(ngroups) * 4, -1);
    std::vector<int32_t> gptr(ngroups + 1, 0);
    std::vector<int32_t> cost(ngroups + 1, 0);
    for (int gi = 0; gi < ngroups; ++gi) {
        int quads = 0;
        for (int q = 0; q < 4 && 4 * gi + q < nbr; ++q) {
            const int r = rows_sorted[4 * gi + q];
            grow[4 * gi + q] = r;
            quads = std::max(quads, (indptr[r + 1] - indptr[r] + 3) / 4);
        }
        quads = (quads + bsg::kBlock - 1) / bsg::kBlock * bsg::kBlock;  // whole blocks of the kernel's ring
        gptr[gi + 1] = gptr[gi] + quads;
        cost[gi + 1] = static_cast<int32_t>(cost[gi] + quads + (quads > 0 ? kGroupCost : 0));
    }
    const int S = gptr[ngroups];
    // 128-byte step records: each step's columns in the order order_steps
    // gives, its channel words beside them.
    std::vector<int32_t> recs(static_cast<size_t>(S + bsg::kStepPad) * 32, 0);
    {
        std::vector<int32_t> ent;
        order_steps(indptr, colidx, ngroups, grow, gptr, bsg::bank_key, ent);
        for (int s = 0; s < S; ++s) {
            int32_t* rec = &recs[static_cast<size_t>(s) * 32];
            uint32_t wwords[4][4] = {};
            step_entries(ent.data() + 16 * static_cast<size_t>(s), colidx, values, bsg::tile_row_offset, rec, wwords);
            for (int q = 0; q < 4; ++q)
                for (int c = 0; c < 4; ++c) rec[16 + 4 * q + c] = static_cast<int32_t>(wwords[q][c]);
        }
    }
    Repacked rp;
    rp.shape = kShape4x1;
    rp.N = N;
    rp.K = K;
    rp.nnzb = nnzb;
    rp.ngroups = ngroups;
    rp.S = S;
    rp.grow = std::move(grow);
    rp.gptr = std::move(gptr);
    rp.cost = std::move(cost);
    rp.recs = std::move(recs);
    return upload(rp, scales, bias);
}

// Weights sparse in 1 x 4 blocks (one output row x 4 consecutive input
// columns), repacked for the layer kernel's 1 x 4 form: rows sorted by block
// count (longest first, ties by index) are taken 4 at a time into a group;
// a step holds one block of each of the group's 4 rows (a "quad" = the
// block's 4 columns, its one weight word), and a group has as many steps as
// its longest row has blocks, rounded up to a multiple of kBlock.  In each
// half of a step (the blocks of rows 2h and 2h + 1: one pass of the
// shared-memory gather) one block has an even and one an odd column group
// where the rows allow it: the 4 columns of an even group sit on bank keys
// {0, 1, 4, 5} of the swizzled tile, of an odd group on {2, 3, 6, 7}.
bsgemm_t bsgemm_create_1x4(int N, int K, const int32_t* indices, const int8_t* values, const float* scales,
                           const float* bias) {
    clear_error();
    if (N < 1 || N > 65535 || K < 4 || K % 4 != 0) {
        fail(BSGEMM_ERR_INVALID, "need 1 <= N <= 65535 and K >= 4 a multiple of 4");
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
    const int ng4 = K / 4;  // column groups
    const int32_t* indptr = indices;
    const int32_t* colgrp = indices + N + 1;
    const int64_t nnz = indptr[N];
    if (indptr[0] != 0 || nnz < 0 || nnz > static_cast<int64_t>(N) * ng4) {
        fail(BSGEMM_ERR_INVALID, "indptr[0] must be 0 and 0 <= indptr[N] <= N * K / 4");
        return nullptr;
    }
    if (nnz > 0 && !values) {
        fail(BSGEMM_ERR_INVALID, "values must not be NULL when blocks are stored");
        return nullptr;
    }
    for (int n = 0; n < N; ++n) {
        if (indptr[n + 1] < indptr[n]) {
            fail(BSGEMM_ERR_INVALID, "indptr must be non-decreasing (row " + std::to_string(n) + ")");
            return nullptr;
        }
        for (int e = indptr[n]; e < indptr[n + 1]; ++e) {
            if (colgrp[e] < 0 || colgrp[e] >= ng4 || (e > indptr[n] && colgrp[e - 1] >= colgrp[e])) {
                fail(BSGEMM_ERR_INVALID, "column groups must lie in [0, K/4) and strictly increase within row " +
                                             std::to_string(n));
                return nullptr;
            }
        }
        if (!std::isfinite(scales[n]) || (bias && !std::isfinite(bias[n]))) {
            fail(BSGEMM_ERR_INVALID, "scales and bias must be finite (channel " + std::to_string(n) + ")");
            return nullptr;
        }
    }
    Repacked rp;
    rp.shape = kShape1x4;
    rp.N = N;
    rp.K = K;
    rp.nnzb = nnz;
    rp.ngroups = (N + 3) / 4;
    std::vector<int> rows(N);
    for (int n = 0; n < N; ++n) rows[n] = n;
    std::stable_sort(rows.begin(), rows.end(),
                     [&](int x, int y) { return indptr[x + 1] - indptr[x] > indptr[y + 1] - indptr[y]; });
    rp.grow.assign(static_cast<size_t>(rp.ngroups) * 4, -1);
    rp.gptr.assign(rp.ngroups + 1, 0);
    rp.cost.assign(rp.ngroups + 1, 0);
    for (int gi = 0; gi < rp.ngroups; ++gi) {
        int steps = 0;
        for (int q = 0; q < 4 && 4 * gi + q < N; ++q) {
            rp.grow[4 * gi + q] = rows[4 * gi + q];
            steps = std::max(steps, indptr[rows[4 * gi + q] + 1] - indptr[rows[4 * gi + q]]);
        }
        steps = (steps + bsg::kBlock - 1) / bsg::kBlock * bsg::kBlock;
        rp.gptr[gi + 1] = rp.gptr[gi] + steps;
        rp.cost[gi + 1] = static_cast<int32_t>(rp.cost[gi] + steps + (steps > 0 ? kGroupCost : 0));
    }
    rp.S = rp.gptr[rp.ngroups];
    rp.recs.assign(static_cast<size_t>(rp.S + bsg::kStepPad) * 32, 0);
    const int pad_grp[2] = {0, ng4 > 1 ? 1 : 0};  // padding blocks: column group 0 (even) or 1 (odd)
    std::vector<int> left[4][2];                   // a row's remaining blocks by column-group parity
    for (int gi = 0; gi < rp.ngroups; ++gi) {
        for (int q = 0; q < 4; ++q) {
            left[q][0].clear();
            left[q][1].clear();
            const int n = rp.grow[4 * gi + q];
            if (n < 0) continue;
            for (int e = indptr[n + 1] - 1; e >= indptr[n]; --e) left[q][colgrp[e] & 1].push_back(e);
        }
        for (int st = rp.gptr[gi]; st < rp.gptr[gi + 1]; ++st) {
            int32_t* rec = &rp.recs[static_cast<size_t>(st) * 32];
            for (int h = 0; h < 2; ++h) {
                const int qa = 2 * h, qb = 2 * h + 1;
                // parity of row qa's block this step: the pairing (pa, 1 - pa)
                // that both rows can serve, from the fuller lists first
                auto have = [&](int q, int par) { return !left[q][par].empty(); };
                int pa;
                const bool ok0 = have(qa, 0) && have(qb, 1), ok1 = have(qa, 1) && have(qb, 0);
                if (ok0 && ok1)
                    pa = left[qa][0].size() + left[qb][1].size() >= left[qa][1].size() + left[qb][0].size() ? 0 : 1;
                else if (ok0 || ok1)
                    pa = ok0 ? 0 : 1;
                else  // one row (or neither) has blocks left: it takes its fuller list, the other pads opposite
                    pa = have(qa, 0) || have(qa, 1) ? (left[qa][0].size() >= left[qa][1].size() ? 0 : 1)
                                                     : (have(qb, 0) || have(qb, 1)
                                                            ? 1 - (left[qb][0].size() >= left[qb][1].size() ? 0 : 1)
                                                            : 0);
                for (int x = 0; x < 2; ++x) {
                    const int q = x == 0 ? qa : qb;
                    const int par = x == 0 ? pa : 1 - pa;
                    int blk = -1;
                    if (have(q, par)) {
                        blk = left[q][par].back();
                        left[q][par].pop_back();
                    } else if (have(q, 1 - par)) {  // a conflict rather than an extra step
                        blk = left[q][1 - par].back();
                        left[q][1 - par].pop_back();
                    }
                    const int j = blk >= 0 ? colgrp[blk] : pad_grp[par];
                    uint32_t word = 0;
                    if (blk >= 0)
                        for (int e = 0; e < 4; ++e)
                            word |= static_cast<uint32_t>(static_cast<uint8_t>(values[static_cast<size_t>(blk) * 4 + e]))
                                    << (8 * e);
                    for (int e = 0; e < 4; ++e) rec[4 * q + e] = static_cast<int32_t>(bsg::tile_row_offset(4 * j + e));
                    rec[16 + 4 * q] = static_cast<int32_t>(word);  // w[q][0]; w[q][1..3] stay 0
                }
            }
        }
    }
    return upload(rp, scales, bias);
}

// 2:4-sparse weights: run as the 4 x 1 blocks that hold their values (a
// block (r, k) is stored when one of rows 4r..4r+3 has a nonzero value in
// column k), through the 4 x 1 path.
bsgemm_t bsgemm_create_2to4(int N, int K, const int8_t* values, const uint8_t* idx, const float* scales,
                            const float* bias) {
    clear_error();
    if (N < 1 || K < 4 || K % 4 != 0 || !values || !idx) {
        fail(BSGEMM_ERR_INVALID, "need N >= 1, K >= 4 a multiple of 4, and values and idx");
        return nullptr;
    }
    const int half = K / 2;
    const int nbr = (N + 3) / 4;
    std::vector<int8_t> dense(static_cast<size_t>(nbr) * 4 * K, 0);
    for (int n = 0; n < N; ++n) {
        for (int gj = 0; gj < K / 4; ++gj) {
            const size_t p = static_cast<size_t>(n) * half + 2 * gj;
            const int i0 = idx[p], i1 = idx[p + 1];
            if (i0 >= i1 || i1 > 3) {
                fail(BSGEMM_ERR_INVALID, "2:4 positions must strictly increase within [0, 4) (row " +
                                             std::to_string(n) + ", group " + std::to_string(gj) + ")");
                return nullptr;
            }
            dense[static_cast<size_t>(n) * K + 4 * gj + i0] = values[p];
            dense[static_cast<size_t>(n) * K + 4 * gj + i1] = values[p + 1];
        }
    }
    std::vector<int32_t> indices(nbr + 1, 0);
    std::vector<int8_t> vals;
    std::vector<int32_t> cols;
    for (int r = 0; r < nbr; ++r) {
        for (int k = 0; k < K; ++k) {
            int8_t v[4];
            bool any = false;
            for (int c = 0; c < 4; ++c) {
                v[c] = dense[static_cast<size_t>(4 * r + c) * K + k];
                any = any || v[c] != 0;
            }
            if (!any) continue;
            cols.push_back(k);
            vals.insert(vals.end(), v, v + 4);
        }
        indices[r + 1] = static_cast<int32_t>(cols.size());
    }
    indices.insert(indices.end(), cols.begin(), cols.end());
    bsgemm_t h = bsgemm_create(N, K, BSGEMM_BLOCK, indices.data(), vals.empty() ? nullptr : vals.data(), scales, bias);
    if (!h || N % 128 != 0 || K % 128 != 0 || K > 4096) return h;

    // The sparse tensor cores' operands.  Per (channel tile ct, stage s of
    // 128 columns): the stored values of rows 128 ct .. + 127 and columns
    // 128 s .. + 127 as the shared-memory image the MMA reads (row m: 64 f16,
    // element e = 2 (group - 32 s) + t in 16-byte chunk e / 8, placed at chunk
    // (e / 8) ^ (m % 8) of the row's 128 bytes); and the metadata of its 4
    // MMAs (MMA i: columns 128 s + 32 i .. + 31, 8 groups): row m's word has
    // nibble g = first position | second position << 2 of group 8 i + g, and
    // within every 16 rows the tensor memory lanes hold (lane r < 8: row r's
    // groups 0-3 | row r + 8's groups 0-3; lane 8 + r: row r's groups 4-7 |
    // row r + 8's groups 4-7) -- the layout tcgen05.mma.sp reads.
    const int ntile = N / 128, nst = K / 128;
    std::vector<uint16_t> aimg(static_cast<size_t>(ntile) * nst * (bsg::kTc24AImage / 2), 0);
    std::vector<uint32_t> meta(static_cast<size_t>(ntile) * nst * 128 * 4, 0);
    for (int ct = 0; ct < ntile; ++ct) {
        for (int st = 0; st < nst; ++st) {
            uint16_t* img = &aimg[(static_cast<size_t>(ct) * nst + st) * (bsg::kTc24AImage / 2)];
            uint32_t word[4][128];
            for (int m = 0; m < 128; ++m) {
                const int n = 128 * ct + m;
                for (int e = 0; e < 64; ++e) {
                    const size_t p = static_cast<size_t>(n) * half + 64 * st + e;
                    const int c = e / 8;
                    img[(128 * m + 16 * (c ^ (m % 8))) / 2 + e % 8] = f16_of_int(values[p]);
                }
                for (int i = 0; i < 4; ++i) {
                    uint32_t w = 0;
                    for (int g = 0; g < 8; ++g) {
                        const size_t p = static_cast<size_t>(n) * half + 64 * st + 16 * i + 2 * g;
                        w |= static_cast<uint32_t>(idx[p] | (idx[p + 1] << 2)) << (4 * g);
                    }
                    word[i][m] = w;
                }
            }
            uint32_t* mt = &meta[(static_cast<size_t>(ct) * nst + st) * 128 * 4];
            for (int i = 0; i < 4; ++i) {
                for (int b16 = 0; b16 < 128; b16 += 16) {
                    for (int r = 0; r < 8; ++r) {
                        const uint32_t lo = word[i][b16 + r], hi = word[i][b16 + 8 + r];
                        mt[4 * (b16 + r) + i] = (lo & 0xFFFFu) | (hi << 16);
                        mt[4 * (b16 + 8 + r) + i] = (lo >> 16) | (hi & 0xFFFF0000u);
                    }
                }
            }
        }
    }
    return attach_tc(h, aimg, meta, false);
}

// Any block-compressed weight, also run dense over K on the tensor cores
// (launch_tc_linear, dense form) when N and K are multiples of 128: per
// (channel tile ct, stage s of 128 columns) the weight's 128 x 128 values
// as f16, row m = channel 128 ct + m, in two sub-tiles of 64 columns, the
// 16-byte chunk c of a sub-tile row placed at chunk c ^ (m % 8) of its 128
// bytes; zero where no block is stored.
bsgemm_t bsgemm_create_tc(int N, int K, int block, const int32_t* indices, const int8_t* values, const float* scales,
                          const float* bias) {
    bsgemm_t h = bsgemm_create(N, K, block, indices, values, scales, bias);
    if (!h || N % 128 != 0 || K % 128 != 0 || K > 4096) return h;
    const int nbr = N / 4, nst = K / 128;
    constexpr size_t kImg = bsg::kTcDenseAImage / 2;  // f16 values per (tile, stage)
    std::vector<uint16_t> aimg(static_cast<size_t>(N / 128) * nst * kImg, 0);
    const int32_t* indptr = indices;
    const int32_t* colidx = indices + nbr + 1;
    for (int r = 0; r < nbr; ++r) {
        for (int j = indptr[r]; j < indptr[r + 1]; ++j) {
            const int k = colidx[j], st = k / 128, kk = k % 128, c = (kk % 64) / 8;
            for (int i = 0; i < 4; ++i) {
                const int n = 4 * r + i, m = n % 128;
                aimg[(static_cast<size_t>(n / 128) * nst + st) * kImg + (kk / 64) * (kImg / 2) + 64 * m +
                     8 * (c ^ (m % 8)) + kk % 8] = f16_of_int(values[4 * static_cast<size_t>(j) + i]);
            }
        }
    }
    return attach_tc(h, aimg, std::vector<uint32_t>(), true);
}

// mode: 0 = gather from act (no scratch), 1 = relayout act into workspace
// then stage tiles, 2 = stage tiles already in workspace (act unused),
// 3 = act is x^T [K][M] with row stride ld (no scratch).  Modes 0 and 1
// stage from act by tensor copies instead when tensor_staging() allows.
static int run_common(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                      size_t workspace_bytes, int mode, void* stream, int ld = 0) {
    const bool use_ws = mode == 1 || mode == 2;
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    if (M < 0) return fail(BSGEMM_ERR_INVALID, "M must be >= 0");
    if (epi.kind < BSGEMM_OUT_I32 || epi.kind > BSGEMM_OUT_F32_RESID)
        return fail(BSGEMM_ERR_INVALID, "unknown epilogue kind " + std::to_string(epi.kind));
    if (epi.kind == BSGEMM_OUT_F32_RESID && M > 0) {
        if (!epi.residual || reinterpret_cast<uintptr_t>(epi.residual) % 4 != 0)
            return fail(BSGEMM_ERR_INVALID, "the residual must be a 4-byte aligned device array");
        if (!std::isfinite(epi.residual_scale)) return fail(BSGEMM_ERR_INVALID, "residual_scale must be finite");
    }
    if (h->shape == kShape1x4 && epi.kind == BSGEMM_OUT_F32_RESID)
        return fail(BSGEMM_ERR_UNSUPPORTED, "the residual epilogue takes 4 x 1-block weights");
    if (epi.flags & ~static_cast<uint32_t>(BSGEMM_ACT_READY))
        return fail(BSGEMM_ERR_INVALID, "unknown bits in epi.flags");
    float inv = 0.0f;
    if (epi.kind == BSGEMM_OUT_I8 || epi.kind == BSGEMM_OUT_I8_GELU) {
        if (!(epi.out_scale > 0.0f) || !std::isfinite(epi.out_scale))
            return fail(BSGEMM_ERR_INVALID, "out_scale must be finite and > 0 for int8 outputs");
        inv = 1.0f / epi.out_scale;
        if (!std::isfinite(inv)) return fail(BSGEMM_ERR_INVALID, "1 / out_scale overflows fp32");
    }
    if (mode == 3 && M > 0) {
        if (ld < M || ld % 16 != 0) return fail(BSGEMM_ERR_INVALID, "ld must be >= M and a multiple of 16");
        if (reinterpret_cast<uintptr_t>(act) % 16 != 0) return fail(BSGEMM_ERR_INVALID, "act must be 16-byte aligned");
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

    // With K a multiple of 16 and act 16-byte aligned the layer kernel stages
    // its tiles from act itself (tensor copies); the relayout kernel and the
    // workspace serve the other shapes and bsgemm_run_tiled.
    const bool tensor = (mode == 0 || mode == 1) && bsg::tensor_staging(h->w.K, act);
    bsg::LaunchArgs a{};
    a.x = act;
    a.xb = use_ws && !tensor ? static_cast<const int8_t*>(workspace) : nullptr;
    a.tensor = tensor;
    a.kmajor = mode == 3;
    a.ld = ld;
    a.act_ready = (epi.flags & BSGEMM_ACT_READY) != 0 && (tensor || mode == 3);
    a.res = epi.residual;
    a.res_scale = epi.residual_scale;
    a.out = out;
    a.M = M;
    a.kind = epi.kind;
    a.shape = h->shape;
    a.inv_out_scale = inv;
    a.x_vec16 = (reinterpret_cast<uintptr_t>(act) % 16 == 0) && (h->w.K % 16 == 0);
    a.skip_copy = (g_test_hooks.load() & BSGEMM_TEST_SKIP_TILE_COPY) != 0;
    a.wait_limit = a.skip_copy ? 64u : 0u;
    // weights on the tensor cores (2:4 sparse, or dense over K): row-major
    // act, any kind but the residual
    if (h->tc_aimg && (mode == 0 || mode == 1) && epi.kind != BSGEMM_OUT_F32_RESID &&
        (reinterpret_cast<uintptr_t>(act) & 15u) == 0) {
        e = bsg::launch_tc_linear(act, M, h->w.N, h->w.K, h->tc_aimg, h->tc_meta, h->tc_dense, h->w.scale, h->w.bias,
                                  out, epi.kind, inv, (epi.flags & BSGEMM_ACT_READY) != 0, h->w.status, s);
        if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("tensor-core kernel launch", e));
        return BSGEMM_OK;
    }
    const long long ntiles = (static_cast<long long>(M) + bsg::kTile - 1) / bsg::kTile;
    const long long upt = h->w.ngroups;  // units per token tile
    long long cap = static_cast<long long>(h->num_sms) * h->ctas_per_sm;
    if (cap > bsg::kMaxGrid) cap = bsg::kMaxGrid;
    bsg::Schedule sched;
    int grid = 0;
    {
        std::lock_guard<std::mutex> lock(h->sched_mu);
        if (h->sched_m != M) {
            h->sched_grid = make_schedule(h->cost, upt, ntiles, static_cast<int>(cap), tile_cost(h->w.K), h->sched);
            h->sched_m = M;
        }
        grid = h->sched_grid;
        std::memcpy(sched.u, h->sched.u, sizeof(long long) * (grid + 1));
    }
    if (mode == 1 && !tensor) {
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

int bsgemm_run_kmajor(bsgemm_t h, const int8_t* act_t, int M, int ld, void* out, bsgemm_epilogue epi, void* stream) {
    return run_common(h, act_t, M, out, epi, nullptr, 0, 3, stream, ld);
}

int bsgemm_run_tiled(bsgemm_t h, const void* tiles, size_t tiles_bytes, int M, void* out, bsgemm_epilogue epi,
                     void* stream) {
    return run_common(h, nullptr, M, out, epi, const_cast<void*>(tiles), tiles_bytes, 2, stream);
}

int bsgemm_run_static(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* stream) {
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    // With K % 16 == 0 and act 16-byte aligned the layer kernel stages its
    // tiles itself and the scratch is not touched: bsgemm_run's one kernel,
    // with no limit on M.
    if (bsg::tensor_staging(h->w.K, act)) return run_common(h, act, M, out, epi, nullptr, 0, 0, stream);
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

// Workspace of bsgemm_run_host: [act copy | token tiles | device result],
// each part at a 256-byte aligned offset.  Returns 0 for an unknown kind.
static size_t host_parts(bsgemm_t h, int M, int32_t kind, size_t* off_tiles, size_t* off_out, size_t* out_bytes) {
    static const size_t elem[6] = {4, 4, 4, 1, 1, 4};
    if (kind < BSGEMM_OUT_I32 || kind > BSGEMM_OUT_F32_RESID) return 0;
    const size_t m = static_cast<size_t>(M);
    *off_tiles = align_up(m * static_cast<size_t>(h->w.K), 256);
    *off_out = *off_tiles + align_up(bsg::tiled_bytes(h->w.K, M), 256);
    *out_bytes = m * static_cast<size_t>(h->w.N) * elem[kind];
    return *off_out + *out_bytes;
}

size_t bsgemm_host_workspace_bytes(bsgemm_t h, int M, int32_t kind) {
    if (!h || M <= 0) return 0;
    size_t ot = 0, oo = 0, ob = 0;
    return host_parts(h, M, kind, &ot, &oo, &ob);
}

int bsgemm_run_host(bsgemm_t h, const int8_t* act, int M, void* out, bsgemm_epilogue epi, void* workspace,
                    size_t workspace_bytes, void* stream) {
    clear_error();
    if (!h) return fail(BSGEMM_ERR_INVALID, "NULL handle");
    if (M < 0) return fail(BSGEMM_ERR_INVALID, "M must be >= 0");
    if (epi.kind < BSGEMM_OUT_I32 || epi.kind > BSGEMM_OUT_F32_RESID)
        return fail(BSGEMM_ERR_INVALID, "unknown epilogue kind " + std::to_string(epi.kind));
    if (M == 0) return BSGEMM_OK;
    if (!act || !out) return fail(BSGEMM_ERR_INVALID, "act and out must not be NULL");
    size_t off_tiles = 0, off_out = 0, out_bytes = 0;
    const size_t need = host_parts(h, M, epi.kind, &off_tiles, &off_out, &out_bytes);
    if (!workspace || workspace_bytes < need)
        return fail(BSGEMM_ERR_INVALID, "workspace must hold bsgemm_host_workspace_bytes(h, M, kind) = " +
                                            std::to_string(need) + " bytes");
    if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
        return fail(BSGEMM_ERR_INVALID, "workspace must be 16-byte aligned");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("cudaGetDevice", e));
    if (dev != h->device)
        return fail(BSGEMM_ERR_INVALID, "current device " + std::to_string(dev) + " is not the handle's device " +
                                            std::to_string(h->device));
    char* ws = static_cast<char*>(workspace);
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    e = cudaMemcpyAsync(ws, act, static_cast<size_t>(M) * static_cast<size_t>(h->w.K), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("copy of act to the device", e));
    bsgemm_epilogue e2 = epi;
    e2.flags |= BSGEMM_ACT_READY;  // the copy above completes before the kernel starts (stream order)
    const int rc = run_common(h, reinterpret_cast<const int8_t*>(ws), M, ws + off_out, e2, ws + off_tiles,
                              off_out - off_tiles, 1, stream);
    if (rc != BSGEMM_OK) return rc;
    e = cudaMemcpyAsync(out, ws + off_out, out_bytes, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("copy of the result to the host", e));
    return BSGEMM_OK;
}

int64_t bsgemm_block_prune(int N, int K, const float* W, double sparsity, uint8_t* keep, void* stream) {
    clear_error();
    if (N < 4 || N % 4 != 0 || K < 1) return fail(BSGEMM_ERR_INVALID, "N must be a positive multiple of 4 and K >= 1");
    if (!W || !keep) return fail(BSGEMM_ERR_INVALID, "W and keep must not be NULL");
    if (!(sparsity >= 0.0 && sparsity <= 1.0)) return fail(BSGEMM_ERR_INVALID, "sparsity must lie in [0, 1]");
    const long long total = static_cast<long long>(N / 4) * K;
    long long npruned = static_cast<long long>(std::floor(sparsity * static_cast<double>(total) + 0.5));
    if (npruned > total) npruned = total;
    int dev = -1, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("device query", e));
    bool bad = false;
    e = bsg::block_prune(W, N, K, npruned, keep, sms, static_cast<cudaStream_t>(stream), &bad);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("block pruning", e));
    if (bad) return fail(BSGEMM_ERR_INVALID, "W holds a value that is not finite");
    return total - npruned;
}

int bsgemm_layernorm(const float* z, int M, int N, const float* gamma, const float* beta, float eps, void* out,
                     bsgemm_epilogue epi, void* stream) {
    clear_error();
    if (M < 0 || N < 1) return fail(BSGEMM_ERR_INVALID, "need M >= 0 and N >= 1");
    if (epi.kind != BSGEMM_OUT_F32 && epi.kind != BSGEMM_OUT_I8)
        return fail(BSGEMM_ERR_INVALID, "LayerNorm writes BSGEMM_OUT_F32 or BSGEMM_OUT_I8");
    if (!(eps >= 0.0f) || !std::isfinite(eps)) return fail(BSGEMM_ERR_INVALID, "eps must be finite and >= 0");
    float inv = 0.0f;
    if (epi.kind == BSGEMM_OUT_I8) {
        if (!(epi.out_scale > 0.0f) || !std::isfinite(epi.out_scale))
            return fail(BSGEMM_ERR_INVALID, "out_scale must be finite and > 0 for int8 outputs");
        inv = 1.0f / epi.out_scale;
        if (!std::isfinite(inv)) return fail(BSGEMM_ERR_INVALID, "1 / out_scale overflows fp32");
    }
    if (M == 0) return BSGEMM_OK;
    if (!z || !gamma || !beta || !out) return fail(BSGEMM_ERR_INVALID, "z, gamma, beta and out must not be NULL");
    const cudaError_t e = bsg::launch_layernorm(z, M, N, gamma, beta, eps, epi.kind, inv, out,
                                                static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("LayerNorm launch", e));
    return BSGEMM_OK;
}

int bsgemm_attention(const int8_t* qkv, int batch, int seq, int heads, int head_dim, int ld, float qkv_scale,
                     void* out, bsgemm_epilogue epi, void* stream) {
    clear_error();
    if (batch < 0 || batch > 65535 || heads < 1 || heads > 65535 || seq < 0)
        return fail(BSGEMM_ERR_INVALID, "need 0 <= batch <= 65535, 1 <= heads <= 65535 and seq >= 0");
    if (head_dim != 64) return fail(BSGEMM_ERR_UNSUPPORTED, "head_dim must be 64");
    if (seq > BSGEMM_ATTN_MAX_SEQ)
        return fail(BSGEMM_ERR_UNSUPPORTED, "seq exceeds BSGEMM_ATTN_MAX_SEQ = " + std::to_string(BSGEMM_ATTN_MAX_SEQ));
    if (epi.kind != BSGEMM_OUT_F32 && epi.kind != BSGEMM_OUT_I8)
        return fail(BSGEMM_ERR_INVALID, "attention writes BSGEMM_OUT_F32 or BSGEMM_OUT_I8");
    if (epi.flags & ~static_cast<uint32_t>(BSGEMM_ACT_READY))
        return fail(BSGEMM_ERR_INVALID, "unknown bits in epi.flags");
    const long long d = static_cast<long long>(heads) * head_dim;
    if (ld < 3 * d || ld % 16 != 0) return fail(BSGEMM_ERR_INVALID, "ld must be >= 3 * heads * head_dim and a multiple of 16");
    if (static_cast<long long>(batch) * seq > INT32_MAX) return fail(BSGEMM_ERR_INVALID, "batch * seq exceeds 2^31 - 1");
    if (!(qkv_scale > 0.0f) || !std::isfinite(qkv_scale)) return fail(BSGEMM_ERR_INVALID, "qkv_scale must be finite and > 0");
    const double c = static_cast<double>(qkv_scale) * qkv_scale / std::sqrt(static_cast<double>(head_dim));
    if (!(c >= static_cast<double>(FLT_MIN)) || !(c < 0x1p100))
        return fail(BSGEMM_ERR_INVALID, "qkv_scale^2 / sqrt(head_dim) must be a normal fp32 number below 2^100");
    float inv = 0.0f;
    if (epi.kind == BSGEMM_OUT_I8) {
        if (!(epi.out_scale > 0.0f) || !std::isfinite(epi.out_scale))
            return fail(BSGEMM_ERR_INVALID, "out_scale must be finite and > 0 for int8 outputs");
        inv = 1.0f / epi.out_scale;
        if (!std::isfinite(inv)) return fail(BSGEMM_ERR_INVALID, "1 / out_scale overflows fp32");
    }
    if (batch == 0) return BSGEMM_OK;
    if (seq < 1) return fail(BSGEMM_ERR_INVALID, "seq must be >= 1");
    if (!qkv || !out) return fail(BSGEMM_ERR_INVALID, "qkv and out must not be NULL");
    if ((reinterpret_cast<uintptr_t>(qkv) & 15u) || (reinterpret_cast<uintptr_t>(out) & 15u))
        return fail(BSGEMM_ERR_INVALID, "qkv and out must be 16-byte aligned");
    const cudaError_t e = bsg::launch_attention(qkv, batch, seq, heads, ld, static_cast<float>(c), qkv_scale, epi.kind,
                                                inv, out, (epi.flags & BSGEMM_ACT_READY) != 0,
                                                static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("attention launch", e));
    return BSGEMM_OK;
}

int bsgemm_attention_status(int clear) {
    clear_error();
    unsigned v = 0;
    const cudaError_t e = bsg::attention_status(clear != 0, &v);
    if (e != cudaSuccess) return fail(BSGEMM_ERR_CUDA, cuda_msg("reading the attention status", e));
    return static_cast<int>(v);
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
    if (h->tc_arena) cudaFree(h->tc_arena);
    delete h;
}

int bsgemm_info(bsgemm_t h, int64_t* out, int n) {
    clear_error();
    if (!h || (!out && n > 0)) return fail(BSGEMM_ERR_INVALID, "NULL handle or output");
    const int64_t v[7] = {h->w.N, h->w.K, h->nnzb, 4 * static_cast<int64_t>(h->w.S), bsg::kTile,
                          static_cast<int64_t>(h->num_sms) * h->ctas_per_sm, static_cast<int64_t>(h->arena_bytes + h->tc_bytes)};
    for (int i = 0; i < n && i < 7; ++i) out[i] = v[i];
    return 7;
}

}  // extern "C"
