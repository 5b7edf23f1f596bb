// Internal declarations shared by the host API (bsgemm_api.cpp) and the
// kernels (bsgemm_kernel.cu).  Not part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace bsg {

// Token tile: the layer kernel holds kTile tokens x all K columns of the
// activations in shared memory.
constexpr int kTile = 64;

// Shared-memory layout of one token tile ("swizzled k-major").  Column k of
// the activations is a row of 64 bytes (the tile's 64 tokens), cut into 4
// chunks of 16 tokens.  Rows 2i and 2i+1 share the 128-byte line i; chunk c
// of row k sits in 16-byte slot ((4 (k & 1) + c) XOR (i & 3)) of its line.
// Row k's chunk 0 is therefore at byte tile_row_offset(k), and chunk c at
// tile_row_offset(k) XOR 16 c.  The XOR spreads the chunks of different rows
// over the 8 bank groups of shared memory, so a gather of 8 rows whose
// "bank keys" (slot of chunk 0) differ reads in one pass.  It is also the
// 64-byte swizzle of the tensor copies: a box of 64-byte rows k lands in
// exactly this layout (row k at 64 k, chunk c at slot c XOR ((k >> 1) & 3)).
inline uint32_t tile_row_offset(int k) {
    const uint32_t line = static_cast<uint32_t>(k) >> 1;
    const uint32_t slot = ((static_cast<uint32_t>(k) & 1u) << 2) ^ (line & 3u);
    return (line << 7) | (slot << 4);
}
inline int bank_key(int k) { return static_cast<int>((tile_row_offset(k) >> 4) & 7u); }

// Device form of one block-compressed weight (built once by bsgemm_create).
//
// A block-row r holds output rows 4r..4r+3.  Block-rows are sorted by their
// number of stored blocks and taken 4 at a time into "row groups"
// (grow[gi] = the group's block-rows, -1 where the last group has fewer
// than 4).  A group is processed in steps; step s of group gi (gptr[gi] <=
// s < gptr[gi+1]) holds one quad -- 4 stored columns, the analogue of
// Algorithm 1's k_block = 4 -- of each of the group's 4 block-rows, as a
// 128-byte record (8 int4):
//   int32 off[16]  : tile_row_offset(k_e) of its 16 columns; columns 4q..4q+3
//                    belong to the group's block-row q
//   uint32 w[4][4] : w[q][c] = bytes W[4 r_q + c][k_{4q}] .. W[4 r_q + c][k_{4q+3}],
//                    one dot-4 operand per output channel c of block-row q
// A group has as many steps as its longest block-row has quads, rounded up
// to a multiple of kBlock; shorter block-rows and the extra steps are padded
// with zero-weight entries whose columns are valid tile rows.  Within each half of a step (columns 0-7, 8-15) the columns'
// bank keys differ wherever the two block-rows' columns allow it.
struct DeviceWeights {
    const int32_t* gptr;   // [ngroups + 1]
    const int4* grow;      // [ngroups]
    const int4* recs;      // [8 * (S + kStepPad)]
    const float* scale;    // [N]
    const float* bias;     // [N]
    int* status;           // device status word (bounded-wait timeouts), 0 = fine
    int N, K, ngroups, S;
};

// Device status bits written by the kernels.
constexpr int kStatusTimeout = 1;  // a bounded wait on an asynchronous copy gave up

struct LaunchArgs {
    const int8_t* x;       // [M][K]
    const int8_t* xb;      // NULL, or x re-laid as swizzled token tiles: [ntiles][kpad * kTile bytes]
    void* out;             // [M][N]
    int M;
    int kind;
    float inv_out_scale;
    bool x_vec16;          // x 16-byte aligned and K % 16 == 0
    bool tensor;           // stage tiles from x by tensor copies (xb unused; needs tensor_staging())
    bool kmajor;           // x is x^T [K][M] with row stride ld: tensor copies, no transpose
    bool act_ready;        // x may be read before the previous kernel completes (BSGEMM_ACT_READY)
    const int8_t* res;     // kind 5: int8 residual [M][N]
    float res_scale;       // kind 5: the residual's scale
    int ld;                // row stride of x^T in bytes (kmajor only)
    int shape;             // block shape of the weight: 0 = 4 x 1 blocks, 1 = 1 x 4 blocks
    int box_d;             // 64-column boxes per tensor copy (set by launch: >1 with a 3-D map of x)
    unsigned wait_limit;   // polls of a wait on a tile copy before it gives up (0: the default)
    bool skip_copy;        // test hook: issue no tile copy, so that every such wait gives up
};

// Kernel configuration: 8 warps per CTA (2 per SM sub-partition, up to 255
// registers a thread).
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
#ifndef BSG_RING
#define BSG_RING 12
#endif
constexpr int kRing = BSG_RING;     // step records a warp keeps in flight (registers): 3 blocks
constexpr int kBlock = kRing / 3;   // every row group holds a multiple of kBlock steps (zero-weight padding)
constexpr int kStepPad = kRing;     // zero step records after the last one (the record prefetch runs ahead)
constexpr int kGroupWin = 128;      // row groups whose step offsets and block-rows a CTA keeps in shared memory
constexpr int kMaxBoxes = 49;       // 64-column boxes of a token tile (K <= 3136)
constexpr int kStaticSmem = 2304;   // bytes of static shared memory the kernel may use
constexpr int kMaxGrid = 512;       // CTAs per launch at most

// Unit ranges of a launch: CTA c processes units [u[c], u[c+1]) of the
// tile-major list (token tile t, row group gi) -> t * ngroups + gi.
// Computed on the host so that the kernel starts without a search.
struct Schedule {
    long long u[kMaxGrid + 1];
};

size_t tiled_bytes(int K, long long M);    // bytes of the token-tile copy of x
size_t smem_bytes(int K);                  // dynamic shared memory per CTA
// Whether the layer kernel can stage x [M][K] itself by tensor copies (K a
// multiple of 16, x 16-byte aligned, the driver's tensor-map encoder found).
bool tensor_staging(int K, const void* x);
int max_k();                               // largest K a tile supports
cudaError_t prepare_kernels(int K, int* ctas_per_sm);  // set attributes, occupancy
cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, const Schedule& sched, int grid, cudaStream_t s);
// Row-wise LayerNorm of z [M][N] (kind 1: fp32 out, 3: int8 out).
cudaError_t launch_layernorm(const float* z, int M, int N, const float* gamma, const float* beta, float eps, int kind,
                             float inv_out_scale, void* out, cudaStream_t s);
// Multi-head self-attention (head width 64, 1 <= seq <= BSGEMM_ATTN_MAX_SEQ)
// on the int8 QKV rows qkv [batch * seq][ld] into out [batch * seq][heads *
// 64] (kind 1: fp32, 3: int8); score_scale = qkv_scale^2 / 8.
size_t attention_smem_bytes(int seq);
cudaError_t launch_attention(const int8_t* qkv, int batch, int seq, int heads, int ld, float score_scale,
                             float qkv_scale, int kind, float inv_out_scale, void* out, bool act_ready, cudaStream_t s);
// The current device's attention status word (bit 0: a wait gave up),
// reset to 0 when clear is set and it was not.
cudaError_t attention_status(bool clear, unsigned* v);
// Weights on the tensor cores (bsgemm_sparse24.cu), for N and K multiples
// of 128, K <= 4096, M >= 1.  2:4-sparse (dense = false): aimg = per
// (128-channel tile, 128-column stage) the kTc24AImage-byte shared-memory
// image of the stored values (128 rows x 64 f16, 128-byte swizzle); meta =
// per (tile, stage, lane) the 4 sparse-MMA metadata words.  Dense over K
// (dense = true, meta unused): aimg = per (tile, stage) the kTcDenseAImage-
// byte image of all 128 columns (two 128-row x 64-f16 sub-tiles, 128-byte
// swizzle).  kind 0-4 (no residual).
constexpr uint32_t kTc24AImage = 16384;
constexpr uint32_t kTcDenseAImage = 32768;
cudaError_t launch_tc_linear(const int8_t* x, int M, int N, int K, const unsigned char* aimg, const uint32_t* meta,
                             bool dense, const float* scale, const float* bias, void* out, int kind,
                             float inv_out_scale, bool act_ready, int* status, cudaStream_t s);
// x [M][K] -> swizzled token tiles in xb (the layout the kernel stages by TMA).
cudaError_t launch_pretile(const int8_t* x, int M, int K, int8_t* xb, int sms, cudaStream_t s);
// Average-magnitude block pruning of a dense fp32 W [N][K] (DEVICE) into
// keep [N/4][K] (DEVICE): the `npruned` lowest-scoring blocks get 0.  Uses
// stream-ordered scratch and synchronises `s`; *bad = a weight was not finite.
cudaError_t block_prune(const float* W, int N, int K, long long npruned, uint8_t* keep, int sms, cudaStream_t s,
                        bool* bad);
// Test hooks for the bounded waits (BSGEMM_TEST_* bits of
// bsgemm_set_test_hooks), read at each launch.
unsigned test_hooks();
// Address of the fixed token-tile scratch (BSGEMM_STATIC_SCRATCH_BYTES) on
// `device`, which must be the current device; looked up on the first call
// per device, then cached.
cudaError_t static_scratch(int device, int8_t** ptr);

}  // namespace bsg
