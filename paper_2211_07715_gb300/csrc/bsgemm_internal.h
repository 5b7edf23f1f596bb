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
// of row k sits in 16-byte slot ((4 (k & 1) + c) XOR (i & 7)) of its line.
// Row k's chunk 0 is therefore at byte tile_row_offset(k), and chunk c at
// tile_row_offset(k) XOR 16 c.  The XOR spreads the chunks of different rows
// over the 8 bank groups of shared memory, so a gather of 8 rows whose
// "bank keys" (slot of chunk 0) differ reads in one pass.
inline uint32_t tile_row_offset(int k) {
    const uint32_t line = static_cast<uint32_t>(k) >> 1;
    const uint32_t slot = ((static_cast<uint32_t>(k) & 1u) << 2) ^ (line & 7u);
    return (line << 7) | (slot << 4);
}
inline int bank_key(int k) { return static_cast<int>((tile_row_offset(k) >> 4) & 7u); }

// Device form of one block-compressed weight (built once by bsgemm_create).
//
// A block-row r holds output rows 4r..4r+3.  Its stored blocks (columns)
// are ordered and grouped in "steps" of 16; steps of block-row r are
// [sptr[r], sptr[r+1]).  A step is a 128-byte record (8 int4):
//   int32 off[16]  : tile_row_offset(k_j) of its columns k_0..k_15
//   uint32 w[4][4] : w[q][c] = bytes W[4r+c][k_{4q}] .. W[4r+c][k_{4q+3}],
//                    one dot-4 operand per output channel c and quad q
// (quad q = columns 4q..4q+3, the analogue of Algorithm 1's k_block = 4).
// The last step of a block-row is padded with zero-weight entries whose
// columns are valid tile rows.  Within each half of a step (columns 0-7,
// 8-15) the columns' bank keys differ wherever the row's columns allow it.
struct DeviceWeights {
    const int32_t* sptr;   // [nbr + 1]
    const int4* recs;      // [8 * (S + kStepPad)]
    const float* scale;    // [N]
    const float* bias;     // [N]
    int* status;           // device status word (bounded-wait timeouts), 0 = fine
    int N, K, nbr, S;
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
};

// Kernel configuration: 16 warps per CTA.
constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kStepPad = 4;         // zero step records after the last one (record prefetch runs ahead)
constexpr int kRowWin = 256;        // block-rows whose step offsets, scales and biases a CTA keeps in shared memory
constexpr int kStaticSmem = 2304;   // bytes of static shared memory the kernel may use
constexpr int kMaxGrid = 512;       // CTAs per launch at most

// Unit ranges of a launch: CTA c processes units [u[c], u[c+1]) of the
// tile-major list (token tile t, block-row r) -> t * nbr + r.  Computed on
// the host so that the kernel starts without a search.
struct Schedule {
    long long u[kMaxGrid + 1];
};

size_t tiled_bytes(int K, long long M);    // bytes of the token-tile copy of x
size_t smem_bytes(int K);                  // dynamic shared memory per CTA
int max_k();                               // largest K a tile supports
cudaError_t prepare_kernels(int K, int* ctas_per_sm);  // set attributes, occupancy
cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, const Schedule& sched, int grid, cudaStream_t s);
// x [M][K] -> swizzled token tiles in xb (the layout the kernel stages by TMA).
cudaError_t launch_pretile(const int8_t* x, int M, int K, int8_t* xb, int sms, cudaStream_t s);
// Address of the fixed token-tile scratch (BSGEMM_STATIC_SCRATCH_BYTES) on
// `device`, which must be the current device; looked up on the first call
// per device, then cached.
cudaError_t static_scratch(int device, int8_t** ptr);

}  // namespace bsg
