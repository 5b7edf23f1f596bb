// Internal declarations shared by the host API (bsgemm_api.cpp) and the
// kernels (bsgemm_kernel.cu).  Not part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace bsg {

// Device form of one block-compressed weight (built once by bsgemm_create).
//
// A block-row r holds output rows 4r..4r+3.  Its stored blocks are grouped
// in "quads" of 4 (the analogue of Algorithm 1's k_block = 4): quad q is a
// 32-byte record
//   int4 k : the 4 input columns k0..k3 (the last quad of a block-row is
//            padded by repeating its last real column, with zero weights)
//   int4 w : w.{x,y,z,w}[c] = bytes W[4r+c][k0], W[4r+c][k1], W[4r+c][k2],
//            W[4r+c][k3] -- one dot-4 operand per output channel c.
// Quads of block-row r are [qptr[r], qptr[r+1]).
struct DeviceWeights {
    const int32_t* qptr;   // [nbr + 1]
    const int32_t* cost;   // [nbr + 1]: qptr[r] + r, the schedule's prefix cost
    const int4* quads;     // [2 * Q]: k record then w record per quad
    const float* scale;    // [N]
    const float* bias;     // [N]
    int* status;           // device status word (bounded-wait timeouts), 0 = fine
    int N, K, nbr, Q;
};

// Device status bits written by the kernels.
constexpr int kStatusTimeout = 1;  // a bounded wait on an asynchronous copy gave up

struct LaunchArgs {
    const int8_t* x;       // [M][K]
    const int8_t* xb;      // NULL, or x re-laid as token tiles: [ntiles][kpad][MT] (k-major per tile)
    void* out;             // [M][N]
    int M;
    int kind;
    float inv_out_scale;
    bool x_vec16;          // x 16-byte aligned and K % 16 == 0
};

// Kernel configuration: 16 warps per CTA; a token tile holds MT = 64 or 128
// tokens and each lane owns 4 consecutive tokens of it.
constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kQuadPad = 16;        // zero records after the last quad (one ring chunk)
constexpr int kRowWin = 512;        // block-rows whose quad offsets a CTA keeps in shared memory
constexpr int kStaticSmem = 2304;   // bytes of static shared memory the kernel may use
constexpr int kMaxGrid = 512;       // CTAs per launch at most

// Unit ranges of a launch: CTA c processes units [u[c], u[c+1]) of the
// tile-major list (token tile t, block-row r) -> t * nbr + r.  Computed on
// the host so that the kernel starts without a search.
struct Schedule {
    long long u[kMaxGrid + 1];
};

int tile_for_k(int K);                     // MT for a given K (0 if none fits)
// Lane groups per warp for a tile height (a lane owns 8 tokens, so MT/8
// lanes span the tile): each block-row's quad list is padded to a multiple
// of this, so a warp's step (one quad per group) never leaves a block-row.
constexpr int groups_for_tile(int MT) { return 256 / MT; }
size_t tiled_bytes(int MT, int K, long long M);  // bytes of the token-tile copy of x
size_t smem_bytes(int MT, int K);          // dynamic shared memory per CTA
int max_k();                               // largest K any tile supports
cudaError_t prepare_kernels(int MT, int K, int* ctas_per_sm);  // set attributes, occupancy
cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, const Schedule& sched, int MT, int grid,
                   cudaStream_t s);
// x [M][K] -> token tiles [ntiles][kpad][MT] in xb (the layout the kernel stages by TMA).
cudaError_t launch_pretile(const int8_t* x, int M, int K, int MT, int8_t* xb, int sms, cudaStream_t s);
// Address of the fixed token-tile scratch (BSGEMM_STATIC_SCRATCH_BYTES) on
// `device`, which must be the current device; looked up on the first call
// per device, then cached.
cudaError_t static_scratch(int device, int8_t** ptr);

}  // namespace bsg
