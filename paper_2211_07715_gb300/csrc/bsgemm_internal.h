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
    int N, K, nbr, Q;
};

struct LaunchArgs {
    const int8_t* x;       // [M][K]
    void* out;             // [M][N]
    int M;
    int kind;
    float inv_out_scale;
    bool x_vec16;          // x 16-byte aligned and K % 16 == 0
};

// Kernel tile configurations.  MT = tokens per tile; GL = lanes that share
// one block-row (each lane owns 4 consecutive tokens); 16 warps per CTA.
constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;

int tile_for_k(int K);                     // MT for a given K (0 if none fits)
size_t smem_bytes(int MT, int K);          // dynamic shared memory per CTA
int max_k();                               // largest K any tile supports
cudaError_t prepare_kernels(int MT, int K, int* ctas_per_sm);  // set attributes, occupancy
cudaError_t launch(const DeviceWeights& w, const LaunchArgs& a, int MT, int grid, cudaStream_t s);

}  // namespace bsg
