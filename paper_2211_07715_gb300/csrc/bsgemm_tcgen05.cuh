// Fifth-generation tensor-core (tcgen05) helpers for sm_103a: tensor-memory
// allocation, MMA issue from shared-memory matrix descriptors or a tensor-
// memory A operand, completion through an mbarrier, and tensor-memory loads
// and stores.  Included by the .cu files only; internal linkage.
//
// Tensor memory (TMEM) is 512 columns x 128 lanes of 32 bits per SM.  An
// address is (lane << 16) | column.  A warp reaches only the 32 lanes of its
// quarter (warp % 4); in the 32x32b shape thread t of the warp reads or
// writes lane 32 (warp % 4) + t, consecutive columns into consecutive
// registers.  An MMA with M = 128 writes row i of D to lane i, column j to
// column j (fp32); a 16-bit A operand in TMEM holds row i in lane i, two
// consecutive K elements per column (the lower K index in the low half).
#pragma once

#include <cstdint>

namespace bsg {
namespace {

// Shared-memory matrix descriptor of an operand stored with the 128-byte
// swizzle: rows of 128 bytes, 8-row atoms of 1024 bytes in which 16-byte
// chunk c of row r sits at chunk c ^ (r % 8), atoms 1024-byte aligned.
// Fields: start address >> 4 (bits 0-13), leading byte offset >> 4 (16-29),
// stride byte offset >> 4 (32-45), descriptor version 1 (bit 46), swizzle
// mode 2 = 128-byte (bits 61-63); base offset 0 (the atoms are aligned).
// K-major operand (a row = 64 f16 of K): the stride byte offset is the
// distance between 8-row groups (1024), the leading one is unused; an MMA's
// K step of 16 elements advances the start by 32 bytes.  MN-major operand
// (a row = 64 f16 of M or N for one K index): with M or N = 64 only the
// distance between groups of 8 K rows is used (1024); it goes in both
// fields.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return static_cast<uint64_t>((saddr >> 4) & 0x3FFFu) | (static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16) |
           (static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of tcgen05.mma kind::f16 with f16 A and B and an
// fp32 accumulator: D format (bits 4-5) 1 = f32; A and B formats (7-9,
// 10-12) 0 = f16; A K-major (bit 15 = 0); B major (bit 16) 0 = K, 1 = MN;
// N / 8 (bits 17-22); M / 16 (bits 24-28).
__host__ __device__ constexpr uint32_t f16_idesc(int m, int n, bool b_mn_major) {
    return (1u << 4) | (b_mn_major ? (1u << 16) : 0u) | (static_cast<uint32_t>(n >> 3) << 17) |
           (static_cast<uint32_t>(m >> 4) << 24);
}

// Warp-wide: allocate `ncols` columns (a power of two >= 32), the address
// written to shared memory at `slot`; then give up the right to allocate
// again, so that another CTA on the SM waiting to allocate is not delayed.
__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(slot), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols) : "memory");
}

// Order tcgen05 operations across a thread barrier: `before` ahead of the
// barrier by the threads whose loads, stores or MMAs came first, `after`
// behind it by the threads that continue.
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// D (TMEM) = A B (+ D when acc != 0); A and B from shared memory.
__device__ __forceinline__ void mma_f16_ss(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
    asm volatile("{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
                 " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
                 ::"r"(d), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc) : "memory");
}
// D (TMEM) = A B (+ D when acc != 0); A from TMEM, B from shared memory.
__device__ __forceinline__ void mma_f16_ts(uint32_t d, uint32_t a, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
    asm volatile("{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
                 " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n"
                 ::"r"(d), "r"(a), "l"(bdesc), "r"(idesc), "r"(acc) : "memory");
}
// One arrival on the mbarrier once every tcgen05 operation this thread
// issued before has completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
                 : "memory");
}

#define BSG_TC_OUT8(v, i) "=r"(v[i]), "=r"(v[i + 1]), "=r"(v[i + 2]), "=r"(v[i + 3]), "=r"(v[i + 4]), \
    "=r"(v[i + 5]), "=r"(v[i + 6]), "=r"(v[i + 7])
#define BSG_TC_IO8(v, i) "+r"(v[i]), "+r"(v[i + 1]), "+r"(v[i + 2]), "+r"(v[i + 3]), "+r"(v[i + 4]), \
    "+r"(v[i + 5]), "+r"(v[i + 6]), "+r"(v[i + 7])
#define BSG_TC_IN8(v, i) "r"(v[i]), "r"(v[i + 1]), "r"(v[i + 2]), "r"(v[i + 3]), "r"(v[i + 4]), \
    "r"(v[i + 5]), "r"(v[i + 6]), "r"(v[i + 7])

// Warp-wide: 32 consecutive columns of this thread's lane into v (valid only
// after tmem_wait_ld).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
                 "%13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
                 "[%32];\n"
                 : BSG_TC_OUT8(v, 0), BSG_TC_OUT8(v, 8), BSG_TC_OUT8(v, 16), BSG_TC_OUT8(v, 24)
                 : "r"(taddr));
}
// Wait for this thread's outstanding tensor-memory loads; v is tied to the
// wait so that nothing reads it earlier.
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&v)[32]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;\n"
                 : BSG_TC_IO8(v, 0), BSG_TC_IO8(v, 8), BSG_TC_IO8(v, 16), BSG_TC_IO8(v, 24)
                 :
                 : "memory");
}
// Warp-wide: v into 32 consecutive columns of this thread's lane.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
                 "%13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, "
                 "%32};\n"
                 ::"r"(taddr), BSG_TC_IN8(v, 0), BSG_TC_IN8(v, 8), BSG_TC_IN8(v, 16), BSG_TC_IN8(v, 24)
                 : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory"); }
#undef BSG_TC_OUT8
#undef BSG_TC_IO8
#undef BSG_TC_IN8

}  // namespace
}  // namespace bsg
