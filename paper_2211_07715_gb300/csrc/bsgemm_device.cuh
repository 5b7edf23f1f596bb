// Device helpers of the layer kernel (bsgemm_kernel.cu): the fused epilogue
// of Sec. 3's InnerProduct (dequantise + bias, erf-GELU, requantise; App.
// A.3.3), and thin wrappers of the shared-memory, mbarrier, tensor-copy and
// L2-policy instructions.
// Included by the .cu files only; everything here has internal linkage.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "bsgemm_internal.h"

namespace bsg {
namespace {

// 1/b for 1 <= b < 2^25 by Newton's method, as a fixed sequence of IEEE
// round-to-nearest fp32 operations (no branch, no special function unit):
// b = m 2^E (1 <= m < 2, from the bits), y0 = 24/17 - (8/17) m (the minimax
// straight line for 1/m, relative error <= 1/17; both constants rounded to
// fp32), three steps y <- y + y (1 - m y) (each squares the relative error,
// 1/17 -> 3.5e-3 -> 1.2e-5 -> 1.5e-10), then the exact scaling by 2^-E.
// Within about half an ulp of 1/b, the same bits on every IEEE machine.
__device__ __forceinline__ float recip_nr_f32(float b) {
    const uint32_t bits = __float_as_uint(b);
    const uint32_t ex = (bits >> 23) & 0xffu;  // E + 127
    const float m = __uint_as_float((bits & 0x7fffffu) | (127u << 23));
    float y = __fmaf_rn(-0x1.e1e1e2p-2f, m, 0x1.69696ap+0f);
#pragma unroll
    for (int i = 0; i < 3; ++i) y = __fmaf_rn(y, __fmaf_rn(-m, y, 1.0f), y);
    return __fmul_rn(y, __uint_as_float((254u - ex) << 23));  // 2^-E: biased exponent 127 - E
}

// erf-form GELU in fp32 by a fixed sequence of IEEE round-to-nearest ops.
// erf(|x|) = 1 - p(|x|)^-16, p = 1 + a1 x + ... + a6 x^6 (Abramowitz &
// Stegun 7.1.28, |error| <= 3e-7); p^16 by four squarings; 1/p^16 by
// recip_nr_f32 below 2^25, and erf = 1 from there on (where 1 - 1/p^16
// rounds to 1 in fp32 whatever the quotient's last bits).  Branch-free, so
// the 32 values of a lane's epilogue interleave.
__device__ __forceinline__ float gelu_f32(float y) {
    const float x = __fmul_rn(y, 0.70710678f);
    const float ax = fabsf(x);
    float h = __fmaf_rn(ax, 0.0000430638f, 0.0002765672f);
    h = __fmaf_rn(ax, h, 0.0001520143f);
    h = __fmaf_rn(ax, h, 0.0092705272f);
    h = __fmaf_rn(ax, h, 0.0422820123f);
    h = __fmaf_rn(ax, h, 0.0705230784f);
    const float p = __fmaf_rn(ax, h, 1.0f);
    const float p2 = __fmul_rn(p, p);
    const float p4 = __fmul_rn(p2, p2);
    const float p8 = __fmul_rn(p4, p4);
    const float p16 = __fmul_rn(p8, p8);
    const float r = recip_nr_f32(fminf(p16, 0x1.fffffep24f));  // p16 below 2^25 unchanged; unused from there on
    const float e = (p16 >= 0x1p25f) ? 1.0f : __fsub_rn(1.0f, r);
    const float erf_x = (x < 0.0f) ? -e : e;
    return __fmul_rn(__fmul_rn(0.5f, y), __fadd_rn(1.0f, erf_x));
}

// The same erf-form GELU for fp32 outputs, with the hardware's approximate
// reciprocal (relative error <= 2^-22) in place of the IEEE one: fp32
// outputs are checked against a tolerance, not bit for bit, and the extra
// error stays below 2e-7 |y|.  int8 outputs use gelu_f32, which an int8
// decision must reproduce exactly.
__device__ __forceinline__ float gelu_f32_fast(float y) {
    const float x = y * 0.70710678f;
    const float ax = fabsf(x);
    float h = fmaf(ax, 0.0000430638f, 0.0002765672f);
    h = fmaf(ax, h, 0.0001520143f);
    h = fmaf(ax, h, 0.0092705272f);
    h = fmaf(ax, h, 0.0422820123f);
    h = fmaf(ax, h, 0.0705230784f);
    const float p = fmaf(ax, h, 1.0f);
    const float p2 = p * p, p4 = p2 * p2, p8 = p4 * p4, p16 = p8 * p8;
    float rcp;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(rcp) : "f"(p16));
    const float e = 1.0f - rcp;
    return 0.5f * y * (1.0f + ((x < 0.0f) ? -e : e));
}

// fp32 -> int8 for 4 values: one fp32 multiply each, round half to even
// (to int32, saturating), then saturate to [-128, 127] and pack v0 into
// byte 0 .. v3 into byte 3 (cvt.pack.sat: b into the low byte, a into the
// next, c's low half above).
__device__ __forceinline__ uint32_t requant4_s8(float v0, float v1, float v2, float v3, float inv) {
    const int q0 = __float2int_rn(__fmul_rn(v0, inv)), q1 = __float2int_rn(__fmul_rn(v1, inv));
    const int q2 = __float2int_rn(__fmul_rn(v2, inv)), q3 = __float2int_rn(__fmul_rn(v3, inv));
    uint32_t hi, d;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(hi) : "r"(q3), "r"(q2), "r"(0));
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(q1), "r"(q0), "r"(hi));
    return d;
}

// Epilogue for one token m (nothing past M): v = acc of the 4 channels of
// block-row r (scales s, bias b), written as out[m][4r .. 4r+3].
// The epilogue value of channel c (c < 4) of one token: acc, or y =
// fmaf((float)acc, s, b) with optional GELU.
template <int KIND>
__device__ __forceinline__ float epilogue_value(int v, float s, float b) {
    float y = __fmaf_rn(__int2float_rn(v), s, b);
    if (KIND == 2) y = gelu_f32_fast(y);
    if (KIND == 4) y = gelu_f32(y);
    return y;
}

template <int KIND>
__device__ __forceinline__ void store_token(const LaunchArgs& a, int N, long long m, int r, const int* v, float4 s,
                                            float4 b) {
    if (m >= a.M) return;
    const size_t o = static_cast<size_t>(m) * N + 4 * r;
    if (KIND == 0) {
        *reinterpret_cast<int4*>(static_cast<int32_t*>(a.out) + o) = make_int4(v[0], v[1], v[2], v[3]);
        return;
    }
    float y0 = __fmaf_rn(__int2float_rn(v[0]), s.x, b.x);
    float y1 = __fmaf_rn(__int2float_rn(v[1]), s.y, b.y);
    float y2 = __fmaf_rn(__int2float_rn(v[2]), s.z, b.z);
    float y3 = __fmaf_rn(__int2float_rn(v[3]), s.w, b.w);
    if (KIND == 2) {
        y0 = gelu_f32_fast(y0);
        y1 = gelu_f32_fast(y1);
        y2 = gelu_f32_fast(y2);
        y3 = gelu_f32_fast(y3);
    } else if (KIND == 4) {
        y0 = gelu_f32(y0);
        y1 = gelu_f32(y1);
        y2 = gelu_f32(y2);
        y3 = gelu_f32(y3);
    }
    if (KIND == 5) {  // residual add: z = y + res_scale * (float)r, two fp32 operations
        const uint32_t r4 = __ldg(reinterpret_cast<const uint32_t*>(a.res + o));
        y0 = __fadd_rn(y0, __fmul_rn(a.res_scale, __int2float_rn(static_cast<int8_t>(r4))));
        y1 = __fadd_rn(y1, __fmul_rn(a.res_scale, __int2float_rn(static_cast<int8_t>(r4 >> 8))));
        y2 = __fadd_rn(y2, __fmul_rn(a.res_scale, __int2float_rn(static_cast<int8_t>(r4 >> 16))));
        y3 = __fadd_rn(y3, __fmul_rn(a.res_scale, __int2float_rn(static_cast<int8_t>(r4 >> 24))));
    }
    if (KIND == 1 || KIND == 2 || KIND == 5) {
        *reinterpret_cast<float4*>(static_cast<float*>(a.out) + o) = make_float4(y0, y1, y2, y3);
    } else {
        *reinterpret_cast<uint32_t*>(static_cast<int8_t*>(a.out) + o) = requant4_s8(y0, y1, y2, y3, a.inv_out_scale);
    }
}

// N % 4 != 0: rows of out are not 16-byte aligned and the last block-row
// has fewer than 4 channels -- one store a channel, channels < N only
// (constant indices throughout, so acc stays in registers).  The lane holds
// NT tokens m_g + 8 i, i < NT, x 4 channels in acc[4 i + c].
template <int KIND, int NT>
__device__ __forceinline__ void store_lane_narrow(const LaunchArgs& a, int N, long long m_g, int r,
                                                  const int (&acc)[4 * NT], float4 sc, float4 bi) {
    const int nc = min(4, N - 4 * r);
    const float s4[4] = {sc.x, sc.y, sc.z, sc.w}, b4[4] = {bi.x, bi.y, bi.z, bi.w};
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const long long m = m_g + 8 * i;
        if (m >= a.M) continue;
        const size_t o = static_cast<size_t>(m) * N + 4 * r;
        if (KIND == 0) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c < nc) static_cast<int32_t*>(a.out)[o + c] = acc[4 * i + c];
        } else if (KIND == 1 || KIND == 2) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c < nc) static_cast<float*>(a.out)[o + c] = epilogue_value<KIND>(acc[4 * i + c], s4[c], b4[c]);
        } else if (KIND == 5) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c < nc)
                    static_cast<float*>(a.out)[o + c] =
                        __fadd_rn(epilogue_value<1>(acc[4 * i + c], s4[c], b4[c]),
                                  __fmul_rn(a.res_scale, __int2float_rn(a.res[o + c])));
        } else {
            float y[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) y[c] = epilogue_value<KIND>(acc[4 * i + c], s4[c], b4[c]);
            const uint32_t q = requant4_s8(y[0], y[1], y[2], y[3], a.inv_out_scale);
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c < nc) static_cast<int8_t*>(a.out)[o + c] = static_cast<int8_t>(q >> (8 * c));
        }
    }
}

__device__ __forceinline__ float4 load_s4(const float* p, int r) { return __ldg(reinterpret_cast<const float4*>(p) + r); }

// Last index r in [lo, hi) with sp[r] <= q, given sp[lo] <= q < sp[hi]
// (sp: the shared-memory window of row-group step offsets).
__device__ __forceinline__ int row_of(const int* sp, int lo, int hi, int q) {
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (sp[mid] <= q) lo = mid; else hi = mid;
    }
    return lo;
}

// 32-bit shared-window address of a shared-memory pointer.
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Gather two 16 x 16 byte matrices from shared memory, transposed: lane i
// gives the address of row (i % 16) of matrix i / 16 (16 bytes, 16-byte
// aligned); lane l receives, for matrix 0 (r0, r1) and matrix 1 (r2, r3),
// the bytes of rows 4 (l % 4) .. 4 (l % 4) + 3 at column l / 4 (r0, r2) and
// column l / 4 + 8 (r1, r3), row 4 (l % 4) in the lowest byte.
__device__ __forceinline__ void ldsm_x2_trans_b8(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                                 uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m16n16.x2.trans.shared.b8 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}

// mbarrier + bulk-copy (TMA) helpers.  Waits are bounded: a wait that
// gives up reports false and the caller records kStatusTimeout.
constexpr unsigned kWaitLimit = 1u << 20;

__device__ __forceinline__ void mbar_init(uint32_t bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
// n consecutive barriers (8 bytes apart) with one arrival each, then one
// fence that makes all the initialisations visible to the async proxy.
__device__ __forceinline__ void mbar_init_n(uint32_t bar, int n) {
    for (int i = 0; i < n; ++i)
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(bar + 8u * static_cast<uint32_t>(i)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, unsigned bytes) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n"
                 ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, unsigned parity, unsigned limit) {
    for (unsigned i = 0; i < limit; ++i) {
        unsigned done;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                     " selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(done) : "r"(bar), "r"(parity) : "memory");
        if (done) return true;
    }
    return false;
}
// Global -> shared bulk copy completing on an mbarrier (16-byte aligned, size % 16 == 0).
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, unsigned bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// One 2-D box of a tensor map (x = innermost coordinate, y = row) into
// shared memory, completing on an mbarrier.
__device__ __forceinline__ void tensor_g2s(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n"
                 ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar) : "memory");
}
__device__ __forceinline__ void st_shared_u32(uint32_t addr, uint32_t v) {
    asm volatile("st.shared.u32 [%0], %1;\n" ::"r"(addr), "r"(v) : "memory");
}
// Programmatic dependent launch: both kernels are launched so that they may
// start while the previous kernel of the stream finishes.  Before a kernel
// reads its activations or writes any global memory, every thread waits
// until the previous grid has completed and its writes are visible (a no-op
// when there is none); early on it lets the next kernel launch.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

// L2 eviction priorities (createpolicy): the weights' step records, group
// offsets, scales and biases are read by every CTA of every launch and are
// kept (evict_last); the activation tiles stream through once per launch
// (evict_first), so that they do not push the weights out of L2.
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;\n" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(p));
    return p;
}
// Read-only global loads with an L2 eviction policy.
__device__ __forceinline__ int ldg_hint(const int* p, uint64_t pol) {
    int v;
    asm volatile("ld.global.nc.L2::cache_hint.b32 %0, [%1], %2;\n" : "=r"(v) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ unsigned short ldg_hint(const unsigned short* p, uint64_t pol) {
    unsigned short v;
    asm volatile("ld.global.nc.L2::cache_hint.u16 %0, [%1], %2;\n" : "=h"(v) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ int4 ldg_hint(const int4* p, uint64_t pol) {
    int4 v;
    asm volatile("ld.global.nc.L2::cache_hint.v4.b32 {%0, %1, %2, %3}, [%4], %5;\n"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ float4 ldg_hint(const float4* p, uint64_t pol) {
    float4 v;
    asm volatile("ld.global.nc.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;\n"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p), "l"(pol));
    return v;
}
// tensor_g2s with an L2 eviction policy for the copied bytes.
__device__ __forceinline__ void tensor_g2s_hint(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar,
                                                uint64_t pol) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
                 " [%0], [%1, {%2, %3}], [%4], %5;\n"
                 ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(pol) : "memory");
}

// One 3-D box (x innermost, then y, then z) with an L2 eviction policy.
__device__ __forceinline__ void tensor_g2s_3d_hint(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                                   uint32_t bar, uint64_t pol) {
    asm volatile("cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
                 " [%0], [%1, {%2, %3, %4}], [%5], %6;\n"
                 ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar), "l"(pol)
                 : "memory");
}

// Order this thread's earlier generic-proxy shared-memory accesses before
// later asynchronous-proxy (bulk copy) writes.
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }

}  // namespace
}  // namespace bsg
