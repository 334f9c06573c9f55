// Shared device helpers of the CLEAR-MoE library (sm_103a): status word, bounded waits,
// bf16 packing, mbarrier / TMA / tcgen05 wrappers written as inline PTX.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/clearmoe.h"

#define CM_MAX_E 16
#define CM_MAX_R 256

namespace cm {

// ------------------------------------------------------------------ status word
__device__ __forceinline__ void set_status(int32_t* status, int32_t code) {
    if (status) atomicCAS(status, 0, code);  // the first device error wins
}

__device__ __forceinline__ uint64_t globaltimer() {
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// ------------------------------------------------------------------ bf16 helpers
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);  // round to nearest even
    return *reinterpret_cast<uint32_t*>(&p);
}
__device__ __forceinline__ float bf16_to_f32(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }
__device__ __forceinline__ uint16_t f32_to_bf16(float v) {
    const __nv_bfloat16 b = __float2bfloat16_rn(v);  // round to nearest even
    return *reinterpret_cast<const uint16_t*>(&b);
}

__device__ __forceinline__ float gelu_erf(float u) {
    // GELU(u) = u * Phi(u) = u * (1 + erf(u / sqrt 2)) / 2, with CUDA's erff.
    return 0.5f * u * (1.0f + erff(u * 0.70710678118654752440f));
}

// GELU of a pair for the bf16 layer, whose hidden state is stored in bf16. erf is evaluated by
// the rational approximation of Abramowitz & Stegun, Handbook of Mathematical Functions, 7.1.28
// (C. Hastings): erf(x) = 1 - (1 + a1 x + ... + a6 x^6)^-16 for x >= 0, |error| <= 3e-7, with
// x = |u| / sqrt(2) folded into the coefficients. With y = P^-16, GELU(u) = u - |u| y / 2 for
// u >= 0 and -|u| y / 2 for u < 0, i.e. max(u, 0) + m y with m = -|u| / 2 for every u. Horner's
// rule runs on m with the coefficients scaled by 2^k and alternating in sign, which yields -P bit
// for bit (power-of-two scaling is exact, and an fma rounds symmetrically in sign), so the last
// step is one fma; max(u, 0) is formed as u / 2 - m, one exact packed fma. Packed fp32x2
// arithmetic; the absolute error of the result is below 7.5e-7
// for every u (checked against float64 on a 2M-point grid), far below the bf16 spacing of z.
// The fp32 layer keeps gelu_erf (CUDA's erff).
struct GeluAS {
    static constexpr double S = 0.70710678118654752440;  // 1 / sqrt(2)
    // b_k 2^k with b_k = a_k / sqrt(2)^k, signs alternating for Horner's rule on m = -|u| / 2
    static constexpr float C6 = (float)(-0.0000430638 * S * S * S * S * S * S * 64.0);
    static constexpr float C5 = (float)(0.0002765672 * S * S * S * S * S * 32.0);
    static constexpr float C4 = (float)(-0.0001520143 * S * S * S * S * 16.0);
    static constexpr float C3 = (float)(0.0092705272 * S * S * S * 8.0);
    static constexpr float C2 = (float)(-0.0422820123 * S * S * 4.0);
    static constexpr float C1 = (float)(0.0705230784 * S * 2.0);
    static constexpr float C0 = -1.0f;
};

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float2 gelu_pair_as(float2 u) {
    const float2 m = make_float2(-0.5f * fabsf(u.x), -0.5f * fabsf(u.y));
    float2 p = __ffma2_rn(make_float2(GeluAS::C6, GeluAS::C6), m, make_float2(GeluAS::C5, GeluAS::C5));
    p = __ffma2_rn(p, m, make_float2(GeluAS::C4, GeluAS::C4));
    p = __ffma2_rn(p, m, make_float2(GeluAS::C3, GeluAS::C3));
    p = __ffma2_rn(p, m, make_float2(GeluAS::C2, GeluAS::C2));
    p = __ffma2_rn(p, m, make_float2(GeluAS::C1, GeluAS::C1));
    p = __ffma2_rn(p, m, make_float2(GeluAS::C0, GeluAS::C0));  // = -P
    p = __fmul2_rn(p, p);
    p = __fmul2_rn(p, p);
    p = __fmul2_rn(p, p);
    p = __fmul2_rn(p, p);  // P^16 (overflows to +inf for |u| > ~10, where y = 0 is exact in fp32)
    const float2 y = make_float2(rcp_approx(p.x), rcp_approx(p.y));
    // max(u, 0) = u / 2 - m exactly (both terms are exact halves, their sum is u or 0)
    const float2 r = __ffma2_rn(make_float2(0.5f, 0.5f), u, make_float2(-m.x, -m.y));
    return __ffma2_rn(m, y, r);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------------ programmatic dependent launch
// A kernel launched with programmatic stream serialisation may start while its predecessor in the
// stream is still running; it must call pdl_wait() before touching anything that predecessor
// writes (or reads, if it overwrites it). pdl_launch_dependents() lets the successor start early.
// Both are no-ops for kernels launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase of `parity` to complete, giving up after limit_ns or when another role of
// the CTA has already given up (*abort != 0; abort may be null). Returns false on give-up; the first waiter to run
// out raises *abort and writes CLEARMOE_ETIMEOUT to the status word.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort,
                                          int32_t* status, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    while (true) {
        if (abort && *abort) return false;
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer() - t0 > limit_ns) {
            if (abort) *abort = 1;
            set_status(status, CLEARMOE_ETIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ unsigned int ld_acquire_u32(const unsigned int* p) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release_u32(unsigned int* p, unsigned int v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// ------------------------------------------------------------------ TMA
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t c0,
                                            int32_t c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int32_t c0, int32_t c1,
                                            int32_t c2, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------------------------------ tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t slot_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     slot_smem),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulator), one CTA.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive once on an mbarrier when every tcgen05.mma issued so far by this thread completes.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

#define CM_TMEM_LD_X16(taddr, r)                                                                 \
    asm volatile(                                                                                \
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13," \
        "%14,%15}, [%16];"                                                                       \
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),    \
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),             \
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])                                                  \
        : "r"(taddr))

#define CM_TMEM_LD_X8(taddr, r)                                                                  \
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"         \
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),        \
                   "=r"(r[6]), "=r"(r[7])                                                         \
                 : "r"(taddr))

// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with 128-byte swizzle:
// rows of 128 bytes (64 elements of K), 8-row swizzle atoms 1024 bytes apart (SBO), descriptor
// version 1, layout SWIZZLE_128B. The tile base must be 1024-byte aligned; advancing along K
// inside the atom is done by adding the byte offset to the start address.
__device__ __forceinline__ uint64_t sdesc_kmajor_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;            // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1 << 46;            // descriptor version
    d |= (uint64_t)2 << 61;            // SWIZZLE_128B
    return d;
}

// The same K-major 128-byte-swizzled descriptor with 8-row atoms `sbo` bytes apart (a multiple of
// 16 below 256 KB), for tiles whose row groups are interleaved with other K blocks' in shared memory.
__device__ __forceinline__ uint64_t sdesc_kmajor_sw128_sbo(uint32_t saddr, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, M x N tile.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}

}  // namespace cm
