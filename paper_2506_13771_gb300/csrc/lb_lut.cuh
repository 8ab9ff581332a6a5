// lb_lut.cuh -- shared-memory nibble lookup tables, bulk copies and the
// self-counting exchange words used by the decode kernels (internal).
//
// A +-1 sum over 32 values is 8 lookups in 4-bit tables: table n of a
// vector v holds, for e = 0..15, sum_{k<4} (bit k of e ? -v : +v)[4n + k],
// stored twice (entries e and 16 + e) so the two half-warps read disjoint
// banks.  An exchange word is a 64-bit fixed-point sum whose low 8 bits count
// its contributions.
#pragma once

#include "lb_common.cuh"

namespace lb {
namespace {

extern __shared__ __align__(1024) unsigned char g_smem[];

constexpr float kFix = 16777216.f;            // 2^24
constexpr float kFixInv = 1.f / 16777216.f;

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t saddr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(unsigned long long *bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(saddr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(unsigned long long *bar, unsigned bytes) {
    asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(saddr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(unsigned long long *bar) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(saddr(bar))
        : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(unsigned long long *bar, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(saddr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// 1D TMA bulk copy global -> this CTA's shared memory, completing on bar.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, unsigned bytes,
                                         unsigned long long *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(saddr(dst)),
        "l"(src), "r"(bytes), "r"(saddr(bar))
        : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void red_add_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void ld_relaxed_v2_u64(const unsigned long long *p,
                                                  unsigned long long &a, unsigned long long &b) {
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];"
                 : "=l"(a), "=l"(b)
                 : "l"(p)
                 : "memory");
}

// Sum of 8 nibble-table lookups for the 32 sign bits of one word: lo holds
// nibbles 0,2,4,6 and hi nibbles 1,3,5,7 as (4 * nibble + 64 * copy) bytes;
// PRMT splices that byte into the 256-aligned base of the word's 8 tables.
__device__ __forceinline__ float lut8(uint32_t lo, uint32_t hi, uint32_t base) {
    const unsigned char *s = g_smem;
    const float a0 = *reinterpret_cast<const float *>(s + __byte_perm(lo, base, 0x7650));
    const float a1 = *reinterpret_cast<const float *>(s + __byte_perm(hi, base, 0x7650) + 128);
    const float a2 = *reinterpret_cast<const float *>(s + __byte_perm(lo, base, 0x7651) + 256);
    const float a3 = *reinterpret_cast<const float *>(s + __byte_perm(hi, base, 0x7651) + 384);
    const float a4 = *reinterpret_cast<const float *>(s + __byte_perm(lo, base, 0x7652) + 512);
    const float a5 = *reinterpret_cast<const float *>(s + __byte_perm(hi, base, 0x7652) + 640);
    const float a6 = *reinterpret_cast<const float *>(s + __byte_perm(lo, base, 0x7653) + 768);
    const float a7 = *reinterpret_cast<const float *>(s + __byte_perm(hi, base, 0x7653) + 896);
    return ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
}

__device__ __forceinline__ float lut_word(uint32_t word, uint32_t copy, uint32_t base) {
    const uint32_t lo = ((word << 2) & 0x3C3C3C3Cu) | copy;
    const uint32_t hi = ((word >> 2) & 0x3C3C3C3Cu) | copy;
    return lut8(lo, hi, base);
}

// One contribution to an exchange word: (round(v * 2^24) << 8) + 1.
__device__ __forceinline__ unsigned long long enc_fix(float v, float limit, unsigned *err) {
    if (!(fabsf(v) < limit)) {
        atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_RANGE));
        v = 0.f;
    }
    const long long f = __float2ll_rn(v * kFix);
    return (static_cast<unsigned long long>(f) << 8) + 1ull;
}

__device__ __forceinline__ float dec_fix(unsigned long long w) {
    return __ll2float_rn((long long)w >> 8) * kFixInv;
}
__device__ __forceinline__ bool counted(unsigned long long w, unsigned n_ctas) {
    return (unsigned)(w & 0xffull) == n_ctas;
}

// Stores table n of a unit at T from its four values (see run_tables).
__device__ __forceinline__ void store_table(unsigned char *T, float4 x, int lane) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int q = (k + lane) & 7;
        // chunk q: entries 4(q&3) .. +3; high bits (e3 e2) = q & 3
        const float qv = ((q & 1) ? -x.z : x.z) + ((q & 2) ? -x.w : x.w);
        *reinterpret_cast<float4 *>(T + 16 * q) =
            make_float4(x.x + x.y + qv, x.y - x.x + qv, x.x - x.y + qv, -x.x - x.y + qv);
    }
}

}  // namespace
}  // namespace lb
