// lb_lut.cuh -- shared-memory nibble lookup tables, bulk copies and the
// self-counting exchange words used by the decode kernels (internal).
//
// A +-1 sum over 32 values is 8 lookups in 4-bit tables: table n of a
// vector v holds, for e = 0..15, sum_{k<4} (bit k of e ? -v : +v)[4n + k],
// stored twice (entries e and 16 + e) so the two half-warps read disjoint
// banks.  An exchanged element is a pair of 64-bit fixed-point words whose
// low 8 bits count its contributions (see send_fix2).
#pragma once

#include "lb_common.cuh"

namespace lb {
namespace {

extern __shared__ __align__(1024) unsigned char g_smem[];


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

// ---------------------------------------------------------------- clusters

__device__ __forceinline__ unsigned cluster_rank() {
    unsigned r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// CTAs in this CTA's cluster (1 when the launch formed no clusters).
__device__ __forceinline__ unsigned cluster_size() {
    unsigned n;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(n));
    return n;
}

// The shared::cluster address of byte offset `local` (a shared::cta address)
// in the CTA of rank `rank` of this cluster.
__device__ __forceinline__ uint32_t mapa(uint32_t local, unsigned rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}

// 4 bytes into another CTA's shared memory, completing 4 bytes of the
// transaction count of that CTA's mbarrier (both shared::cluster addresses).
__device__ __forceinline__ void st_async_f32(uint32_t raddr, float v, uint32_t rbar) {
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(raddr),
        "r"(__float_as_uint(v)), "r"(rbar)
        : "memory");
}

// Arrival of this thread on bar with `bytes` more transaction bytes expected.
__device__ __forceinline__ void mbar_arrive_expect_tx(unsigned long long *bar, unsigned bytes) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(
            saddr(bar)),
        "r"(bytes)
        : "memory");
}

// try_wait with cluster-scope acquire: data written into this CTA's shared
// memory by other CTAs of the cluster (st.async) is visible once it succeeds.
__device__ __forceinline__ bool mbar_try_wait_cluster(unsigned long long *bar, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], "
        "%2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(saddr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Cluster-wide barrier of every thread (not .aligned: threads may arrive
// from divergent paths).
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
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

// ---------------------------------------------------------------- exchange
//
// An element of an exchange (one value of the rank-r t all-reduced across
// the CTAs) is a pair of 64-bit words (hi, lo) that holds the EXACT sum of
// its fp32 contributions in fixed point with resolution 2^-64.  Elements are
// laid out in blocks of 32: the hi words of elements 32b .. 32b + 31, then
// their lo words (fix2_at), so a warp's 32 consecutive elements take two
// cache lines of hi words and two of lo words.  A
// contribution v is split as v * 2^64 = H * 2^47 + L with H = trunc(v 2^17)
// and |L| < 2^47, and adds (H << 8) + 1 to hi and (L << 8) + 1 to lo with
// one red.add each: the low 8 bits of both words count the contributions
// (at most 255), the high 56 bits carry the integer sums.  Every fp32 v with
// 2^-41 <= |v| < 2^34 / n (n contributions) is represented exactly, smaller
// ones to within 2^-65, so the sum is exact whatever the order of arrival
// and, decoded with one correct rounding, scales exactly with the inputs:
// Prop. 1 is linear, and so is this exchange over 66 binades.  A
// contribution outside the range records LB_ERR_RANGE and is sent as zero.

// 2^34 / n: the largest |contribution| that keeps the sum of n of them
// below 2^51 in H (the range dec_fix2 rounds correctly).
__host__ __device__ constexpr float fix2_limit(int n) { return 17179869184.f / (float)n; }

// The hi word of element e of an exchange buffer at x (its lo word is 32
// words further).  Buffers hold a whole number of 32-element blocks.
__host__ __device__ __forceinline__ size_t fix2_words(size_t elements) {
    return 2 * ((elements + 31) & ~(size_t)31);
}
__device__ __forceinline__ unsigned long long *fix2_at(unsigned long long *x, int e) {
    return x + 64 * (e >> 5) + (e & 31);
}
__device__ __forceinline__ const unsigned long long *fix2_at(const unsigned long long *x, int e) {
    return x + 64 * (e >> 5) + (e & 31);
}

// One contribution v to the element whose hi word is w.
__device__ __forceinline__ void send_fix2(unsigned long long *w, float v, float limit,
                                          unsigned *err) {
    if (!(fabsf(v) < limit)) {
        atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_RANGE));
        v = 0.f;
    }
    const float a = v * 0x1p17f;  // exact
    const float t = truncf(a);
    const long long H = __float2ll_rz(t);
    const long long L = __float2ll_rn((a - t) * 0x1p47f);  // a - t is exact, |.| < 1
    red_add_u64(w, (static_cast<unsigned long long>(H) << 8) + 1ull);
    red_add_u64(w + 32, (static_cast<unsigned long long>(L) << 8) + 1ull);
}

// A contribution of zero that only counts (a CTA with nothing to add).
__device__ __forceinline__ void send_count2(unsigned long long *w) {
    red_add_u64(w, 1ull);
    red_add_u64(w + 32, 1ull);
}

// The hi and lo words of one element (hi word at w), relaxed.
__device__ __forceinline__ void ld_fix2(const unsigned long long *w, unsigned long long &hi,
                                        unsigned long long &lo) {
    hi = ld_relaxed_u64(w);
    lo = ld_relaxed_u64(w + 32);
}

__device__ __forceinline__ bool counted2(unsigned long long hi, unsigned long long lo,
                                         unsigned n) {
    return (unsigned)(hi & 0xffull) == n && (unsigned)(lo & 0xffull) == n;
}

// Elements e .. e + 3 (e a multiple of 4; hi word of e at p), relaxed:
// a[2k], a[2k + 1] = hi, lo of element e + k.
__device__ __forceinline__ void ld_fix2x4(const unsigned long long *p, unsigned long long (&a)[8]) {
    ld_relaxed_v2_u64(p, a[0], a[2]);
    ld_relaxed_v2_u64(p + 2, a[4], a[6]);
    ld_relaxed_v2_u64(p + 32, a[1], a[3]);
    ld_relaxed_v2_u64(p + 34, a[5], a[7]);
}

__device__ __forceinline__ bool counted2x4(const unsigned long long (&a)[8], unsigned n) {
    return counted2(a[0], a[1], n) && counted2(a[2], a[3], n) && counted2(a[4], a[5], n) &&
           counted2(a[6], a[7], n);
}

// The same with n0 contributions expected for the first element (element 0
// of an exchange, which every CTA counts into) and n for the others.
__device__ __forceinline__ bool counted2x4(const unsigned long long (&a)[8], unsigned n0,
                                           unsigned n) {
    return counted2(a[0], a[1], n0) && counted2(a[2], a[3], n) && counted2(a[4], a[5], n) &&
           counted2(a[6], a[7], n);
}

// The sum held by a complete pair, (H 2^47 + L) 2^-64, rounded to nearest
// fp32 (ties to even): exactly while it fits 64 bits (|H| < 2^15); beyond
// that from floor(sum / 2^36) with a sticky bit for the dropped remainder
// (the quotient then has more than 26 bits, so the sticky bit sits below the
// rounding position and cannot move a tie).  |H| < 2^51 (fix2_limit) keeps
// 2 floor(sum / 2^36) + 1 inside 64 bits.
__device__ __forceinline__ float dec_fix2(unsigned long long hi, unsigned long long lo) {
    const long long H = static_cast<long long>(hi) >> 8;
    const long long L = static_cast<long long>(lo) >> 8;
    if (H > -32768ll && H < 32768ll) return __ll2float_rn(H * 140737488355328ll + L) * 0x1p-64f;
    const long long q = H * 2048ll + (L >> 36);
    const long long sticky = (L & 68719476735ll) != 0 ? 1 : 0;
    return __ll2float_rn(2 * q + sticky) * 0x1p-29f;
}

// ---------------------------------------------------------------- bounded one-word exchange
//
// The stack kernel's exchanges are one 64-bit word per element: the sum of
// the contributions round(v 2^s) in the high 56 bits, their count in the low
// 8.  The scale 2^s is chosen per exchange, by every CTA alike, from a bound
// B on every contribution's magnitude (fix1_scale): n B 2^s < 2^54, so no sum
// of n contributions can leave the word, and the resolution 2^-s is about
// 2^-53 n B -- relative to a typical value t, n (B / t) 2^-53, far below fp32
// rounding for any bound within 2^20 of the values, whatever their scale.

// 2^s and 2^-s with n B 2^s < 2^54 (B >= 0; a zero or non-finite bound gives
// the scale of B = 1).
__device__ __forceinline__ float2 fix1_scale(float B, int n) {
    float x = B * (float)n;
    if (!(x > 0.f) || !(x < 3.0e38f)) x = (float)n;
    int e = (int)((__float_as_uint(x) >> 23) & 0xffu) - 127;  // floor(log2 x), x normal
    int sh = 53 - e;
    sh = sh > 126 ? 126 : (sh < -126 ? -126 : sh);
    return make_float2(__uint_as_float((unsigned)(sh + 127) << 23),
                       __uint_as_float((unsigned)(127 - sh) << 23));
}

// One contribution v at scale sc (= 2^s); |v sc| must stay below lim = 2^54
// / n (else LB_ERR_RANGE is recorded and zero sent: the bound was wrong).
__device__ __forceinline__ void send_fix1(unsigned long long *w, float v, float sc, float lim,
                                          unsigned *err) {
    float a = v * sc;
    if (!(fabsf(a) < lim)) {
        atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_RANGE));
        a = 0.f;
    }
    red_add_u64(w, (static_cast<unsigned long long>(__float2ll_rn(a)) << 8) + 1ull);
}

__device__ __forceinline__ bool counted1(unsigned long long w, unsigned n) {
    return (unsigned)(w & 0xffull) == n;
}

// The sum held by a complete word, in fp32 (one rounding), at inverse scale inv.
__device__ __forceinline__ float dec_fix1(unsigned long long w, float inv) {
    return __ll2float_rn(static_cast<long long>(w) >> 8) * inv;
}

// ---------------------------------------------------------------- single-linear stage 2
//
// Stage 2 of the single-linear kernels (k_decode, k_decode_multi) runs in
// parts: rows [32 b, 32 b + 32) of path p (lane = row) over words [4 s,
// 4 s + 4) of the row (the last part may be shorter), so a CTA's rows spread
// over many warps however few rows it has.  Each part leaves (the sum of its
// +-1 lookups, even words then odd words) * h[row] in a slot of its own;
// s2_combine adds a row's slots in slot order (path 0's parts, then path
// 1's), so both kernels give the same bits whichever warp ran which part.
constexpr int kPartWords = 4;
__host__ __device__ inline int s2_parts(int R) { return (R + kPartWords - 1) / kPartWords; }

// One part: U (the path's rows, R words each, row 0 at U), h (fp16 of row 0),
// tables tb (word 0's), into dst[row] for rows below nrows.
__device__ __forceinline__ void s2_part(const uint32_t *U, int R, const uint16_t *h,
                                        uint32_t tb, int nrows, int b, int s, float *dst,
                                        uint32_t copy, int lane) {
    const int row = 32 * b + lane, rr = min(row, nrows - 1);
    const uint32_t *Uw = U + rr * R;
    const int w0 = kPartWords * s, w1 = min(R, w0 + kPartWords);
    float acc0 = 0.f, acc1 = 0.f;
    if (w1 - w0 == 4 && (R & 3) == 0) {
        // rows of R = 4k words are 16-byte aligned: one 128-bit load takes the
        // part (a warp's 32 rows at a stride of R words fall in few banks, so
        // a 32-bit load per word would replay up to 16 times)
        const uint4 q = *reinterpret_cast<const uint4 *>(Uw + w0);
        acc0 += lut_word(q.x, copy, tb + w0 * 1024);
        acc1 += lut_word(q.y, copy, tb + (w0 + 1) * 1024);
        acc0 += lut_word(q.z, copy, tb + (w0 + 2) * 1024);
        acc1 += lut_word(q.w, copy, tb + (w0 + 3) * 1024);
    } else {
        int w = w0;
        for (; w + 2 <= w1; w += 2) {
            acc0 += lut_word(Uw[w], copy, tb + w * 1024);
            acc1 += lut_word(Uw[w + 1], copy, tb + (w + 1) * 1024);
        }
        if (w < w1) acc0 += lut_word(Uw[w], copy, tb + w * 1024);
    }
    if (row < nrows) dst[row] = (acc0 + acc1) * half_bits_to_float(h[rr]);
}

// Output row `row`: its nslot slots (stride `stride` floats) added in order.
__device__ __forceinline__ float s2_combine(const float *slots, int stride, int nslot, int row) {
    float y = slots[row];
    for (int k = 1; k < nslot; ++k) y += slots[k * stride + row];
    return y;
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
