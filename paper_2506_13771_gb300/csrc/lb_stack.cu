// lb_stack.cu -- one decode token through n_layers Llama-shaped decoder blocks
// whose seven linears are LittleBit linears, as ONE persistent launch with one
// CTA per SM (littlebit_stack_forward).
//
// Per linear, Prop. 1 (LittleBit, arXiv 2506.13771) is a +-1 reduction over
// d_in (stage 1, rank-r result t) followed by a +-1 reduction over r (stage
// 2), per path, paths summed (Eq. 6).  CTA c owns
//   R_c : a slice of d rows, whole 32-row words    (q, o, down outputs; the
//         residual stream a/h; stage-1 inputs of q, k, v, o, gate, up)
//   F_c : a slice of d_ff rows, whole 32-row words (gate, up outputs; m;
//         stage-1 input of down)
//   K_c : a slice of d_kv rows, multiples of 8     (k, v outputs)
// so stage 2 of one linear and stage 1 of the next run back to back on the
// same CTA; the only exchange is the rank-r all-reduce of t (four per layer).
//
// GB300 choices:
//  * every weight byte a CTA needs for phase X of layer l+1 is fetched by
//    TMA bulk copies (cp.async.bulk) into its phase-X shared buffer right
//    after phase X of layer l finishes: HBM streams in the background of the
//    exchange latency, one layer ahead;
//  * +-1 sums use 4-bit lookup tables in shared memory: 16 signed sums of 4
//    values, stored twice so the two half-warps use disjoint banks; a 32-bit
//    sign word costs 8 table lookups (PRMT forms the address, LDS reads it);
//  * the all-reduce of t accumulates fixed-point values in 64-bit words whose
//    low 8 bits count contributions: each CTA adds (round(v * 2^24) << 8) + 1
//    with one red.add per element and readers poll the words they need until
//    the count reaches the CTA count -- no fence, no separate barrier, and an
//    order-independent (bitwise reproducible) sum;
//  * q and k (not read again at position 0) are computed after the CTA has
//    sent its share of the next exchange, off the critical path.
// Every wait is bounded (about one second); on a timeout the CTA records
// LB_ERR_TIMEOUT, waits for its own bulk copies to land, and returns.
#include <algorithm>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kST = 512;        // threads per CTA
constexpr int kCW = 15;         // compute warps; warp 15 issues the bulk copies
constexpr int kCT = kCW * 32;   // compute threads
constexpr float kFix = 16777216.f;            // 2^24
constexpr float kFixInv = 1.f / 16777216.f;

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

__device__ __forceinline__ void ld_relaxed_v2_u64(const unsigned long long *p,
                                                  unsigned long long &a, unsigned long long &b) {
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];"
                 : "=l"(a), "=l"(b)
                 : "l"(p)
                 : "memory");
}

// ---------------------------------------------------------------- parameters

enum { LQ = 0, LK = 1, LV = 2, LO = 3, LG = 4, LU = 5, LD = 6 };

// Byte offsets (relative to g_smem) of every chunk a phase buffer holds,
// computed on the host from the largest slices of any CTA.
struct Offsets {
    // phase A: stage 2 of the previous layer's down, stage 1 of q, k, v
    int a_Ud[2], a_hd[2], a_ld[2], a_V[3][2], a_g[3][2];
    // phase B: v on the rows attention reads, stage 1 of o, then q, k, v(kv)
    int b_Uat[2], b_hat[2], b_lv[2], b_Vo[2], b_go[2], b_Uq[2], b_hq[2], b_lq[2], b_Uk[2],
        b_hk[2], b_lk[2], b_Uvk[2], b_hvk[2];
    // phase C: stage 2 of o, stage 1 of gate, up
    int c_Uo[2], c_ho[2], c_lo[2], c_Vg[2], c_Vu[2], c_gg[2], c_gu[2];
    // phase D: stage 2 of gate, up, stage 1 of down
    int d_Ug[2], d_Uu[2], d_hg[2], d_hu[2], d_lg[2], d_lu[2], d_Vd[2], d_gd[2];
    int tables, tz, res, xs, ys, yq, tsave;  // work areas
};

struct Params {
    const LinDesc *lin;  // 7 * n_layers descriptors in the workspace
    int n_layers, d, dkv, dff, hd;
    int np[7], r[7][2];  // paths and ranks of q, k, v, o, gate, up, down
    const uint16_t *x0;
    float *out, *q_out, *kv_out;
    unsigned *ws_words;
    unsigned long long plan;
    unsigned long long *xacc;  // exchange words, n_layers * acc_layer
    int acc_layer, offA, offB, offC, offD, lenA, lenB, lenC, lenD;
    float fix_limit;  // |contribution| bound that keeps the fixed-point sum in range
    Offsets o;
};

// ---------------------------------------------------------------- small pieces

__device__ __forceinline__ int wordsR(int r) { return (r + 31) >> 5; }

__device__ __forceinline__ float *sm_f(int off) { return reinterpret_cast<float *>(g_smem + off); }
__device__ __forceinline__ const uint32_t *sm_u32(int off) {
    return reinterpret_cast<const uint32_t *>(g_smem + off);
}
__device__ __forceinline__ const uint16_t *sm_u16(int off) {
    return reinterpret_cast<const uint16_t *>(g_smem + off);
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

__device__ __forceinline__ void split_word(uint32_t word, uint32_t copy, uint32_t &lo,
                                           uint32_t &hi) {
    lo = ((word << 2) & 0x3C3C3C3Cu) | copy;
    hi = ((word >> 2) & 0x3C3C3C3Cu) | copy;
}

// Compute helpers.  Job arrays have a compile-time size NJ (the jobs a step
// could have with two paths per linear) and are indexed with compile-time
// indices only, so they stay in registers; a job that does not exist (a
// linear with one path) has no rows / columns / tables.  All buffers are
// byte offsets into g_smem.

// Nibble tables of one value vector: table n (n < n_tab), entry e = 0..15 is
// sum_{k<4} (bit k of e ? -v : +v)[4n + k] with v_i = src[i] * mul * scale[i]
// (scale: fp16 offset, or -1 for none), stored twice (entries e and 16 + e,
// one copy per half-warp).  Tables at or past n_vals / 4 are zero, so sign
// bits beyond the data (padding) add nothing.
struct TJ {
    int tb;      // byte offset of table 0 (256-aligned)
    int n_tab;   // tables to fill (0: job absent)
    int n_vals;  // values available
    int src;     // byte offset of the fp32 values
    int scale;   // byte offset of the fp16 scales, or -1
    float mul;
};

// One thread per (table, 16-byte quarter): 8 consecutive threads write one
// table's 128 bytes, so the float4 stores of a warp are bank-conflict free.
template <int NJ>
__device__ __forceinline__ void build_tables(const TJ (&J)[NJ]) {
    int cum[NJ + 1];
    cum[0] = 0;
#pragma unroll
    for (int j = 0; j < NJ; ++j) cum[j + 1] = cum[j] + 8 * J[j].n_tab;
    for (int idx = threadIdx.x; idx < cum[NJ]; idx += kCT) {
        int tb = J[0].tb, n_vals = J[0].n_vals, src = J[0].src, scale = J[0].scale, t = idx;
        float mul = J[0].mul;
#pragma unroll
        for (int j = 1; j < NJ; ++j)
            if (idx >= cum[j]) {
                tb = J[j].tb;
                n_vals = J[j].n_vals;
                src = J[j].src;
                scale = J[j].scale;
                mul = J[j].mul;
                t = idx - cum[j];
            }
        const int n = t >> 3, q = t & 7;
        float z[4] = {0.f, 0.f, 0.f, 0.f};
        if (4 * n < n_vals) {
            const float4 v = *reinterpret_cast<const float4 *>(g_smem + src + 16 * n);
            z[0] = v.x * mul;
            z[1] = v.y * mul;
            z[2] = v.z * mul;
            z[3] = v.w * mul;
            if (scale >= 0) {
                const uint2 hb = *reinterpret_cast<const uint2 *>(g_smem + scale + 8 * n);
                z[0] *= half_bits_to_float((uint16_t)(hb.x & 0xffffu));
                z[1] *= half_bits_to_float((uint16_t)(hb.x >> 16));
                z[2] *= half_bits_to_float((uint16_t)(hb.y & 0xffffu));
                z[3] *= half_bits_to_float((uint16_t)(hb.y >> 16));
            }
        }
        // entries 4(q&3) .. 4(q&3)+3: high bits (e3 e2) = q & 3, low bits run 0..3
        const int hb2 = q & 3;
        const float s2 = (hb2 & 1) ? -z[2] : z[2];
        const float s3 = (hb2 & 2) ? -z[3] : z[3];
        const float qv = s2 + s3;
        const float4 r = make_float4(z[0] + z[1] + qv, z[1] - z[0] + qv, z[0] - z[1] + qv,
                                     -z[0] - z[1] + qv);
        *reinterpret_cast<float4 *>(g_smem + tb + n * 128 + q * 16) = r;
    }
}

// Stage 2 job: ys[row] += h[row] * sum_j U_sign[row][j] z[j] for rows
// [0, nrows) of one path; U words [nrows][R] and h at U / h; z tables at tb.
struct UJ {
    int U, h, R, nrows, tb, ys;
};

// A task is 32 rows x a run of words of one job; its lanes (rows) read the
// same 8 tables per word, so lookups are bank-conflict free.  When the jobs
// have fewer 32-row blocks than twice the compute warps, each row's words are
// split into a power-of-two number of runs (shifts only: this runs on the
// critical path of every phase).
template <int NJ>
__device__ __forceinline__ void u_stage(const UJ (&J)[NJ]) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    int blocks = 0;
#pragma unroll
    for (int j = 0; j < NJ; ++j) blocks += (J[j].nrows + 31) >> 5;
    int slog = 0;
#pragma unroll
    for (int k = 0; k < 5; ++k) slog += (blocks << slog) < 2 * kCW ? 1 : 0;
    int cum[NJ + 1], nlog[NJ], wc[NJ];
    cum[0] = 0;
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
        const int R = J[j].R;
        nlog[j] = min(slog, 31 - __clz(max(R, 1)));
        wc[j] = (R + (1 << nlog[j]) - 1) >> nlog[j];
        cum[j + 1] = cum[j] + (((J[j].nrows + 31) >> 5) << nlog[j]);
    }
    for (int task = warp; task < cum[NJ]; task += kCW) {
        int U = J[0].U, h = J[0].h, R = J[0].R, nrows = J[0].nrows, tb = J[0].tb, ys = J[0].ys;
        int t = task, nl = nlog[0], w_c = wc[0];
#pragma unroll
        for (int j = 1; j < NJ; ++j)
            if (task >= cum[j]) {
                U = J[j].U;
                h = J[j].h;
                R = J[j].R;
                nrows = J[j].nrows;
                tb = J[j].tb;
                ys = J[j].ys;
                t = task - cum[j];
                nl = nlog[j];
                w_c = wc[j];
            }
        const int rb = t >> nl, w0 = (t & ((1 << nl) - 1)) * w_c;
        const int w1 = min(w0 + w_c, R);
        const int row = 32 * rb + lane;
        if (row < nrows) {
            const uint32_t *Uw = sm_u32(U) + row * R;
            float acc = 0.f;
            for (int w = w0; w < w1; ++w) {
                uint32_t lo, hi;
                split_word(Uw[w], copy, lo, hi);
                acc += lut8(lo, hi, (uint32_t)(tb + w * 1024));
            }
            atomicAdd(sm_f(ys) + row, acc * half_bits_to_float(sm_u16(h)[row]));
        }
    }
}

// Stage 1 job: all r columns of one path over the CTA's nw input words; V
// words [nw][r] at V, input tables at tb; the partial t goes to dst.
struct VJ {
    int V, r, nw, tb;
    unsigned long long *dst;
};

__device__ __forceinline__ void red_fix(unsigned long long *p, float v, float limit,
                                        unsigned *err) {
    if (!(fabsf(v) < limit)) {
        atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_RANGE));
        v = 0.f;
    }
    const long long f = __float2ll_rn(v * kFix);
    red_add_u64(p, (static_cast<unsigned long long>(f) << 8) + 1ull);
}

// t[j] partial over the slice, added to the exchange words (one contribution
// per CTA per element, also when the slice is empty).  A task is 32 columns
// x all slice words of one job.
template <int NJ>
__device__ __forceinline__ void v_stage(const VJ (&J)[NJ], float limit, unsigned *err) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    int cum[NJ + 1];
    cum[0] = 0;
#pragma unroll
    for (int j = 0; j < NJ; ++j) cum[j + 1] = cum[j] + ((J[j].r + 31) >> 5);
    for (int task = warp; task < cum[NJ]; task += kCW) {
        int V = J[0].V, r = J[0].r, nw = J[0].nw, tb = J[0].tb, t = task;
        unsigned long long *dst = J[0].dst;
#pragma unroll
        for (int j = 1; j < NJ; ++j)
            if (task >= cum[j]) {
                V = J[j].V;
                r = J[j].r;
                nw = J[j].nw;
                tb = J[j].tb;
                dst = J[j].dst;
                t = task - cum[j];
            }
        const int col = 32 * t + lane;
        if (col < r) {
            float acc = 0.f;
            const uint32_t *Vw = sm_u32(V) + col;
            for (int w = 0; w < nw; ++w) {
                uint32_t lo, hi;
                split_word(Vw[w * r], copy, lo, hi);
                acc += lut8(lo, hi, (uint32_t)(tb + w * 1024));
            }
            red_fix(dst + col, acc, limit, err);
        }
    }
}

// Barrier over the compute warps only (named barrier 1).
__device__ __forceinline__ void csync() { asm volatile("bar.sync 1, %0;" ::"n"(kCT) : "memory"); }

// AND of pred over the compute threads, returned to each of them.
__device__ __forceinline__ int csync_and(int pred) {
    int r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.s32 p, %1, 0;\n\tbar.red.and.pred q, 1, %2, p;\n\t"
        "selp.s32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(pred), "n"(kCT)
        : "memory");
    return r;
}

// Sum of v over the compute threads, returned to each of them (one barrier:
// the partials are read back before any later barrier lets them be rewritten).
__device__ float csum(float v) {
    __shared__ float s_part[kCW];
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = v;
    csync();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kCW; ++w) t += s_part[w];
    return t;
}

__device__ __forceinline__ float sum_sq(const float *v, int n) {
    float s = 0.f;
    for (int i = threadIdx.x; i < n; i += kCT) s += v[i] * v[i];
    return csum(s);
}

__device__ __forceinline__ void zero_f(float *p, int n) {
    for (int i = threadIdx.x; i < n; i += kCT) p[i] = 0.f;
}

// Zero this CTA's stripe of an exchange region whose readers are all done.
__device__ __forceinline__ void zero_stripe(unsigned long long *region, int len) {
    const int a = (int)((long long)blockIdx.x * len / gridDim.x);
    const int b = (int)((long long)(blockIdx.x + 1) * len / gridDim.x);
    for (int i = a + threadIdx.x; i < b; i += kCT) region[i] = 0ull;
}

__device__ __forceinline__ bool sticky(const unsigned *ws_words) {
    return ld_relaxed_gpu(ws_words + kErrWord) != 0u;
}

__device__ __forceinline__ void record(unsigned *ws_words, lb_status st) {
    atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(st));
}

// Wait until each of region[0..n) counts n_ctas contributions and decode the
// sums into out[0..n).  Bounded; returns false (to every compute thread) on
// failure.
__device__ __noinline__ bool poll_decode(const unsigned long long *region, int n, unsigned n_ctas,
                                         float *out, unsigned *ws_words) {
    int ok = 1;
    for (int i = 2 * threadIdx.x; i < n && ok; i += 2 * kCT) {
        unsigned long long t0 = 0;
        for (int spin = 0;; ++spin) {
            unsigned long long a, b;
            ld_relaxed_v2_u64(region + i, a, b);
            const bool done = (a & 0xffull) == n_ctas && (i + 1 >= n || (b & 0xffull) == n_ctas);
            if (done) {
                out[i] = __ll2float_rn((long long)a >> 8) * kFixInv;
                if (i + 1 < n) out[i + 1] = __ll2float_rn((long long)b >> 8) * kFixInv;
                break;
            }
            if ((spin & 15) == 15) {
                if (sticky(ws_words)) {
                    ok = 0;
                    break;
                }
                const unsigned long long now = globaltimer_ns();
                if (t0 == 0) t0 = now;
                if (now - t0 > kWaitLimitNs) {
                    record(ws_words, LB_ERR_TIMEOUT);
                    ok = 0;
                    break;
                }
            }
        }
    }
    return csync_and(ok) != 0;
}

// Bounded wait on an mbarrier phase by every compute thread.
__device__ bool wait_full(unsigned long long *bar, unsigned parity, unsigned *ws_words) {
    int ok = 1;
    if (!mbar_try_wait(bar, parity)) {
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(bar, parity)) {
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                record(ws_words, LB_ERR_TIMEOUT);
                ok = 0;
                break;
            }
        }
    }
    return csync_and(ok) != 0;
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }

// ---------------------------------------------------------------- the kernel

struct Part {
    int dw0, nd, fw0, nf, k0, nkv;
};

// The bulk-copy producer (lane 0 of warp 15).  Phase X of layer l has its
// own buffer; the copies for X(l+1) are issued once the compute warps have
// released X(l) (empty barrier), and land on the full barrier of X.
struct Loader {
    const Params *P;
    Part s;
    unsigned long long *full;

    __device__ void copy(int dst, const void *src, unsigned bytes, unsigned long long *b) const {
        if (bytes == 0) return;
        mbar_expect_tx(b, bytes);
        bulk_g2s(g_smem + dst, src, bytes, b);
    }
    // U rows [row0, row0 + nrows) of a path (R words each) and their h.
    __device__ void rows(int dU, int dh, const LinDesc &L, int p, int row0, int nrows,
                         unsigned long long *b) const {
        const int R = wordsR(L.r[p]);
        copy(dU, L.u[p] + (size_t)row0 * R, (unsigned)(nrows * R * 4), b);
        copy(dh, L.h[p] + row0, (unsigned)(nrows * 2), b);
    }
    __device__ void vslice(int dV, int dg, const LinDesc &L, int p, int w0, int nw,
                           unsigned long long *b) const {
        copy(dV, L.v[p] + (size_t)w0 * L.r[p], (unsigned)(nw * L.r[p] * 4), b);
        copy(dg, L.g[p] + 32 * w0, (unsigned)(nw * 64), b);
    }
    __device__ void lat(int dl, const LinDesc &L, int p, unsigned long long *b) const {
        copy(dl, L.l[p], (unsigned)(L.r[p] * 2), b);
    }

    // phase A of layer l (0 <= l <= n_layers): down of layer l-1 on R_c rows,
    // stage 1 of q, k, v of layer l on R_c (absent for l = n_layers).
    __device__ void issue_A(int l) const {
        unsigned long long *b = full + 0;
        const Offsets &o = P->o;
        if (l > 0) {
            const LinDesc &D = P->lin[7 * (l - 1) + LD];
            for (int p = 0; p < D.n_paths; ++p) {
                rows(o.a_Ud[p], o.a_hd[p], D, p, 32 * s.dw0, 32 * s.nd, b);
                lat(o.a_ld[p], D, p, b);
            }
        }
        if (l < P->n_layers) {
            for (int k = 0; k < 3; ++k) {
                const LinDesc &L = P->lin[7 * l + k];
                for (int p = 0; p < L.n_paths; ++p)
                    vslice(o.a_V[k][p], o.a_g[k][p], L, p, s.dw0, s.nd, b);
            }
        }
        mbar_arrive(b);
    }
    __device__ void issue_B(int l) const {
        unsigned long long *b = full + 1;
        const Offsets &o = P->o;
        const LinDesc &Q = P->lin[7 * l + LQ], &K = P->lin[7 * l + LK], &V = P->lin[7 * l + LV],
                      &O = P->lin[7 * l + LO];
        const int grp = P->d / P->dkv;
        for (int p = 0; p < V.n_paths; ++p) {
            const int R = wordsR(V.r[p]);
            // the v rows read by each 32-row word of R_c are contiguous
            for (int g = 0; g < s.nd; ++g) {
                const int o0 = 32 * (s.dw0 + g), head = o0 / P->hd;
                const int vrow = (head / grp) * P->hd + (o0 - head * P->hd);
                copy(o.b_Uat[p] + g * 32 * R * 4, V.u[p] + (size_t)vrow * R, 32u * R * 4, b);
                copy(o.b_hat[p] + g * 64, V.h[p] + vrow, 64u, b);
            }
            lat(o.b_lv[p], V, p, b);
            rows(o.b_Uvk[p], o.b_hvk[p], V, p, s.k0, s.nkv, b);
        }
        for (int p = 0; p < O.n_paths; ++p) vslice(o.b_Vo[p], o.b_go[p], O, p, s.dw0, s.nd, b);
        for (int p = 0; p < Q.n_paths; ++p) {
            rows(o.b_Uq[p], o.b_hq[p], Q, p, 32 * s.dw0, 32 * s.nd, b);
            lat(o.b_lq[p], Q, p, b);
        }
        for (int p = 0; p < K.n_paths; ++p) {
            rows(o.b_Uk[p], o.b_hk[p], K, p, s.k0, s.nkv, b);
            lat(o.b_lk[p], K, p, b);
        }
        mbar_arrive(b);
    }
    __device__ void issue_C(int l) const {
        unsigned long long *b = full + 2;
        const Offsets &o = P->o;
        const LinDesc &O = P->lin[7 * l + LO], &G = P->lin[7 * l + LG], &U = P->lin[7 * l + LU];
        for (int p = 0; p < O.n_paths; ++p) {
            rows(o.c_Uo[p], o.c_ho[p], O, p, 32 * s.dw0, 32 * s.nd, b);
            lat(o.c_lo[p], O, p, b);
        }
        for (int p = 0; p < G.n_paths; ++p) vslice(o.c_Vg[p], o.c_gg[p], G, p, s.dw0, s.nd, b);
        for (int p = 0; p < U.n_paths; ++p) vslice(o.c_Vu[p], o.c_gu[p], U, p, s.dw0, s.nd, b);
        mbar_arrive(b);
    }
    __device__ void issue_D(int l) const {
        unsigned long long *b = full + 3;
        const Offsets &o = P->o;
        const LinDesc &G = P->lin[7 * l + LG], &U = P->lin[7 * l + LU], &D = P->lin[7 * l + LD];
        for (int p = 0; p < G.n_paths; ++p) {
            rows(o.d_Ug[p], o.d_hg[p], G, p, 32 * s.fw0, 32 * s.nf, b);
            lat(o.d_lg[p], G, p, b);
        }
        for (int p = 0; p < U.n_paths; ++p) {
            rows(o.d_Uu[p], o.d_hu[p], U, p, 32 * s.fw0, 32 * s.nf, b);
            lat(o.d_lu[p], U, p, b);
        }
        for (int p = 0; p < D.n_paths; ++p) vslice(o.d_Vd[p], o.d_gd[p], D, p, s.fw0, s.nf, b);
        mbar_arrive(b);
    }
    __device__ void issue(int buf, int l) const {
        if (buf == 0) issue_A(l);
        else if (buf == 1) issue_B(l);
        else if (buf == 2) issue_C(l);
        else issue_D(l);
    }
};

// Producer loop: issue every phase buffer of every layer in consumption
// order, each after the compute warps released its previous use.  Waits are
// bounded and stop at the first recorded error; before returning, the
// producer waits (bounded) for all copies it issued to land, so none arrives
// after the CTA is gone.
__device__ void producer(const Loader &ld, unsigned long long *empty, unsigned *ws_words) {
    const int L = ld.P->n_layers;
    int last_use[4] = {0, 0, 0, 0};
    for (int b = 0; b < 4; ++b) ld.issue(b, 0);
    bool ok = true;
    for (int l = 1; l <= L && ok; ++l) {
        for (int b = 0; b < 4 && ok; ++b) {
            if (b > 0 && l == L) break;  // the final phase needs only buffer A
            const unsigned parity = (unsigned)((l - 1) & 1);
            unsigned long long t0 = 0;
            for (int spin = 0; !mbar_try_wait(empty + b, parity); ++spin) {
                if ((spin & 63) == 63) {
                    if (sticky(ws_words)) {
                        ok = false;
                        break;
                    }
                    const unsigned long long now = globaltimer_ns();
                    if (t0 == 0) t0 = now;
                    if (now - t0 > kWaitLimitNs) {
                        record(ws_words, LB_ERR_TIMEOUT);
                        ok = false;
                        break;
                    }
                }
            }
            if (!ok) break;
            fence_proxy_async();
            ld.issue(b, l);
            last_use[b] = l;
        }
    }
    // drain: the last issued use of each buffer has parity last_use & 1
    for (int b = 0; b < 4; ++b) {
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(ld.full + b, (unsigned)(last_use[b] & 1)))
            if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
}

__global__ void __launch_bounds__(kST, 1) k_stack(const __grid_constant__ Params P) {
    __shared__ __align__(8) unsigned long long full[4], empty[4];
    __shared__ int s_last;
    unsigned *err = P.ws_words + kErrWord;
    if (sticky(P.ws_words)) return;
    if (*reinterpret_cast<const volatile unsigned long long *>(P.ws_words + kPlanWord) != P.plan) {
        if (blockIdx.x == 0 && threadIdx.x == 0) record(P.ws_words, LB_ERR_PLAN);
        return;
    }
    const int N = gridDim.x, c = blockIdx.x;
    const unsigned n_ctas = (unsigned)N;
    Part s;
    {
        const int Wd = P.d >> 5, Wf = P.dff >> 5, Ukv = P.dkv >> 3;
        s.dw0 = (int)((long long)c * Wd / N);
        s.nd = (int)((long long)(c + 1) * Wd / N) - s.dw0;
        s.fw0 = (int)((long long)c * Wf / N);
        s.nf = (int)((long long)(c + 1) * Wf / N) - s.fw0;
        const int u0 = (int)((long long)c * Ukv / N), u1 = (int)((long long)(c + 1) * Ukv / N);
        s.k0 = 8 * u0;
        s.nkv = 8 * (u1 - u0);
    }
    if (threadIdx.x == 0) {
        for (int b = 0; b < 4; ++b) {
            mbar_init(full + b, 1);
            mbar_init(empty + b, 1);
        }
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x >= kCT) {
        if (threadIdx.x == kCT) producer(Loader{&P, s, full}, empty, P.ws_words);
        return;
    }

    // ------------------------------------------------------------ compute warps
    const int nd = s.nd, nf = s.nf, nkv = s.nkv;
    const int rows_d = 32 * nd, rows_f = 32 * nf;
    const Offsets &o = P.o;
    float *res = sm_f(o.res), *xs = sm_f(o.xs), *ys = sm_f(o.ys), *yq = sm_f(o.yq);
    float *tz = sm_f(o.tz);
    for (int i = threadIdx.x; i < rows_d; i += kCT)
        res[i] = bf16_bits_to_float(P.x0[32 * s.dw0 + i]);
    int nr[7];
#pragma unroll
    for (int k = 0; k < 7; ++k) nr[k] = P.r[k][0] + (P.np[k] > 1 ? P.r[k][1] : 0);
    const int ssA = nr[LQ] + nr[LK] + nr[LV], ssC = nr[LG] + nr[LU];
    const bool lead = threadIdx.x == 0;
    // rank and presence of path p of linear k
    auto rk = [&](int k, int p) { return p < P.np[k] ? P.r[k][p] : 0; };
    auto release = [&](int b) {
        csync();
        if (lead) mbar_arrive(empty + b);
    };
    // stage 2 of down (both paths) on R_c into ys, from t in tz
    auto down_rows = [&]() {
        TJ T[2];
        UJ U[2];
        int tb = o.tables, off = 0;
#pragma unroll
        for (int p = 0; p < 2; ++p) {
            const int r = rk(LD, p), R = r ? wordsR(r) : 1;
            T[p] = TJ{tb, r ? 8 * R : 0, r, o.tz + 4 * off, o.a_ld[p], 1.f};
            U[p] = UJ{o.a_Ud[p], o.a_hd[p], R, r ? rows_d : 0, tb, o.ys};
            tb += r ? R * 1024 : 0;
            off += r;
        }
        zero_f(ys, rows_d);
        build_tables(T);
        csync();
        u_stage(U);
        csync();
    };
#define FAIL_EXIT() return

    for (int l = 0; l < P.n_layers; ++l) {
        unsigned long long *xA = P.xacc + (size_t)l * P.acc_layer + P.offA;
        unsigned long long *xB = P.xacc + (size_t)l * P.acc_layer + P.offB;
        unsigned long long *xC = P.xacc + (size_t)l * P.acc_layer + P.offC;
        unsigned long long *xD = P.xacc + (size_t)l * P.acc_layer + P.offD;
        const unsigned par = (unsigned)(l & 1);

        // ================= phase A: a = h + Down_{l-1}(m) on R_c; stage 1 of q, k, v
        if (l > 0) {
            if (!poll_decode(xD - P.acc_layer, nr[LD], n_ctas, tz, P.ws_words)) FAIL_EXIT();
            zero_stripe(xC - P.acc_layer, P.lenC);
        }
        if (!wait_full(full + 0, par, P.ws_words)) FAIL_EXIT();
        if (l > 0) {
            down_rows();
            for (int i = threadIdx.x; i < rows_d; i += kCT) res[i] += ys[i];
            csync();
        }
        {
            const float ss = sum_sq(res, rows_d);
            if (lead) red_fix(xA + ssA, ss, P.fix_limit, err);
            TJ T[6];
            VJ V[6];
            int tb = o.tables;
            unsigned long long *dst = xA;
#pragma unroll
            for (int k = 0; k < 3; ++k)
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const int r = rk(k, p);
                    T[2 * k + p] = TJ{tb, r ? 8 * nd : 0, rows_d, o.res, o.a_g[k][p], 1.f};
                    V[2 * k + p] = VJ{o.a_V[k][p], r, nd, tb, dst};
                    tb += r ? nd * 1024 : 0;
                    dst += r;
                }
            build_tables(T);
            csync();
            v_stage(V, P.fix_limit, err);
        }
        release(0);

        // ================= phase B: v rows for attention, stage 1 of o; then q, k, v out
        if (!poll_decode(xA, ssA + 1, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        if (l > 0) zero_stripe(xD - P.acc_layer, P.lenD);
        if (!wait_full(full + 1, par, P.ws_words)) FAIL_EXIT();
        {
            const float inv = rsqrtf(tz[ssA] / (float)P.d);
            int tb = o.tables;
            const int tb_v = tb;
            {
                TJ T[2];
                UJ U[2];
#pragma unroll
                for (int p = 0, off = nr[LQ] + nr[LK]; p < 2; ++p) {
                    const int r = rk(LV, p), R = r ? wordsR(r) : 1;
                    T[p] = TJ{tb, r ? 8 * R : 0, r, o.tz + 4 * off, o.b_lv[p], inv};
                    U[p] = UJ{o.b_Uat[p], o.b_hat[p], R, r ? rows_d : 0, tb, o.xs};
                    tb += r ? R * 1024 : 0;
                    off += r;
                }
                zero_f(xs, rows_d);
                build_tables(T);
                csync();
                u_stage(U);
                csync();
            }
            {
                TJ T[2];
                VJ V[2];
                unsigned long long *dst = xB;
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const int r = rk(LO, p);
                    T[p] = TJ{tb, r ? 8 * nd : 0, rows_d, o.xs, o.b_go[p], 1.f};
                    V[p] = VJ{o.b_Vo[p], r, nd, tb, dst};
                    tb += r ? nd * 1024 : 0;
                    dst += r;
                }
                build_tables(T);
                csync();
                v_stage(V, P.fix_limit, err);
            }
            // ---- off the critical path, while exchange B is in flight:
            //      k and v on K_c, and path 0 of q on R_c (path 1 of q runs
            //      after exchange C is sent, from the saved t and rms)
            {
                const int rq1 = rk(LQ, 1);
                if (rq1) {
                    float *sv = sm_f(o.tsave);
                    for (int i = threadIdx.x; i < rq1; i += kCT) sv[i] = tz[rk(LQ, 0) + i];
                    if (lead) sv[rq1] = inv;
                }
                TJ T[3];
                UJ U[5];
                int tbv = tb_v;
                {
                    const int r = rk(LQ, 0), R = wordsR(r);
                    T[0] = TJ{tb, 8 * R, r, o.tz, o.b_lq[0], inv};
                    U[0] = UJ{o.b_Uq[0], o.b_hq[0], R, rows_d, tb, o.yq};
                    tb += R * 1024;
                }
#pragma unroll
                for (int p = 0, off = nr[LQ]; p < 2; ++p) {
                    const int r = rk(LK, p), R = r ? wordsR(r) : 1;
                    T[1 + p] = TJ{tb, r ? 8 * R : 0, r, o.tz + 4 * off, o.b_lk[p], inv};
                    U[1 + p] = UJ{o.b_Uk[p], o.b_hk[p], R, r ? nkv : 0, tb, o.ys};
                    tb += r ? R * 1024 : 0;
                    off += r;
                }
#pragma unroll
                for (int p = 0; p < 2; ++p) {  // v on K_c reuses v's tables
                    const int r = rk(LV, p), R = r ? wordsR(r) : 1;
                    U[3 + p] = UJ{o.b_Uvk[p], o.b_hvk[p], R, r ? nkv : 0, tbv, o.ys + 4 * nkv};
                    tbv += r ? R * 1024 : 0;
                }
                zero_f(yq, rows_d);
                zero_f(ys, 2 * nkv);
                build_tables(T);
                csync();
                u_stage(U);
                csync();
                if (P.kv_out)
                    for (int i = threadIdx.x; i < nkv; i += kCT) {
                        P.kv_out[((size_t)l * 2 + 0) * P.dkv + s.k0 + i] = ys[i];
                        P.kv_out[((size_t)l * 2 + 1) * P.dkv + s.k0 + i] = ys[nkv + i];
                    }
                if (!rq1 && P.q_out)
                    for (int i = threadIdx.x; i < rows_d; i += kCT)
                        P.q_out[(size_t)l * P.d + 32 * s.dw0 + i] = yq[i];
            }
        }

        // ================= phase C: h = a + O(attn) on R_c; stage 1 of gate, up
        if (!poll_decode(xB, nr[LO], n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(xA, P.lenA);
        if (!wait_full(full + 2, par, P.ws_words)) FAIL_EXIT();
        {
            {
                TJ T[2];
                UJ U[2];
                int tb = o.tables;
#pragma unroll
                for (int p = 0, off = 0; p < 2; ++p) {
                    const int r = rk(LO, p), R = r ? wordsR(r) : 1;
                    T[p] = TJ{tb, r ? 8 * R : 0, r, o.tz + 4 * off, o.c_lo[p], 1.f};
                    U[p] = UJ{o.c_Uo[p], o.c_ho[p], R, r ? rows_d : 0, tb, o.ys};
                    tb += r ? R * 1024 : 0;
                    off += r;
                }
                zero_f(ys, rows_d);
                build_tables(T);
                csync();
                u_stage(U);
                csync();
            }
            for (int i = threadIdx.x; i < rows_d; i += kCT) res[i] += ys[i];
            csync();
            const float ss = sum_sq(res, rows_d);
            if (lead) red_fix(xC + ssC, ss, P.fix_limit, err);
            TJ T[4];
            VJ V[4];
            int tb = o.tables;
            unsigned long long *dst = xC;
#pragma unroll
            for (int k = 0; k < 2; ++k)
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const int r = rk(LG + k, p);
                    const int g = k ? o.c_gu[p] : o.c_gg[p], Vw = k ? o.c_Vu[p] : o.c_Vg[p];
                    T[2 * k + p] = TJ{tb, r ? 8 * nd : 0, rows_d, o.res, g, 1.f};
                    V[2 * k + p] = VJ{Vw, r, nd, tb, dst};
                    tb += r ? nd * 1024 : 0;
                    dst += r;
                }
            build_tables(T);
            csync();
            v_stage(V, P.fix_limit, err);
        }
        // ---- off the critical path, while exchange C is in flight: path 1 of q
        if (rk(LQ, 1)) {
            csync();
            const int r = rk(LQ, 1), R = wordsR(r);
            TJ T[1] = {TJ{o.tables, 8 * R, r, o.tsave, o.b_lq[1], sm_f(o.tsave)[r]}};
            UJ U[1] = {UJ{o.b_Uq[1], o.b_hq[1], R, rows_d, o.tables, o.yq}};
            build_tables(T);
            csync();
            u_stage(U);
            csync();
            if (P.q_out)
                for (int i = threadIdx.x; i < rows_d; i += kCT)
                    P.q_out[(size_t)l * P.d + 32 * s.dw0 + i] = yq[i];
        }
        release(1);
        release(2);

        // ================= phase D: m = silu(gate) * up on F_c; stage 1 of down
        if (!poll_decode(xC, ssC + 1, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(xB, P.lenB);
        if (!wait_full(full + 3, par, P.ws_words)) FAIL_EXIT();
        {
            const float inv = rsqrtf(tz[ssC] / (float)P.d);
            {
                TJ T[4];
                UJ U[4];
                int tb = o.tables;
#pragma unroll
                for (int k = 0; k < 2; ++k)
#pragma unroll
                    for (int p = 0; p < 2; ++p) {
                        const int r = rk(LG + k, p), R = r ? wordsR(r) : 1;
                        const int off = (k ? nr[LG] : 0) + (p ? rk(LG + k, 0) : 0);
                        const int lo16 = k ? o.d_lu[p] : o.d_lg[p];
                        const int Uw = k ? o.d_Uu[p] : o.d_Ug[p], h = k ? o.d_hu[p] : o.d_hg[p];
                        T[2 * k + p] = TJ{tb, r ? 8 * R : 0, r, o.tz + 4 * off, lo16, inv};
                        U[2 * k + p] = UJ{Uw, h, R, r ? rows_f : 0, tb, o.ys + (k ? 4 * rows_f : 0)};
                        tb += r ? R * 1024 : 0;
                    }
                zero_f(ys, 2 * rows_f);
                build_tables(T);
                csync();
                u_stage(U);
                csync();
            }
            for (int i = threadIdx.x; i < rows_f; i += kCT) xs[i] = silu(ys[i]) * ys[rows_f + i];
            csync();
            TJ T[2];
            VJ V[2];
            int tb = o.tables;
            unsigned long long *dst = xD;
#pragma unroll
            for (int p = 0; p < 2; ++p) {
                const int r = rk(LD, p);
                T[p] = TJ{tb, r ? 8 * nf : 0, rows_f, o.xs, o.d_gd[p], 1.f};
                V[p] = VJ{o.d_Vd[p], r, nf, tb, dst};
                tb += r ? nf * 1024 : 0;
                dst += r;
            }
            build_tables(T);
            csync();
            v_stage(V, P.fix_limit, err);
        }
        release(3);
    }

    // ================= final: out = h + Down_{L-1}(m) on R_c
    {
        const int l = P.n_layers;
        unsigned long long *xDl = P.xacc + (size_t)(l - 1) * P.acc_layer + P.offD;
        if (!poll_decode(xDl, nr[LD], n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(P.xacc + (size_t)(l - 1) * P.acc_layer + P.offC, P.lenC);
        if (!wait_full(full + 0, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        down_rows();
        for (int i = threadIdx.x; i < rows_d; i += kCT) P.out[32 * s.dw0 + i] = res[i] + ys[i];
        // The last CTA to finish has seen every other CTA's reads of the final
        // region: it clears that region and the counters for the next launch.
        if (lead) {
            __threadfence();
            s_last = atomicAdd(P.ws_words + kDoneWord, 1u) == n_ctas - 1;
        }
        csync();
        if (s_last) {
            __threadfence();
            for (int i = threadIdx.x; i < P.lenD; i += kCT) xDl[i] = 0ull;
            if (lead) P.ws_words[kDoneWord] = 0u;
        }
    }
#undef FAIL_EXIT
}

// ---------------------------------------------------------------- descriptors

constexpr int kDescChunk = 256;
struct DescChunk {
    int count;
    LinDesc d[kDescChunk];
};

// Copies descriptors from kernel-parameter space into the workspace, so the
// host array reaches the device with the launch itself.
__global__ void k_upload_desc(const __grid_constant__ DescChunk chunk, LinDesc *dst) {
    const int nwords = chunk.count * (int)(sizeof(LinDesc) / sizeof(uint32_t));
    const uint32_t *src = reinterpret_cast<const uint32_t *>(chunk.d);
    uint32_t *out = reinterpret_cast<uint32_t *>(dst);
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nwords; i += gridDim.x * blockDim.x)
        out[i] = src[i];
}

__global__ void k_set_plan(unsigned *ws_words, unsigned long long plan) {
    *reinterpret_cast<unsigned long long *>(ws_words + kPlanWord) = plan;
}

int rsum(const lb_linear &L) {
    int s = 0;
    for (int p = 0; p < L.n_paths; ++p) s += L.path[p].r;
    return s;
}

int up(int n, int a) { return (n + a - 1) / a * a; }

// Exchange words per layer: A = t of q, k, v + ss(a); B = t of o;
// C = t of gate, up + ss(h); D = t of down; each region padded to 32 words.
struct XLayout {
    int acc_layer, offA, offB, offC, offD, lenA, lenB, lenC, lenD;
};

XLayout xlayout(const lb_linear *lin) {
    XLayout X{};
    X.lenA = rsum(lin[LQ]) + rsum(lin[LK]) + rsum(lin[LV]) + 1;
    X.lenB = rsum(lin[LO]);
    X.lenC = rsum(lin[LG]) + rsum(lin[LU]) + 1;
    X.lenD = rsum(lin[LD]);
    X.offA = 0;
    X.offB = X.offA + up(X.lenA, 32);
    X.offC = X.offB + up(X.lenB, 32);
    X.offD = X.offC + up(X.lenC, 32);
    X.acc_layer = X.offD + up(X.lenD, 32);
    return X;
}

size_t desc_bytes_for(int n_layers) {
    return ((size_t)7 * n_layers * sizeof(LinDesc) + 255) & ~(size_t)255;
}

// Shared-memory plan from the largest slices any CTA gets.
struct SmemPlan {
    Offsets o;
    int bytes;
};

SmemPlan smem_plan(const lb_linear *lin, const StackShape &sh, int N) {
    const int nd = (sh.d / 32 + N - 1) / N, nf = (sh.dff / 32 + N - 1) / N;
    const int nkv = 8 * ((sh.dkv / 8 + N - 1) / N);
    SmemPlan S{};
    Offsets &o = S.o;
    int at = 0;
    auto take = [&at](int bytes) {
        const int off = at;
        at += up(bytes, 16);
        return off;
    };
    auto R = [&](int k, int p) { return (lin[k].path[p].r + 31) / 32; };
    auto r = [&](int k, int p) { return lin[k].path[p].r; };
    for (int p = 0; p < 2; ++p) {
        const bool dn = p < lin[LD].n_paths;
        o.a_Ud[p] = take(dn ? 32 * nd * R(LD, p) * 4 : 0);
        o.a_hd[p] = take(dn ? 64 * nd : 0);
        o.a_ld[p] = take(dn ? 2 * r(LD, p) : 0);
        for (int k = 0; k < 3; ++k) {
            const bool ok = p < lin[k].n_paths;
            o.a_V[k][p] = take(ok ? nd * r(k, p) * 4 : 0);
            o.a_g[k][p] = take(ok ? 64 * nd : 0);
        }
    }
    at = up(at, 128);
    for (int p = 0; p < 2; ++p) {
        const bool v = p < lin[LV].n_paths, oo = p < lin[LO].n_paths, q = p < lin[LQ].n_paths,
                   k = p < lin[LK].n_paths;
        o.b_Uat[p] = take(v ? 32 * nd * R(LV, p) * 4 : 0);
        o.b_hat[p] = take(v ? 64 * nd : 0);
        o.b_lv[p] = take(v ? 2 * r(LV, p) : 0);
        o.b_Uvk[p] = take(v ? nkv * R(LV, p) * 4 : 0);
        o.b_hvk[p] = take(v ? 2 * nkv : 0);
        o.b_Vo[p] = take(oo ? nd * r(LO, p) * 4 : 0);
        o.b_go[p] = take(oo ? 64 * nd : 0);
        o.b_Uq[p] = take(q ? 32 * nd * R(LQ, p) * 4 : 0);
        o.b_hq[p] = take(q ? 64 * nd : 0);
        o.b_lq[p] = take(q ? 2 * r(LQ, p) : 0);
        o.b_Uk[p] = take(k ? nkv * R(LK, p) * 4 : 0);
        o.b_hk[p] = take(k ? 2 * nkv : 0);
        o.b_lk[p] = take(k ? 2 * r(LK, p) : 0);
    }
    at = up(at, 128);
    for (int p = 0; p < 2; ++p) {
        const bool oo = p < lin[LO].n_paths, g = p < lin[LG].n_paths, u = p < lin[LU].n_paths;
        o.c_Uo[p] = take(oo ? 32 * nd * R(LO, p) * 4 : 0);
        o.c_ho[p] = take(oo ? 64 * nd : 0);
        o.c_lo[p] = take(oo ? 2 * r(LO, p) : 0);
        o.c_Vg[p] = take(g ? nd * r(LG, p) * 4 : 0);
        o.c_gg[p] = take(g ? 64 * nd : 0);
        o.c_Vu[p] = take(u ? nd * r(LU, p) * 4 : 0);
        o.c_gu[p] = take(u ? 64 * nd : 0);
    }
    at = up(at, 128);
    for (int p = 0; p < 2; ++p) {
        const bool g = p < lin[LG].n_paths, u = p < lin[LU].n_paths, dd = p < lin[LD].n_paths;
        o.d_Ug[p] = take(g ? 32 * nf * R(LG, p) * 4 : 0);
        o.d_hg[p] = take(g ? 64 * nf : 0);
        o.d_lg[p] = take(g ? 2 * r(LG, p) : 0);
        o.d_Uu[p] = take(u ? 32 * nf * R(LU, p) * 4 : 0);
        o.d_hu[p] = take(u ? 64 * nf : 0);
        o.d_lu[p] = take(u ? 2 * r(LU, p) : 0);
        o.d_Vd[p] = take(dd ? nf * r(LD, p) * 4 : 0);
        o.d_gd[p] = take(dd ? 64 * nf : 0);
    }
    // nibble tables: the largest set one phase holds at once
    auto utab = [&](int k) {
        int b = 0;
        for (int p = 0; p < lin[k].n_paths; ++p) b += R(k, p) * 1024;
        return b;
    };
    auto vtab = [&](int k, int nw) { return lin[k].n_paths * nw * 1024; };
    int tabs = utab(LD);
    tabs = std::max(tabs, vtab(LQ, nd) + vtab(LK, nd) + vtab(LV, nd));
    tabs = std::max(tabs, utab(LV) + vtab(LO, nd) + utab(LQ) + utab(LK));
    tabs = std::max(tabs, utab(LO));
    tabs = std::max(tabs, vtab(LG, nd) + vtab(LU, nd));
    tabs = std::max(tabs, utab(LG) + utab(LU));
    tabs = std::max(tabs, vtab(LD, nf));
    at = up(at, 256);
    o.tables = at;
    at += tabs;
    int tz_n = rsum(lin[LQ]) + rsum(lin[LK]) + rsum(lin[LV]) + 1;
    tz_n = std::max(tz_n, rsum(lin[LO]));
    tz_n = std::max(tz_n, rsum(lin[LG]) + rsum(lin[LU]) + 1);
    tz_n = std::max(tz_n, rsum(lin[LD]));
    o.tz = take(4 * (tz_n + 1));
    o.res = take(4 * 32 * nd);
    o.xs = take(4 * 32 * std::max(nd, nf));
    o.ys = take(4 * std::max(32 * nd, std::max(2 * nkv, 2 * 32 * nf)));
    o.yq = take(4 * 32 * nd);
    o.tsave = take(4 * (lin[LQ].path[lin[LQ].n_paths - 1].r + 4));
    S.bytes = up(at, 128);
    return S;
}

}  // namespace

static_assert(sizeof(LinDesc) % sizeof(uint32_t) == 0, "descriptor is copied as words");

size_t stack_ws_bytes_after_header(const lb_linear *lin, int n_layers) {
    const XLayout X = xlayout(lin);
    return desc_bytes_for(n_layers) + (size_t)n_layers * X.acc_layer * sizeof(unsigned long long);
}

cudaError_t launch_stack_prepare(const lb_linear *lin, int n_layers, unsigned long long plan,
                                 unsigned *ws_words, char *ws_after_header, cudaStream_t s) {
    const XLayout X = xlayout(lin);
    LinDesc *desc = reinterpret_cast<LinDesc *>(ws_after_header);
    char *xacc = ws_after_header + desc_bytes_for(n_layers);
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, 2 * sizeof(unsigned), s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(xacc, 0, (size_t)n_layers * X.acc_layer * sizeof(unsigned long long),
                            s);
    if (e != cudaSuccess) return e;
    const int n_lin = 7 * n_layers;
    for (int first = 0; first < n_lin; first += kDescChunk) {
        DescChunk ch;
        ch.count = n_lin - first < kDescChunk ? n_lin - first : kDescChunk;
        for (int i = 0; i < ch.count; ++i) ch.d[i] = make_desc(lin[first + i]);
        k_upload_desc<<<8, 256, 0, s>>>(ch, desc + first);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    k_set_plan<<<1, 1, 0, s>>>(ws_words, plan);
    return cudaGetLastError();
}

bool stack_supported(const lb_linear *lin, const StackShape &sh, int num_sms) {
    for (int k = 0; k < 7; ++k)
        for (int p = 0; p < lin[k].n_paths; ++p)
            if (lin[k].path[p].r % 8 != 0) return false;
    if (sh.head_dim % 32 != 0 || sh.dkv % 8 != 0 || num_sms > 255) return false;
    const SmemPlan S = smem_plan(lin, sh, num_sms);
    int max_optin = 0, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess)
        return false;
    return S.bytes + 1024 <= max_optin;
}

cudaError_t launch_stack(const lb_linear *lin, int n_layers, const StackShape &sh,
                         unsigned long long plan, const uint16_t *x0, float *out, float *q_out,
                         float *kv_out, unsigned *ws_words, char *ws_after_header, int num_sms,
                         cudaStream_t s) {
    const XLayout X = xlayout(lin);
    const SmemPlan S = smem_plan(lin, sh, num_sms);
    Params P{};
    P.lin = reinterpret_cast<const LinDesc *>(ws_after_header);
    P.n_layers = n_layers;
    P.d = sh.d;
    P.dkv = sh.dkv;
    P.dff = sh.dff;
    P.hd = sh.head_dim;
    for (int k = 0; k < 7; ++k) {
        P.np[k] = lin[k].n_paths;
        for (int p = 0; p < 2; ++p) P.r[k][p] = p < lin[k].n_paths ? lin[k].path[p].r : 0;
    }
    P.x0 = x0;
    P.out = out;
    P.q_out = q_out;
    P.kv_out = kv_out;
    P.ws_words = ws_words;
    P.plan = plan;
    P.xacc = reinterpret_cast<unsigned long long *>(ws_after_header + desc_bytes_for(n_layers));
    P.acc_layer = X.acc_layer;
    P.offA = X.offA;
    P.offB = X.offB;
    P.offC = X.offC;
    P.offD = X.offD;
    P.lenA = X.lenA;
    P.lenB = X.lenB;
    P.lenC = X.lenC;
    P.lenD = X.lenD;
    P.fix_limit = 2147483648.f / (float)num_sms;
    P.o = S.o;
    const size_t smem = (size_t)S.bytes;
    cudaError_t e = cudaFuncSetAttribute((const void *)k_stack,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, (const void *)k_stack, kST, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorCooperativeLaunchTooLarge;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)k_stack, dim3(num_sms), dim3(kST), args, smem,
                                       s);
}

}  // namespace lb
