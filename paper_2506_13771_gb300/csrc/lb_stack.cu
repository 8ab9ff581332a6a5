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
constexpr int kSW = kST / 32;   // warps per CTA
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
    int tables, tz, res, xs, ys, yq;  // work areas
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

// Fill n_tab nibble tables at byte offset tb: table n holds, for e = 0..15,
// sum_{k<4} (bit k of e ? -v : +v)[4n + k] with v_i = src[i] * scale[i] * mul
// (scale: fp16, may be null), twice (entries e and 16 + e).  Tables past the
// n_vals values are zero, so sign bits beyond them contribute nothing.
__device__ void build_tables(int tb, int n_tab, const float *src, const uint16_t *scale, float mul,
                             int n_vals) {
    float *T = sm_f(tb);
    for (int idx = threadIdx.x; idx < n_tab * 16; idx += blockDim.x) {
        const int n = idx >> 4, e = idx & 15;
        float v = 0.f;
        if (4 * n < n_vals) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int i = 4 * n + k;
                float x = src[i] * mul;
                if (scale) x *= half_bits_to_float(scale[i]);
                v += ((e >> k) & 1) ? -x : x;
            }
        }
        T[n * 32 + e] = v;
        T[n * 32 + 16 + e] = v;
    }
}

// One stage-2 job: rows [0, nrows) of one path, U words and h in shared memory.
struct UJob {
    int U, h;     // byte offsets: U words [nrows][R], h fp16 [nrows]
    int R, nrows;
    int tb;       // byte offset of the z tables (R * 1024 bytes)
    float *ys;    // output rows (accumulated with atomicAdd)
};

// ys[row] += h[row] * sum_j U_sign[row][j] z[j]; a warp takes 32 rows x one
// word at a time, so all its lanes read the same 8 tables.
__device__ void u_stage(const UJob *jobs, int njobs) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    int total = 0;
    for (int j = 0; j < njobs; ++j) total += ((jobs[j].nrows + 31) >> 5) * jobs[j].R;
    for (int task = warp; task < total; task += kSW) {
        int jb = 0, t = task;
        while (t >= ((jobs[jb].nrows + 31) >> 5) * jobs[jb].R) {
            t -= ((jobs[jb].nrows + 31) >> 5) * jobs[jb].R;
            ++jb;
        }
        const UJob &J = jobs[jb];
        const int rb = t / J.R, w = t - rb * J.R;
        const int row = 32 * rb + lane;
        if (row < J.nrows) {
            const uint32_t word = sm_u32(J.U)[row * J.R + w];
            uint32_t lo, hi;
            split_word(word, copy, lo, hi);
            const float acc = lut8(lo, hi, (uint32_t)(J.tb + w * 1024));
            atomicAdd(J.ys + row, acc * half_bits_to_float(sm_u16(J.h)[row]));
        }
    }
}

// One stage-1 job: all r columns of one path over the CTA's nw input words.
struct VJob {
    int V;        // byte offset of V words [nw][r]
    int r, nw;
    int tb;       // byte offset of the input tables (nw * 1024 bytes)
    unsigned long long *dst;  // exchange words of this path's t
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
// per CTA per element, also when the slice is empty).
__device__ void v_stage(const VJob *jobs, int njobs, float limit, unsigned *err) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    int total = 0;
    for (int j = 0; j < njobs; ++j) total += (jobs[j].r + 31) >> 5;
    for (int task = warp; task < total; task += kSW) {
        int jb = 0, t = task;
        while (t >= ((jobs[jb].r + 31) >> 5)) {
            t -= (jobs[jb].r + 31) >> 5;
            ++jb;
        }
        const VJob &J = jobs[jb];
        const int col = 32 * t + lane;
        if (col < J.r) {
            float acc = 0.f;
            const uint32_t *V = sm_u32(J.V);
            for (int w = 0; w < J.nw; ++w) {
                uint32_t lo, hi;
                split_word(V[w * J.r + col], copy, lo, hi);
                acc += lut8(lo, hi, (uint32_t)(J.tb + w * 1024));
            }
            red_fix(J.dst + col, acc, limit, err);
        }
    }
}

__device__ __forceinline__ float block_sum_sq(const float *v, int n) {
    float s = 0.f;
    for (int i = threadIdx.x; i < n; i += blockDim.x) s += v[i] * v[i];
    return block_sum(s);
}

__device__ __forceinline__ void zero_f(float *p, int n) {
    for (int i = threadIdx.x; i < n; i += blockDim.x) p[i] = 0.f;
}

// Zero this CTA's stripe of an exchange region whose readers are all done.
__device__ __forceinline__ void zero_stripe(unsigned long long *region, int len) {
    const int a = (int)((long long)blockIdx.x * len / gridDim.x);
    const int b = (int)((long long)(blockIdx.x + 1) * len / gridDim.x);
    for (int i = a + threadIdx.x; i < b; i += blockDim.x) region[i] = 0ull;
}

__device__ __forceinline__ bool sticky(const unsigned *ws_words) {
    return ld_relaxed_gpu(ws_words + kErrWord) != 0u;
}

// Wait until each of region[0..n) counts n_ctas contributions and decode the
// sums into out[0..n).  Bounded; returns false (to every thread) on failure.
__device__ bool poll_decode(const unsigned long long *region, int n, unsigned n_ctas, float *out,
                            unsigned *ws_words) {
    int ok = 1;
    for (int i = 2 * threadIdx.x; i < n && ok; i += 2 * blockDim.x) {
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
                    atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                    ok = 0;
                    break;
                }
            }
        }
    }
    return __syncthreads_and(ok) != 0;
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }

// ---------------------------------------------------------------- the kernel

struct Part {
    int dw0, nd, fw0, nf, k0, nkv;
};

struct Loader {
    const Params *P;
    Part s;
    unsigned long long *bar;  // 4 mbarriers: phases A, B, C, D

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
        unsigned long long *b = bar + 0;
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
        unsigned long long *b = bar + 1;
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
        unsigned long long *b = bar + 2;
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
        unsigned long long *b = bar + 3;
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
};

// Bounded wait for a phase buffer.  On failure records LB_ERR_TIMEOUT.
__device__ bool wait_buffer(unsigned long long *bar, unsigned parity, unsigned *ws_words) {
    __shared__ int s_ok;
    if (threadIdx.x == 0) {
        int ok = 1;
        if (!mbar_try_wait(bar, parity)) {
            const unsigned long long t0 = globaltimer_ns();
            while (!mbar_try_wait(bar, parity)) {
                if (globaltimer_ns() - t0 > kWaitLimitNs) {
                    atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                    ok = 0;
                    break;
                }
            }
        }
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

// Error exit: wait (bounded) for the bulk copies still in flight into this
// CTA's buffers, so none lands after the CTA is gone.
__device__ void drain(unsigned long long *bar, const int *pending_parity) {
    if (threadIdx.x != 0) return;
    for (int b = 0; b < 4; ++b) {
        if (pending_parity[b] < 0) continue;
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(bar + b, (unsigned)pending_parity[b]))
            if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
}

__global__ void __launch_bounds__(kST, 1) k_stack(const __grid_constant__ Params P) {
    __shared__ __align__(8) unsigned long long bars[4];
    __shared__ int s_last;
    unsigned *err = P.ws_words + kErrWord;
    if (sticky(P.ws_words)) return;
    if (*reinterpret_cast<const volatile unsigned long long *>(P.ws_words + kPlanWord) != P.plan) {
        if (blockIdx.x == 0 && threadIdx.x == 0)
            atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_PLAN));
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
    const int rows_d = 32 * s.nd, rows_f = 32 * s.nf;
    const Offsets &o = P.o;
    Loader ld{&P, s, bars};
    // parity of the load outstanding in each buffer (-1: none)
    int pending[4] = {-1, -1, -1, -1};

    if (threadIdx.x == 0) {
        for (int b = 0; b < 4; ++b) mbar_init(bars + b, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        ld.issue_A(0);
        ld.issue_B(0);
        ld.issue_C(0);
        ld.issue_D(0);
    }
    for (int b = 0; b < 4; ++b) pending[b] = 0;

    float *res = sm_f(o.res), *xs = sm_f(o.xs), *ys = sm_f(o.ys), *yq = sm_f(o.yq);
    float *tz = sm_f(o.tz);
    for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
        res[i] = bf16_bits_to_float(P.x0[32 * s.dw0 + i]);

    UJob uj[6];
    VJob vj[6];
    const int rq[2] = {P.r[LQ][0], P.r[LQ][1]};
#define FAIL_EXIT()            \
    do {                       \
        drain(bars, pending);  \
        return;                \
    } while (0)

    for (int l = 0; l < P.n_layers; ++l) {
        const LinDesc *Ly = P.lin + 7 * l;
        unsigned long long *xA = P.xacc + (size_t)l * P.acc_layer + P.offA;
        unsigned long long *xB = P.xacc + (size_t)l * P.acc_layer + P.offB;
        unsigned long long *xC = P.xacc + (size_t)l * P.acc_layer + P.offC;
        unsigned long long *xD = P.xacc + (size_t)l * P.acc_layer + P.offD;
        int nrq = 0, nrk = 0, nrv = 0;
        for (int p = 0; p < P.np[LQ]; ++p) nrq += P.r[LQ][p];
        for (int p = 0; p < P.np[LK]; ++p) nrk += P.r[LK][p];
        for (int p = 0; p < P.np[LV]; ++p) nrv += P.r[LV][p];
        int nro = 0, nrg = 0, nru = 0, nrd = 0;
        for (int p = 0; p < P.np[LO]; ++p) nro += P.r[LO][p];
        for (int p = 0; p < P.np[LG]; ++p) nrg += P.r[LG][p];
        for (int p = 0; p < P.np[LU]; ++p) nru += P.r[LU][p];
        for (int p = 0; p < P.np[LD]; ++p) nrd += P.r[LD][p];
        const int ssA = nrq + nrk + nrv, ssC = nrg + nru;

        // ================= phase A: a = h + Down_{l-1}(m) on R_c; stage 1 of q, k, v
        if (l > 0) {
            unsigned long long *xDp = P.xacc + (size_t)(l - 1) * P.acc_layer + P.offD;
            if (!poll_decode(xDp, nrd, n_ctas, tz, P.ws_words)) FAIL_EXIT();
            zero_stripe(P.xacc + (size_t)(l - 1) * P.acc_layer + P.offC, P.lenC);
        }
        if (!wait_buffer(bars + 0, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        pending[0] = -1;
        if (l > 0) {
            const LinDesc &Dn = P.lin[7 * (l - 1) + LD];
            int tb = o.tables, off = 0, nj = 0;
            for (int p = 0; p < Dn.n_paths; ++p) {
                const int R = wordsR(Dn.r[p]);
                build_tables(tb, 8 * R, tz + off, sm_u16(o.a_ld[p]), 1.f, Dn.r[p]);
                uj[nj++] = UJob{o.a_Ud[p], o.a_hd[p], R, rows_d, tb, ys};
                tb += R * 1024;
                off += Dn.r[p];
            }
            zero_f(ys, rows_d);
            __syncthreads();
            u_stage(uj, nj);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_d; i += blockDim.x) res[i] += ys[i];
        }
        __syncthreads();
        {
            const float ss = block_sum_sq(res, rows_d);
            if (threadIdx.x == 0) red_fix(xA + ssA, ss, P.fix_limit, err);
            int tb = o.tables, nj = 0;
            unsigned long long *dst = xA;
            for (int k = 0; k < 3; ++k) {
                const LinDesc &L = Ly[k];
                for (int p = 0; p < L.n_paths; ++p) {
                    build_tables(tb, 8 * s.nd, res, sm_u16(o.a_g[k][p]), 1.f, rows_d);
                    vj[nj++] = VJob{o.a_V[k][p], L.r[p], s.nd, tb, dst};
                    tb += s.nd * 1024;
                    dst += L.r[p];
                }
            }
            __syncthreads();
            v_stage(vj, nj, P.fix_limit, err);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            fence_proxy_async();
            ld.issue_A(l + 1);
        }
        pending[0] = (l + 1) & 1;

        // ================= phase B: v rows for attention, stage 1 of o; then q, k, v out
        if (!poll_decode(xA, ssA + 1, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        if (l > 0) zero_stripe(P.xacc + (size_t)(l - 1) * P.acc_layer + P.offD, P.lenD);
        if (!wait_buffer(bars + 1, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        pending[1] = -1;
        {
            const float inv = rsqrtf(tz[ssA] / (float)P.d);
            const LinDesc &V = Ly[LV], &O = Ly[LO];
            float *attn = xs;
            int tb = o.tables, nj = 0;
            for (int p = 0, off = nrq + nrk; p < V.n_paths; off += V.r[p], ++p) {
                const int R = wordsR(V.r[p]);
                build_tables(tb, 8 * R, tz + off, sm_u16(o.b_lv[p]), inv, V.r[p]);
                uj[nj++] = UJob{o.b_Uat[p], o.b_hat[p], R, rows_d, tb, attn};
                tb += R * 1024;
            }
            const int tb_after_v = tb;
            zero_f(attn, rows_d);
            __syncthreads();
            u_stage(uj, nj);
            __syncthreads();
            nj = 0;
            unsigned long long *dst = xB;
            for (int p = 0; p < O.n_paths; ++p) {
                build_tables(tb, 8 * s.nd, attn, sm_u16(o.b_go[p]), 1.f, rows_d);
                vj[nj++] = VJob{o.b_Vo[p], O.r[p], s.nd, tb, dst};
                tb += s.nd * 1024;
                dst += O.r[p];
            }
            __syncthreads();
            v_stage(vj, nj, P.fix_limit, err);
            // ---- off the critical path: q on R_c, k and v on K_c
            const LinDesc &Q = Ly[LQ], &K = Ly[LK];
            float *yk = ys, *yv = ys + s.nkv;
            nj = 0;
            int tb2 = tb;
            for (int p = 0, off = 0; p < Q.n_paths; off += Q.r[p], ++p) {
                const int R = wordsR(Q.r[p]);
                build_tables(tb2, 8 * R, tz + off, sm_u16(o.b_lq[p]), inv, Q.r[p]);
                uj[nj++] = UJob{o.b_Uq[p], o.b_hq[p], R, rows_d, tb2, yq};
                tb2 += R * 1024;
            }
            for (int p = 0, off = nrq; p < K.n_paths; off += K.r[p], ++p) {
                const int R = wordsR(K.r[p]);
                build_tables(tb2, 8 * R, tz + off, sm_u16(o.b_lk[p]), inv, K.r[p]);
                uj[nj++] = UJob{o.b_Uk[p], o.b_hk[p], R, s.nkv, tb2, yk};
                tb2 += R * 1024;
            }
            // v on K_c reuses v's tables built above
            for (int p = 0, tbv = o.tables; p < V.n_paths; ++p) {
                const int R = wordsR(V.r[p]);
                uj[nj++] = UJob{o.b_Uvk[p], o.b_hvk[p], R, s.nkv, tbv, yv};
                tbv += R * 1024;
            }
            (void)tb_after_v;
            zero_f(yq, rows_d);
            zero_f(ys, 2 * s.nkv);
            __syncthreads();
            u_stage(uj, nj);
            __syncthreads();
            if (P.q_out)
                for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
                    P.q_out[(size_t)l * P.d + 32 * s.dw0 + i] = yq[i];
            if (P.kv_out)
                for (int i = threadIdx.x; i < s.nkv; i += blockDim.x) {
                    P.kv_out[((size_t)l * 2 + 0) * P.dkv + s.k0 + i] = yk[i];
                    P.kv_out[((size_t)l * 2 + 1) * P.dkv + s.k0 + i] = yv[i];
                }
        }
        __syncthreads();
        if (threadIdx.x == 0 && l + 1 < P.n_layers) {
            fence_proxy_async();
            ld.issue_B(l + 1);
        }
        pending[1] = l + 1 < P.n_layers ? ((l + 1) & 1) : -1;

        // ================= phase C: h = a + O(attn) on R_c; stage 1 of gate, up
        if (!poll_decode(xB, nro, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(xA, P.lenA);
        if (!wait_buffer(bars + 2, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        pending[2] = -1;
        {
            const LinDesc &O = Ly[LO], &G = Ly[LG], &U = Ly[LU];
            int tb = o.tables, nj = 0;
            for (int p = 0, off = 0; p < O.n_paths; off += O.r[p], ++p) {
                const int R = wordsR(O.r[p]);
                build_tables(tb, 8 * R, tz + off, sm_u16(o.c_lo[p]), 1.f, O.r[p]);
                uj[nj++] = UJob{o.c_Uo[p], o.c_ho[p], R, rows_d, tb, ys};
                tb += R * 1024;
            }
            zero_f(ys, rows_d);
            __syncthreads();
            u_stage(uj, nj);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_d; i += blockDim.x) res[i] += ys[i];
            __syncthreads();
            const float ss = block_sum_sq(res, rows_d);
            if (threadIdx.x == 0) red_fix(xC + ssC, ss, P.fix_limit, err);
            tb = o.tables;
            nj = 0;
            unsigned long long *dst = xC;
            for (int p = 0; p < G.n_paths; ++p) {
                build_tables(tb, 8 * s.nd, res, sm_u16(o.c_gg[p]), 1.f, rows_d);
                vj[nj++] = VJob{o.c_Vg[p], G.r[p], s.nd, tb, dst};
                tb += s.nd * 1024;
                dst += G.r[p];
            }
            for (int p = 0; p < U.n_paths; ++p) {
                build_tables(tb, 8 * s.nd, res, sm_u16(o.c_gu[p]), 1.f, rows_d);
                vj[nj++] = VJob{o.c_Vu[p], U.r[p], s.nd, tb, dst};
                tb += s.nd * 1024;
                dst += U.r[p];
            }
            __syncthreads();
            v_stage(vj, nj, P.fix_limit, err);
        }
        __syncthreads();
        if (threadIdx.x == 0 && l + 1 < P.n_layers) {
            fence_proxy_async();
            ld.issue_C(l + 1);
        }
        pending[2] = l + 1 < P.n_layers ? ((l + 1) & 1) : -1;

        // ================= phase D: m = silu(gate) * up on F_c; stage 1 of down
        if (!poll_decode(xC, ssC + 1, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(xB, P.lenB);
        if (!wait_buffer(bars + 3, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        pending[3] = -1;
        {
            const float inv = rsqrtf(tz[ssC] / (float)P.d);
            const LinDesc &G = Ly[LG], &U = Ly[LU], &D = Ly[LD];
            float *yg = ys, *yu = ys + rows_f;
            int tb = o.tables, nj = 0;
            for (int p = 0, off = 0; p < G.n_paths; off += G.r[p], ++p) {
                const int R = wordsR(G.r[p]);
                build_tables(tb, 8 * R, tz + off, sm_u16(o.d_lg[p]), inv, G.r[p]);
                uj[nj++] = UJob{o.d_Ug[p], o.d_hg[p], R, rows_f, tb, yg};
                tb += R * 1024;
            }
            for (int p = 0, off = nrg; p < U.n_paths; off += U.r[p], ++p) {
                const int R = wordsR(U.r[p]);
                build_tables(tb, 8 * R, tz + off, sm_u16(o.d_lu[p]), inv, U.r[p]);
                uj[nj++] = UJob{o.d_Uu[p], o.d_hu[p], R, rows_f, tb, yu};
                tb += R * 1024;
            }
            zero_f(ys, 2 * rows_f);
            __syncthreads();
            u_stage(uj, nj);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_f; i += blockDim.x) xs[i] = silu(yg[i]) * yu[i];
            __syncthreads();
            tb = o.tables;
            nj = 0;
            unsigned long long *dst = xD;
            for (int p = 0; p < D.n_paths; ++p) {
                build_tables(tb, 8 * s.nf, xs, sm_u16(o.d_gd[p]), 1.f, rows_f);
                vj[nj++] = VJob{o.d_Vd[p], D.r[p], s.nf, tb, dst};
                tb += s.nf * 1024;
                dst += D.r[p];
            }
            __syncthreads();
            v_stage(vj, nj, P.fix_limit, err);
        }
        __syncthreads();
        if (threadIdx.x == 0 && l + 1 < P.n_layers) {
            fence_proxy_async();
            ld.issue_D(l + 1);
        }
        pending[3] = l + 1 < P.n_layers ? ((l + 1) & 1) : -1;
        (void)rq;
    }

    // ================= final: out = h + Down_{L-1}(m) on R_c
    {
        const int l = P.n_layers;
        unsigned long long *xDl = P.xacc + (size_t)(l - 1) * P.acc_layer + P.offD;
        const LinDesc &Dn = P.lin[7 * (l - 1) + LD];
        int nrd = 0;
        for (int p = 0; p < Dn.n_paths; ++p) nrd += Dn.r[p];
        if (!poll_decode(xDl, nrd, n_ctas, tz, P.ws_words)) FAIL_EXIT();
        zero_stripe(P.xacc + (size_t)(l - 1) * P.acc_layer + P.offC, P.lenC);
        if (!wait_buffer(bars + 0, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        pending[0] = -1;
        int tb = o.tables, off = 0, nj = 0;
        for (int p = 0; p < Dn.n_paths; ++p) {
            const int R = wordsR(Dn.r[p]);
            build_tables(tb, 8 * R, tz + off, sm_u16(o.a_ld[p]), 1.f, Dn.r[p]);
            uj[nj++] = UJob{o.a_Ud[p], o.a_hd[p], R, rows_d, tb, ys};
            tb += R * 1024;
            off += Dn.r[p];
        }
        zero_f(ys, rows_d);
        __syncthreads();
        u_stage(uj, nj);
        __syncthreads();
        for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
            P.out[32 * s.dw0 + i] = res[i] + ys[i];
        // The last CTA to finish has seen every other CTA's reads of the final
        // region: it clears that region and the counters for the next launch.
        if (threadIdx.x == 0) {
            __threadfence();
            s_last = atomicAdd(P.ws_words + kDoneWord, 1u) == n_ctas - 1;
        }
        __syncthreads();
        if (s_last) {
            __threadfence();
            for (int i = threadIdx.x; i < P.lenD; i += blockDim.x) xDl[i] = 0ull;
            if (threadIdx.x == 0) P.ws_words[kDoneWord] = 0u;
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
