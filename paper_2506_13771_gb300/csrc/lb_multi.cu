// lb_multi.cu -- one token (T = 1) through M LittleBit linears of one shape
// that read the same input x, in ONE persistent launch: the q / k / v (or
// gate / up) projections of a decoder layer, or M independent weight sets.
//
// Per linear and path, Prop. 1 (LittleBit, arXiv 2506.13771): stage 1
// t = V_sign^T (g . x), a +-1 reduction over d_in split across the CTAs and
// summed through self-counting exchange words; stage 2 y = h . (U_sign (l . t))
// over each CTA's output rows; Eq. 6 sums the paths.  The single-linear
// kernel (k_decode) runs the two stages back to back and waits for its
// exchange in between.  Here the compute warps form two groups that run the
// two stages of different linears at once: the stage-1 group sends linear
// m's partial t while the stage-2 group builds the outputs of an earlier
// linear, so each exchange completes behind other linears' work and neither
// stage waits for the other's barriers (for a few linears, a phased schedule
// instead runs every compute warp over stage 1 of all of them, then stage 2,
// when its cost model says that is cheaper).  A producer warp bulk-copies
// (cp.async.bulk) each linear's V slice, g slice, U rows and h into a ring of
// kSlots shared-memory slots, a slot being refilled once its linear's stage 2
// is done (so stage 1 runs at most kSlots linears ahead of stage 2).  The exchange words of all M linears are
// double-buffered by the workspace's launch epoch as in k_decode: every CTA
// clears its stripe of the previous launch's buffer.  In the residual-input
// mode (a decoder's a += y ahead of its q / k / v or gate / up) each CTA adds
// its input slice into a, sends its share of mean(a^2) in one more exchange
// word, and the outputs are scaled by 1 / rms(a) (the linears are homogeneous:
// L(a / rms a) = L(a) / rms a), so no separate norm launch is needed.  Every
// wait is bounded;
// on a timeout the CTA records LB_ERR_TIMEOUT, lets its own copies land and
// returns.
#include <algorithm>
#include <mutex>

#include "lb_common.cuh"
#include "lb_kernels.h"
#include "lb_lut.cuh"

namespace lb {

namespace {

constexpr int kMT = 512;  // threads per CTA
constexpr int kMW = kMT / 32;
constexpr int kSlots = 7;
constexpr int kCW = kMW - 1;       // compute warps; the last warp issues the copies
constexpr int kCT = kCW * 32;

struct MultiPtrs {
    const uint32_t *v[2], *u[2];
    const uint16_t *g[2], *l[2], *h[2];
};

// Shared-memory byte offsets; V / g / U / h / l are offsets inside a slot.
struct MultiLayout {
    int V[2], g[2], U[2], h[2], l[2], slot_bytes, slots, xs, t1, t2, y, bytes;
};

struct MultiParams {
    int d_in, d_out, np, r[2], M, N1, off1;
    int k1;  // compute warps of the stage-1 group (the rest run stage 2); 0: phased
    const void *x;  // bf16 [d_in] (x_fp32 = 0), or fp32 (x_fp32 = 1)
    int x_fp32;     // 3: residual input, see res_a
    // x_fp32 = 3: x = res_a + res_y (fp32 [d_in]), written back to res_a, and
    // every output scaled by 1 / rms(x) (a decoder's residual add and RMS
    // norm ahead of its linears: L(x / rms x) = L(x) / rms x)
    float *res_a;
    const float *res_y;
    void *y;        // [M][d_out], bf16 or fp32
    int y_fp32;
    unsigned *ws_words;
    unsigned long long *xw;  // exchange pairs: two buffers of M * N1 + 1
    float fix_limit;
    MultiLayout o;
    MultiPtrs p[kMaxMultiLinears];
};

__device__ bool wait_bar_m(unsigned long long *bar, unsigned parity, unsigned *ws_words) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (ld_relaxed_gpu(ws_words + kErrWord) != 0u) return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
            return false;
        }
    }
    return true;
}

__device__ __forceinline__ void csync_m() {
    asm volatile("bar.sync 1, %0;" ::"n"(kCT) : "memory");
}
// Barrier over a warp group (named barrier id of n threads, n a multiple of 32).
__device__ __forceinline__ void gsync(int id, int n) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// AND of pred over a warp group, returned to each of its threads.
__device__ __forceinline__ int gsync_and(int id, int n, int pred) {
    int r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.s32 p, %1, 0;\n\tbar.red.and.pred q, %2, %3, p;\n\t"
        "selp.s32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(pred), "r"(id), "r"(n)
        : "memory");
    return r;
}

__global__ void __launch_bounds__(kMT, 1) k_decode_multi(const __grid_constant__ MultiParams P) {
    __shared__ __align__(8) unsigned long long vbar[kSlots], ubar[kSlots], fbar[kSlots];
    __shared__ int s_ok, s_issued;
    __shared__ float s_ss, s_inv;  // residual input: sum of squares of the slice, 1 / rms
    unsigned *err = P.ws_words + kErrWord;
    if (ld_relaxed_gpu(err) != 0u) return;
    const unsigned epoch = ld_relaxed_gpu(P.ws_words + kEpochWord);
    // a buffer holds M * N1 exchange elements of t, then the sum-of-squares
    // element (element `words`)
    const size_t words = (size_t)P.M * P.N1, stride = fix2_words(words + 1);
    unsigned long long *xw = P.xw + (size_t)(epoch & 1u) * stride;
    unsigned long long *xold = P.xw + (size_t)((epoch + 1u) & 1u) * stride;
    const bool res = P.x_fp32 == 3;
    const MultiLayout &o = P.o;
    const int N = gridDim.x, c = blockIdx.x, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31, np = P.np;
    // input words [iw0, iw0 + nw), output rows [o0, o0 + nrows) (whole octets)
    const int W = P.d_in >> 5, Q = P.d_out >> 3;
    int iw0, nw;
    s1_slice(W, N, c, iw0, nw);
    const int q0 = (int)((long long)c * Q / N), nq = (int)((long long)(c + 1) * Q / N) - q0;
    const int o0 = 8 * q0, nrows = 8 * nq;
    // Contributions per exchange word: the stage-1 CTAs; element 0 of linear
    // 0 also counts every other CTA once (so that no CTA can still be about
    // to read the epoch when block 0 moves it on), as does the sum-of-squares
    // element.
    const unsigned n_contrib = (unsigned)s1_ctas(W, N), n_first = (unsigned)N;
    const int R0 = (P.r[0] + 31) >> 5, R1 = np > 1 ? (P.r[1] + 31) >> 5 : 0;
    const int cbs = R0 + R1, nt0 = 8 * R0, ntab = 8 * (R0 + R1);

    if (tid == 0) {
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(vbar + s, 1);
            mbar_init(ubar + s, 1);
            mbar_init(fbar + s, 1);
        }
        fence_barrier_init();
        s_ok = 1;
        s_issued = 0;
        s_ss = 0.f;
        s_inv = 1.f;
    }
    __syncthreads();
    auto slot = [&](int m) { return g_smem + o.slots + (m % kSlots) * o.slot_bytes; };

    if (warp == kCW) {
        // ---------------- producer: the copies of every linear into its slot,
        //                  a slot refilled once the compute warps freed it
        if (lane == 0) {
            for (int m = 0; m < P.M; ++m) {
                if (m >= kSlots &&
                    !wait_bar_m(fbar + m % kSlots, (unsigned)(((m - kSlots) / kSlots) & 1),
                                P.ws_words))
                    break;
                unsigned char *b = slot(m);
                unsigned long long *vb = vbar + m % kSlots, *ub = ubar + m % kSlots;
                const MultiPtrs &L = P.p[m];
                for (int p = 0; p < np; ++p) {
                    const int r = P.r[p], R = (r + 31) >> 5;
                    if (nw > 0) {
                        mbar_expect_tx(vb, (unsigned)(nw * r * 4 + 64 * nw));
                        bulk_g2s(b + o.V[p], L.v[p] + (size_t)iw0 * r, (unsigned)(nw * r * 4), vb);
                        bulk_g2s(b + o.g[p], L.g[p] + 32 * iw0, (unsigned)(64 * nw), vb);
                    }
                    // l with the U rows: stage 2's tables read it next to the exchange
                    mbar_expect_tx(ub, (unsigned)(2 * r + (nrows > 0 ? nrows * R * 4 + 2 * nrows : 0)));
                    bulk_g2s(b + o.l[p], L.l[p], (unsigned)(2 * r), ub);
                    if (nrows > 0) {
                        bulk_g2s(b + o.U[p], L.u[p] + (size_t)o0 * R, (unsigned)(nrows * R * 4), ub);
                        bulk_g2s(b + o.h[p], L.h[p] + o0, (unsigned)(2 * nrows), ub);
                    }
                }
                mbar_arrive(vb);
                mbar_arrive(ub);
                s_issued = m + 1;
            }
        }
        __syncwarp();
    } else {
        // ---------------- compute warps (named barrier 1; then two groups)
        // the x slice (fp32), and the previous launch's exchange words back to zero
        float *xs = reinterpret_cast<float *>(g_smem + o.xs);
        float ss = 0.f;
        for (int i = tid; i < 32 * nw; i += kCT) {
            const int e = 32 * iw0 + i;
            float v;
            if (res) {
                v = P.res_a[e] + P.res_y[e];
                P.res_a[e] = v;  // this CTA's inputs only
                ss += v * v;
            } else {
                v = P.x_fp32 ? static_cast<const float *>(P.x)[e]
                             : bf16_bits_to_float(static_cast<const uint16_t *>(P.x)[e]);
            }
            xs[i] = v;
        }
        if (res) {
#pragma unroll
            for (int of = 16; of > 0; of >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, of);
            if (lane == 0) atomicAdd(&s_ss, ss);
        }
        {
            const size_t a = (size_t)c * stride / N, e = (size_t)(c + 1) * stride / N;
            for (size_t i = a + tid; i < e; i += kCT) xold[i] = 0ull;
        }
        csync_m();
        // every CTA's share of the mean square (sum / d_in: the fixed-point
        // word then holds outlier-sized activations too), counted like linear
        // 0's words
        if (res && tid == 0)
            send_fix2(fix2_at(xw, (int)words), s_ss / (float)P.d_in, P.fix_limit, err);
        const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
        bool ok = true;
        // Two warp groups run the two stages of different linears at once:
        // warps [0, k1) stage 1 of linear m, warps [k1, kCW) stage 2 of linear
        // m - (how far stage 1 has got); each group synchronises on a named
        // barrier of its own.  Stage 1 can run ahead of stage 2 as far as the
        // slot ring allows (the producer refills a slot once stage 2 freed it).
        // Phased (k1 = 0, for few linears): every compute warp runs stage 1 of
        // all the linears, then stage 2 of all of them.
        const bool phased = P.k1 == 0;
        const int k1 = phased ? kCW : P.k1, n1t = 32 * k1;
        const int g2 = phased ? 0 : k1, n2t = kCT - 32 * g2;
        if (warp < k1) {
            // ---------------- stage 1 group (named barrier 2)
            if (nw == 0) {
                // a CTA without input words still counts itself into linear 0's
                // element 0
                if (tid == 0) send_count2(fix2_at(xw, 0));
            } else {
                for (int m = 0; m < P.M && ok; ++m) {
                    unsigned char *b = slot(m);
                    // tables of g . x (8 per input word and path), once the slice landed
                    bool got = true;
                    if (tid == 0)
                        got = wait_bar_m(vbar + m % kSlots, (unsigned)((m / kSlots) & 1),
                                         P.ws_words);
                    if (!gsync_and(2, n1t, got)) {
                        ok = false;
                        break;
                    }
                    if (tid != 0) mbar_try_wait(vbar + m % kSlots, (unsigned)((m / kSlots) & 1));
                    for (int idx = tid; idx < np * 8 * nw; idx += n1t) {
                        const int p = idx / (8 * nw), n = idx - p * 8 * nw;
                        const float4 xv = *reinterpret_cast<const float4 *>(xs + 4 * n);
                        const uint2 gw = *reinterpret_cast<const uint2 *>(b + o.g[p] + 8 * n);
                        const float4 v =
                            make_float4(xv.x * half_bits_to_float((uint16_t)(gw.x & 0xffffu)),
                                        xv.y * half_bits_to_float((uint16_t)(gw.x >> 16)),
                                        xv.z * half_bits_to_float((uint16_t)(gw.y & 0xffffu)),
                                        xv.w * half_bits_to_float((uint16_t)(gw.y >> 16)));
                        store_table(g_smem + o.t1 + idx * 128, v, lane);
                    }
                    gsync(2, n1t);
                    const int xm = m * P.N1;  // the linear's first element
                    for (int u = warp; u < cbs; u += k1) {
                        const int p = u >= R0 ? 1 : 0, cb = u - (p ? R0 : 0);
                        const int r = P.r[p];
                        const int col = 32 * cb + lane, cc = min(col, r - 1);
                        const uint32_t *Vw = reinterpret_cast<const uint32_t *>(b + o.V[p]) + cc;
                        const uint32_t tb = (uint32_t)(o.t1 + p * 8 * nw * 128);
                        float acc0 = 0.f, acc1 = 0.f;
                        int w = 0;
                        for (; w + 2 <= nw; w += 2) {
                            const uint32_t w0 = Vw[w * r], w1 = Vw[(w + 1) * r];
                            acc0 += lut_word(w0, copy, tb + w * 1024);
                            acc1 += lut_word(w1, copy, tb + (w + 1) * 1024);
                        }
                        if (w < nw) acc0 += lut_word(Vw[w * r], copy, tb + w * 1024);
                        if (col < r)
                            send_fix2(fix2_at(xw, xm + (p ? P.off1 : 0) + col), acc0 + acc1,
                                      P.fix_limit, err);
                    }
                    gsync(2, n1t);  // t1 is rebuilt by the next linear
                }
            }
        }
        if (phased) csync_m();
        if (warp >= g2 && ok) {
            // ---------------- stage 2 group (named barrier 3)
            const int t2 = tid - 32 * g2, w2 = warp - g2, nw2 = kCW - g2;
            const bool lead2 = t2 == 0;
            const int S0 = s2_parts(R0), S1 = np > 1 ? s2_parts(R1) : 0;
            const int rb = (nrows + 31) >> 5, nu0 = rb * S0, nu = nu0 + rb * S1;
            float *y = reinterpret_cast<float *>(g_smem + o.y);  // part slots
            // the exchange words a thread polls for stage 2 (its table t2 when
            // t2 < ntab), loaded while the row sums of the linear before run,
            // so that the L2 round trip overlaps them
            unsigned long long pre[8] = {0ull, 0ull, 0ull, 0ull, 0ull, 0ull, 0ull, 0ull};
            auto prefetch = [&](int mm) {
                if (mm < 0 || mm >= P.M || t2 >= ntab) return;
                const int p = t2 >= nt0 ? 1 : 0, n = t2 - (p ? nt0 : 0);
                if (4 * n >= P.r[p]) return;
                ld_fix2x4(fix2_at(xw, mm * P.N1 + (p ? P.off1 : 0) + 4 * n), pre);
            };
            prefetch(0);
            for (int mm = 0; mm < P.M && ok; ++mm) {
                const int xm = mm * P.N1;  // the linear's first element
                unsigned char *b = slot(mm);
                // the slot's U rows, h and l (the lead waits, the rest observe the phase)
                bool u_ok = true;
                if (lead2)
                    u_ok = wait_bar_m(ubar + mm % kSlots, (unsigned)((mm / kSlots) & 1),
                                      P.ws_words);
                if (!gsync_and(3, n2t, u_ok)) {
                    ok = false;
                    break;
                }
                if (!lead2) mbar_try_wait(ubar + mm % kSlots, (unsigned)((mm / kSlots) & 1));
                int pok = 1;
                if (res && mm == 0 && lead2) {
                    // the sum of squares of the whole input (all CTAs counted)
                    unsigned long long wh = 0, wl = 0, t0 = 0;
                    for (int spin = 0;; ++spin) {
                        ld_fix2(fix2_at(xw, (int)words), wh, wl);
                        if (counted2(wh, wl, n_first)) break;
                        if ((spin & 15) == 15) {
                            if (ld_relaxed_gpu(err) != 0u) {
                                pok = 0;
                                break;
                            }
                            const unsigned long long now = globaltimer_ns();
                            if (t0 == 0) t0 = now;
                            if (now - t0 > kWaitLimitNs) {
                                atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                                pok = 0;
                                break;
                            }
                        }
                    }
                    if (pok) s_inv = rsqrtf(dec_fix2(wh, wl));
                }
                for (int idx = t2; idx < ntab && pok; idx += n2t) {
                    const int p = idx >= nt0 ? 1 : 0, n = idx - (p ? nt0 : 0);
                    const int r = P.r[p];
                    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (4 * n < r) {
                        const uint2 lw = *reinterpret_cast<const uint2 *>(b + o.l[p] + 8 * n);
                        const unsigned long long *wd = fix2_at(xw, xm + (p ? P.off1 : 0) + 4 * n);
                        unsigned long long a[8], t0 = 0;
                        for (int spin = 0;; ++spin) {
                            if (spin == 0 && idx == t2) {
#pragma unroll
                                for (int k = 0; k < 8; ++k) a[k] = pre[k];
                            } else {
                                ld_fix2x4(wd, a);
                            }
                            const unsigned want0 = mm == 0 && idx == 0 ? n_first : n_contrib;
                            if (counted2x4(a, want0, n_contrib)) break;
                            if ((spin & 15) == 15) {
                                if (ld_relaxed_gpu(err) != 0u) {
                                    pok = 0;
                                    break;
                                }
                                const unsigned long long now = globaltimer_ns();
                                if (t0 == 0) t0 = now;
                                if (now - t0 > kWaitLimitNs) {
                                    atomicCAS(err, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                                    pok = 0;
                                    break;
                                }
                            }
                        }
                        v = make_float4(
                            dec_fix2(a[0], a[1]) * half_bits_to_float((uint16_t)(lw.x & 0xffffu)),
                            dec_fix2(a[2], a[3]) * half_bits_to_float((uint16_t)(lw.x >> 16)),
                            dec_fix2(a[4], a[5]) * half_bits_to_float((uint16_t)(lw.y & 0xffffu)),
                            dec_fix2(a[6], a[7]) * half_bits_to_float((uint16_t)(lw.y >> 16)));
                    }
                    store_table(g_smem + o.t2 + idx * 128, v, lane);
                }
                if (!gsync_and(3, n2t, pok)) {
                    ok = false;
                    break;
                }
                prefetch(mm + 1);
                // every CTA contributed to linear 0's element 0 before it could
                // complete, so all have read the epoch: the next launch may use
                // the other buffer
                if (mm == 0 && c == 0 && lead2) P.ws_words[kEpochWord] = epoch + 1u;
                // parts of 32 rows x up to four words of one path
                for (int u = w2; u < nu; u += nw2) {
                    const int p = u >= nu0 ? 1 : 0, v = u - (p ? nu0 : 0), S = p ? S1 : S0;
                    const int bb = v / S, sp = v - bb * S;
                    s2_part(reinterpret_cast<const uint32_t *>(b + o.U[p]), p ? R1 : R0,
                            reinterpret_cast<const uint16_t *>(b + o.h[p]),
                            (uint32_t)(o.t2 + (p ? nt0 : 0) * 128), nrows, bb, sp,
                            y + (size_t)((p ? S0 : 0) + sp) * nrows, copy, lane);
                }
                gsync(3, n2t);
                // the slot is free for the producer
                if (lead2) mbar_arrive(fbar + mm % kSlots);
                const float sc = s_inv;  // 1 unless the input is a residual add
                for (int i = t2; i < nrows; i += n2t) {
                    const size_t at = (size_t)mm * P.d_out + o0 + i;
                    const float v = s2_combine(y, nrows, S0 + S1, i) * sc;
                    if (P.y_fp32)
                        static_cast<float *>(P.y)[at] = v;
                    else
                        static_cast<uint16_t *>(P.y)[at] = float_to_bf16_bits(v);
                }
                // the next linear's parts overwrite the slots: its first group
                // barrier (after its slot wait) orders them after these reads
            }
        }
        if (!ok) s_ok = 0;
    }
    __syncthreads();
    if (!s_ok && tid == 0) {
        // every copy this CTA issued must land before it goes away (the last
        // use of each slot; earlier uses were consumed)
        const int issued = s_issued;
        for (int m = issued > kSlots ? issued - kSlots : 0; m < issued; ++m) {
            wait_bar_m(vbar + m % kSlots, (unsigned)((m / kSlots) & 1), P.ws_words);
            wait_bar_m(ubar + m % kSlots, (unsigned)((m / kSlots) & 1), P.ws_words);
        }
    }
}

int up16(int n) { return (n + 15) & ~15; }

MultiLayout layout_of(const lb_linear &L, int N) {
    const int W = L.d_in / 32, n_s1 = s1_ctas(W, N);
    const int nw = (W + n_s1 - 1) / n_s1, nrows = 8 * ((L.d_out / 8 + N - 1) / N);
    MultiLayout o{};
    int at = 0;
    auto take = [&at](int bytes) {
        const int off = at;
        at += up16(bytes);
        return off;
    };
    // one slot: V and g slices, U rows and h of each path
    int ntab2 = 0, nslot = 0;
    for (int p = 0; p < 2; ++p) {
        const bool on = p < L.n_paths;
        const int r = on ? L.path[p].r : 0, R = (r + 31) / 32;
        o.V[p] = take(nw * r * 4);
        o.g[p] = take(on ? 64 * nw : 0);
        o.U[p] = take(nrows * R * 4);
        o.h[p] = take(2 * nrows);
        o.l[p] = take(2 * r);
        ntab2 += 8 * R;
        nslot += on ? s2_parts(R) : 0;
    }
    o.slot_bytes = up16(at);
    at = 0;
    o.slots = take(kSlots * o.slot_bytes);
    o.xs = take(128 * nw);
    // table bases are 1024-aligned: lut8 splices the entry byte into them
    at = (at + 1023) & ~1023;
    o.t1 = take(L.n_paths * 8 * nw * 128);
    at = (at + 1023) & ~1023;
    o.t2 = take(ntab2 * 128);
    o.y = take(4 * nrows * nslot);
    o.bytes = at;
    return o;
}

// Warps of the stage-1 group, or 0 for the phased schedule: the choice with
// the shortest estimated launch for M linears.  Per warp, units cost their
// sign words plus a fixed cost measured per unit: a stage-1 unit (32 columns
// x the input slice) its words + 3 (mostly its exchange sends), a stage-2
// part (32 rows x up to four words) its words + 1, a round of polled tables
// 3; an exchange takes about 20 such units to complete.  Split: max(M t1, t1
// + exchange + M t2); phased: M t1 + what is left of the first exchange
// after the other linears' stage 1, + M t2, both stages on all 15 warps
// (phased needs M <= kSlots).
int stage1_warps(const lb_linear &L, int N, int M) {
    const int W = L.d_in / 32, n_s1 = s1_ctas(W, N);
    const int nw = (W + n_s1 - 1) / n_s1, nrows = 8 * ((L.d_out / 8 + N - 1) / N);
    const int rb = (nrows + 31) / 32;
    int cbs = 0, nu = 0, ntab = 0, part = 0;
    for (int p = 0; p < L.n_paths; ++p) {
        const int R = (L.path[p].r + 31) / 32;
        cbs += R;
        nu += rb * s2_parts(R);
        ntab += 8 * R;
        part = std::max(part, std::min(R, kPartWords));
    }
    const double xchg = 20.0;
    auto t1_of = [&](int k) { return (double)((cbs + k - 1) / k) * (nw + 3); };
    auto t2_of = [&](int k) {
        return (double)((nu + k - 1) / k) * (part + 1) + 3.0 * ((ntab + 32 * k - 1) / (32 * k)) +
               1.0;
    };
    // phased only while every linear has a slot of its own (stage 1 of linear
    // kSlots would wait for a slot that only stage 2 frees)
    int best = 0;
    double best_t = M <= kSlots ? M * t1_of(kCW) + std::max(0.0, xchg - (M - 1) * t1_of(kCW)) +
                                      M * t2_of(kCW)
                                : 1e300;
    for (int k1 = 1; k1 < kCW; ++k1) {
        const double t1 = t1_of(k1), t2 = t2_of(kCW - k1);
        const double t = std::max(M * t1, t1 + xchg + M * t2);
        if (t < best_t - 1e-9) {
            best_t = t;
            best = k1;
        }
    }
    return best;
}

int rsum(const lb_linear &L) {
    int s = 0;
    for (int p = 0; p < L.n_paths; ++p) s += L.path[p].r;
    return s;
}

cudaError_t multi_setup(int *max_smem) {
    static std::mutex mu;
    static int smem_of[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 0 && dev < 64 && smem_of[dev] > 0) {
        *max_smem = smem_of[dev];
        return cudaSuccess;
    }
    int optin = 0;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    const int usable = optin - 1024;  // the kernel's static shared memory
    e = cudaFuncSetAttribute((const void *)k_decode_multi,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, usable);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) smem_of[dev] = usable;
    *max_smem = usable;
    return cudaSuccess;
}

}  // namespace

bool multi_supported(const lb_linear *L, int M, int num_sms) {
    if (M < 1 || M > kMaxMultiLinears || num_sms < 1 || num_sms > 255) return false;
    const lb_linear &A = L[0];
    if (A.d_out % 8 != 0) return false;
    for (int m = 0; m < M; ++m) {
        const lb_linear &B = L[m];
        if (B.d_in != A.d_in || B.d_out != A.d_out || B.n_paths != A.n_paths) return false;
        for (int p = 0; p < A.n_paths; ++p)
            if (B.path[p].r != A.path[p].r || B.path[p].r % 8 != 0) return false;
    }
    return true;
}

size_t multi_ws_bytes(const lb_linear &L, int M) {
    // two buffers of M * rsum exchange elements of t and a sum-of-squares element
    return (2 * fix2_words((size_t)M * rsum(L) + 1) * sizeof(unsigned long long) + 255) &
           ~(size_t)255;
}

cudaError_t launch_decode_multi(const lb_linear *L, int M, const void *x, int x_fp32, void *y,
                                int y_fp32, unsigned *ws_words, void *xw, int num_sms,
                                cudaStream_t s, float *res_a, const float *res_y) {
    int max_smem = 0;
    cudaError_t e = multi_setup(&max_smem);
    if (e != cudaSuccess) return e;
    MultiParams P{};
    const lb_linear &A = L[0];
    P.d_in = A.d_in;
    P.d_out = A.d_out;
    P.np = A.n_paths;
    P.r[0] = A.path[0].r;
    P.r[1] = A.n_paths > 1 ? A.path[1].r : 0;
    P.M = M;
    P.N1 = rsum(A);
    P.off1 = A.path[0].r;
    P.x = x;
    P.x_fp32 = x_fp32;
    P.res_a = res_a;
    P.res_y = res_y;
    P.y = y;
    P.y_fp32 = y_fp32;
    P.ws_words = ws_words;
    P.xw = static_cast<unsigned long long *>(xw);
    P.fix_limit = fix2_limit(num_sms);
    P.o = layout_of(A, num_sms);
    P.k1 = stage1_warps(A, num_sms, M);
    if (P.o.bytes > max_smem) return cudaErrorCooperativeLaunchTooLarge;
    for (int m = 0; m < M; ++m)
        for (int p = 0; p < A.n_paths; ++p) {
            const lb_path &Q = L[m].path[p];
            P.p[m].v[p] = Q.v_bits;
            P.p[m].u[p] = Q.u_bits;
            P.p[m].g[p] = Q.g;
            P.p[m].l[p] = Q.l;
            P.p[m].h[p] = Q.h;
        }
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)k_decode_multi, dim3(num_sms), dim3(kMT), args,
                                       (size_t)P.o.bytes, s);
}

}  // namespace lb
