// lb_decode.cu -- one token through one LittleBit linear (T = 1) in one launch.
//
// Prop. 1 (LittleBit, arXiv 2506.13771), per path: t = V_sign^T (g . x)
// (stage 1, a +-1 reduction over d_in), then y = h . (U_sign (l . t))
// (stage 2, a +-1 reduction over r); Eq. 6 sums the paths.  One CTA per SM:
//   * at launch thread 0 bulk-copies (cp.async.bulk) the CTA's V words (its
//     slice of input words, all columns) and U rows (its slice of output
//     rows, all words); U lands while stage 1 runs;
//   * stage 1: nibble tables of the CTA's g . x, then 32 columns per warp
//     over the slice, each partial t added to the exchange pair of its
//     element (an exact two-word fixed-point sum whose low bits count the
//     contributions, see send_fix2);
//   * stage 2: every thread waits for the four elements of one l . t table
//     and builds it; then each warp sums one part (32 rows x up to 4 words
//     of a path), times h, into its own shared slot, and the slots of a row
//     are added in a fixed order into y;
//   * the exchange words are double-buffered by a launch epoch kept in the
//     workspace header: while a launch uses one buffer, every CTA clears its
//     stripe of the other (the previous launch's), so no launch needs a
//     memset or a clean-up step after its last read.
// Every wait is bounded (about one second); on a timeout the CTA records
// LB_ERR_TIMEOUT, waits for its own copies and returns.
#include <mutex>

#include "lb_common.cuh"
#include "lb_kernels.h"
#include "lb_lut.cuh"

namespace lb {

namespace {

constexpr int kDT = 512;  // threads per CTA
constexpr int kDW = kDT / 32;

// Shared-memory byte offsets, from the largest slices of any CTA.
struct DecodeLayout {
    int V[2], U[2], h[2], xg[2], t1, t2, y, bytes;
};

struct DecodeParams {
    LinDesc L;
    const void *x;     // bf16 [d_in]; fp32 [d_in] (x_fp32 = 1); fp32 [2][d_in] (x_fp32 = 2)
    int x_fp32;        // 2: the input is silu(x[0][i]) * x[1][i] (a decoder MLP's gate, up)
    void *y;
    int y_fp32;
    unsigned *ws_words;
    unsigned long long *xw;  // exchange pairs: two buffers of N1 (paths concatenated)
    int N1, off1;
    float fix_limit;         // |partial| bound that keeps the fixed-point sum in range
    DecodeLayout o;
};

__device__ bool wait_bar(unsigned long long *bar, unsigned *ws_words) {
    if (mbar_try_wait(bar, 0)) return true;
    const unsigned long long t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, 0)) {
        __nanosleep(32);
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
            return false;
        }
    }
    return true;
}

__global__ void __launch_bounds__(kDT, 1) k_decode(const __grid_constant__ DecodeParams P) {
    __shared__ __align__(8) unsigned long long bar[2];
    unsigned *err = P.ws_words + kErrWord;
    if (ld_relaxed_gpu(err) != 0u) return;
    // this launch's buffer of exchange words, and the previous launch's; the
    // epoch moves on only after every CTA has read it (block 0 bumps it once
    // its exchange completed, which needs every CTA's contributions)
    const unsigned epoch = ld_relaxed_gpu(P.ws_words + kEpochWord);
    const int nwords = (int)fix2_words(P.N1);  // one buffer
    unsigned long long *xw = P.xw + (size_t)(epoch & 1u) * nwords;
    unsigned long long *xold = P.xw + (size_t)((epoch + 1u) & 1u) * nwords;
    const LinDesc &L = P.L;
    const DecodeLayout &o = P.o;
    const int N = gridDim.x, c = blockIdx.x, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    // input words [iw0, iw0 + nw) (stage-1 CTAs only), output rows [o0, o0 +
    // nrows) (whole octets)
    const int W = L.d_in >> 5, Q = L.d_out >> 3;
    int iw0, nw;
    s1_slice(W, N, c, iw0, nw);
    // contributions per exchange element: the stage-1 CTAs; element 0 also
    // counts every other CTA once, so that block 0's exchange completes only
    // after every CTA has read the epoch
    const int n_s1 = s1_ctas(W, N);
    const unsigned n_all = (unsigned)N, n_part = (unsigned)n_s1;
    const int q0 = (int)((long long)c * Q / N), nq = (int)((long long)(c + 1) * Q / N) - q0;
    const int o0 = 8 * q0, nrows = 8 * nq;
    const int np = L.n_paths;

    if (tid == 0) {
        mbar_init(bar + 0, 1);
        mbar_init(bar + 1, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0) {
        for (int p = 0; p < np; ++p) {
            const int r = p ? L.r[1] : L.r[0];
            if (nw > 0) {
                const unsigned bytes = (unsigned)(nw * r * 4);
                mbar_expect_tx(bar + 0, bytes);
                bulk_g2s(g_smem + o.V[p], (p ? L.v[1] : L.v[0]) + (size_t)iw0 * r, bytes, bar + 0);
            }
            const int R = (r + 31) >> 5;
            if (nrows > 0) {
                const unsigned bytes = (unsigned)(nrows * R * 4);
                mbar_expect_tx(bar + 1, bytes + (unsigned)(2 * nrows));
                bulk_g2s(g_smem + o.U[p], (p ? L.u[1] : L.u[0]) + (size_t)o0 * R, bytes, bar + 1);
                bulk_g2s(g_smem + o.h[p], (p ? L.h[1] : L.h[0]) + o0, (unsigned)(2 * nrows),
                         bar + 1);
            }
        }
        mbar_arrive(bar + 0);
        mbar_arrive(bar + 1);
    }
    // g . x of the slice by plain loads (l and h are read where they are
    // used, their latency hidden behind the exchange and the stage-2 sums)
    for (int p = 0; p < np; ++p) {
        const uint16_t *g = p ? L.g[1] : L.g[0];
        float *xg = reinterpret_cast<float *>(g_smem + o.xg[p]);
        for (int i = tid; i < 32 * nw; i += kDT) {
            const int e = 32 * iw0 + i;
            float xe;
            if (P.x_fp32 == 2) {
                const float *xf = static_cast<const float *>(P.x);
                const float gt = xf[e];
                xe = xf[L.d_in + e] * (gt / (1.f + expf(-gt)));
            } else {
                xe = P.x_fp32 ? static_cast<const float *>(P.x)[e]
                              : bf16_bits_to_float(static_cast<const uint16_t *>(P.x)[e]);
            }
            xg[i] = xe * half_bits_to_float(g[e]);
        }
    }
    // stage-2 part slots: path 0's s2_parts(R0) slots, then path 1's, nrows each
    float *y = reinterpret_cast<float *>(g_smem + o.y);
    __syncthreads();

    // ---- stage 1: tables of g . x (8 per input word and path), then columns
    for (int idx = tid; idx < np * 8 * nw; idx += kDT) {
        const int p = idx / (8 * nw), n = idx - p * 8 * nw;  // n: table of the slice
        const float4 v = *reinterpret_cast<const float4 *>(g_smem + o.xg[p] + 16 * n);
        store_table(g_smem + o.t1 + idx * 128, v, lane);
    }
    bool ok = wait_bar(bar + 0, P.ws_words);
    ok = __syncthreads_and(ok) != 0;
    if (ok && c >= n_s1 && tid == 0) send_count2(fix2_at(xw, 0));
    if (ok && c < n_s1) {
        const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
        const int cb0 = (L.r[0] + 31) >> 5, cbs = cb0 + (np > 1 ? (L.r[1] + 31) >> 5 : 0);
        for (int u = warp; u < cbs; u += kDW) {
            const int p = u >= cb0 ? 1 : 0, cb = u - (p ? cb0 : 0);
            const int r = p ? L.r[1] : L.r[0];
            const int col = 32 * cb + lane, cc = min(col, r - 1);
            const uint32_t *Vw = reinterpret_cast<const uint32_t *>(g_smem + o.V[p]) + cc;
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
                send_fix2(fix2_at(xw, (p ? P.off1 : 0) + col), acc0 + acc1, P.fix_limit, err);
        }
    }
    // the previous launch's words: this CTA's stripe back to zero
    {
        const int a = (int)((long long)c * nwords / N), b = (int)((long long)(c + 1) * nwords / N);
        for (int i = a + tid; i < b; i += kDT) xold[i] = 0ull;
    }

    // ---- stage 2 tables: thread i waits for the elements of table i (l . t)
    const int nt0 = 8 * ((L.r[0] + 31) >> 5), ntab = nt0 + (np > 1 ? 8 * ((L.r[1] + 31) >> 5) : 0);
    int pok = ok ? 1 : 0;
    for (int idx = tid; idx < ntab && pok; idx += kDT) {
        const int p = idx >= nt0 ? 1 : 0, n = idx - (p ? nt0 : 0);
        const int r = p ? L.r[1] : L.r[0];
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (4 * n < r) {
            const uint2 lw = __ldg(reinterpret_cast<const uint2 *>((p ? L.l[1] : L.l[0]) + 4 * n));
            const unsigned long long *wd = fix2_at(xw, (p ? P.off1 : 0) + 4 * n);
            unsigned long long a[8], t0 = 0;
            for (int spin = 0;; ++spin) {
                ld_fix2x4(wd, a);
                if (counted2x4(a, idx == 0 ? n_all : n_part, n_part)) break;
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
            v = make_float4(dec_fix2(a[0], a[1]) * half_bits_to_float((uint16_t)(lw.x & 0xffffu)),
                            dec_fix2(a[2], a[3]) * half_bits_to_float((uint16_t)(lw.x >> 16)),
                            dec_fix2(a[4], a[5]) * half_bits_to_float((uint16_t)(lw.y & 0xffffu)),
                            dec_fix2(a[6], a[7]) * half_bits_to_float((uint16_t)(lw.y >> 16)));
        }
        store_table(g_smem + o.t2 + idx * 128, v, lane);
    }
    const bool u_ok = wait_bar(bar + 1, P.ws_words);
    ok = __syncthreads_and(pok && u_ok) != 0;
    // every CTA contributed before block 0's exchange could complete, so all
    // of them have read the epoch: the next launch may use the other buffer
    if (ok && c == 0 && tid == 0) P.ws_words[kEpochWord] = epoch + 1u;
    if (ok) {
        // ---- stage 2: parts of 32 rows x up to four words of one path
        const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
        const int rb = (nrows + 31) >> 5;
        const int R0 = (L.r[0] + 31) >> 5, R1 = np > 1 ? (L.r[1] + 31) >> 5 : 0;
        const int S0 = s2_parts(R0), S1 = np > 1 ? s2_parts(R1) : 0;
        const int n0 = rb * S0, nu = n0 + rb * S1;
        for (int u = warp; u < nu; u += kDW) {
            const int p = u >= n0 ? 1 : 0, v = u - (p ? n0 : 0), S = p ? S1 : S0;
            const int b = v / S, sp = v - b * S;
            s2_part(reinterpret_cast<const uint32_t *>(g_smem + o.U[p]), p ? R1 : R0,
                    reinterpret_cast<const uint16_t *>(g_smem + o.h[p]),
                    (uint32_t)(o.t2 + (p ? nt0 : 0) * 128), nrows, b, sp,
                    y + (size_t)((p ? S0 : 0) + sp) * nrows, copy, lane);
        }
        __syncthreads();
        for (int i = tid; i < nrows; i += kDT) {
            const float v = s2_combine(y, nrows, S0 + S1, i);
            if (P.y_fp32)
                static_cast<float *>(P.y)[o0 + i] = v;
            else
                static_cast<uint16_t *>(P.y)[o0 + i] = float_to_bf16_bits(v);
        }
    } else if (tid == 0) {
        // the copies of this CTA must land before it goes away
        wait_bar(bar + 0, P.ws_words);
        wait_bar(bar + 1, P.ws_words);
    }
}

int up16(int n) { return (n + 15) & ~15; }

DecodeLayout layout_of(const lb_linear &L, int N) {
    const int W = L.d_in / 32, n_s1 = s1_ctas(W, N);
    const int nw = (W + n_s1 - 1) / n_s1, nrows = 8 * ((L.d_out / 8 + N - 1) / N);
    DecodeLayout o{};
    int at = 0;
    auto take = [&at](int bytes) {
        const int off = at;
        at += up16(bytes);
        return off;
    };
    int ntab2 = 0, nslot = 0;
    for (int p = 0; p < 2; ++p) {
        const bool on = p < L.n_paths;
        const int r = on ? L.path[p].r : 0, R = (r + 31) / 32;
        o.V[p] = take(nw * r * 4);
        o.U[p] = take(nrows * R * 4);
        o.h[p] = take(2 * nrows);
        o.xg[p] = take(on ? 128 * nw : 0);
        ntab2 += 8 * R;
        nslot += on ? s2_parts(R) : 0;
    }
    // table bases are 1024-aligned: lut8 splices the entry byte into them
    at = (at + 1023) & ~1023;
    o.t1 = take(L.n_paths * 8 * nw * 128);
    at = (at + 1023) & ~1023;
    o.t2 = take(ntab2 * 128);
    o.y = take(4 * nrows * nslot);
    o.bytes = at;
    return o;
}

int rsum_of(const lb_linear &L) {
    int s = 0;
    for (int p = 0; p < L.n_paths; ++p) s += L.path[p].r;
    return s;
}

// Shared-memory opt-in (the device maximum, so one call serves every shape)
// and the largest co-resident grid, once per device.
cudaError_t device_setup(int *max_smem) {
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
    e = cudaFuncSetAttribute((const void *)k_decode, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             usable);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) smem_of[dev] = usable;
    *max_smem = usable;
    return cudaSuccess;
}

}  // namespace

bool decode_supported(const lb_linear &L, int num_sms) {
    if (L.d_out % 8 != 0 || num_sms < 1 || num_sms > 255) return false;
    for (int p = 0; p < L.n_paths; ++p)
        if (L.path[p].r % 8 != 0) return false;
    return true;
}

size_t decode_ws_bytes(const lb_linear &L) {
    // two buffers of rsum exchange elements
    return (2 * fix2_words(rsum_of(L)) * sizeof(unsigned long long) + 255) & ~(size_t)255;
}

cudaError_t launch_decode(const lb_linear &L, const void *x, int x_fp32, void *y, int y_fp32,
                          unsigned *ws_words, void *xw, int num_sms, cudaStream_t s) {
    int max_smem = 0;
    cudaError_t e = device_setup(&max_smem);
    if (e != cudaSuccess) return e;
    DecodeParams P{};
    P.L = make_desc(L);
    P.x = x;
    P.x_fp32 = x_fp32;
    P.y = y;
    P.y_fp32 = y_fp32;
    P.ws_words = ws_words;
    P.xw = static_cast<unsigned long long *>(xw);
    P.N1 = rsum_of(L);
    P.off1 = L.path[0].r;
    P.fix_limit = fix2_limit(num_sms);
    P.o = layout_of(L, num_sms);
    if (P.o.bytes > max_smem) return cudaErrorCooperativeLaunchTooLarge;
    void *args[] = {&P};
    return cudaLaunchCooperativeKernel((const void *)k_decode, dim3(num_sms), dim3(kDT), args,
                                       (size_t)P.o.bytes, s);
}

}  // namespace lb
