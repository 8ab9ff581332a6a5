// lb_stack.cu -- one decode token through n_layers Llama-shaped decoder blocks
// whose seven linears are LittleBit linears, as ONE persistent launch with one
// CTA per SM (littlebit_stack_forward).
//
// Per linear, Prop. 1 (LittleBit, arXiv 2506.13771) is a +-1 reduction over
// d_in (stage 1, rank-r result t) followed by a +-1 reduction over r (stage
// 2), per path, paths summed (Eq. 6).  CTA c owns
//   R_c : a slice of d rows, whole 32-row words    (q, o, down outputs; the
//         residual stream; stage-1 inputs of q, k, v, o, gate, up)
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
//  * the compute warps run a per-CTA program built on the host by
//    littlebit_stack_prepare: for every step, warp-balanced work units with
//    their shared-memory offsets -- stage-2 tables polled from the exchange,
//    row units (16 output rows of a critical linear summed whole by one warp,
//    the two half-warps on the two paths (or on gate and up), followed by
//    the stage-1 tables of those rows), 32 columns x the slice for stage 1.
//    The shapes are those of every layer, so the program is the same for all
//    of them; the device code is a handful of generic loops;
//  * the all-reduce of t accumulates every element as a fixed-point sum in
//    one 64-bit word whose low 8 bits count contributions (send_fix1: one
//    red.add per element and contribution) and readers poll the words they
//    need until the count is complete -- no fence, no separate barrier, an
//    order-independent sum.  Its scale is set per exchange, identically in
//    every CTA, from a rigorous bound on the contributions: |t_j| <= max|g|
//    x the L1 norm of the stage-1 input, that norm bounded through the
//    chain's residual adds, attention and SiLU product from per-linear
//    constants (max|g|, the L1 norm and maximum of |h|, computed once by
//    littlebit_stack_prepare) and the largest per-unit |z| sum of the tables
//    each CTA built from the previous exchange (an order-independent max, so
//    every CTA derives the same scale).  The resolution is then about 2^-53
//    n B at any input scale, and a contribution beyond twice the bound (a
//    broken bound) is recorded as LB_ERR_RANGE, never wrapped;
//  * q and k (not read again at position 0) are computed after the CTA has
//    sent its share of the next exchange, off the critical path.
// Every wait is bounded (about one second); on a timeout the CTA records
// LB_ERR_TIMEOUT, waits for its own bulk copies to land, and returns.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "lb_common.cuh"
#include "lb_kernels.h"
#include "lb_lut.cuh"

namespace lb {

namespace {

constexpr int kST = 512;        // threads per CTA
// CTAs per thread-block cluster, C (the kernel is built for C = 1 and 2 and
// chosen at run time): with C = 2 the stage-1 partial sums of a cluster's
// CTAs meet in distributed shared memory before one exchange contribution
// per cluster goes out; with C = 1 every CTA contributes.
constexpr int kMaxCluster = 2;
constexpr int kCW = 15;         // compute warps; warp 15 issues the bulk copies
constexpr int kCT = kCW * 32;   // compute threads
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
    // the phase's two float4 of exchange-bound constants (cst, per layer)
    int cst[4];
    // work areas: stage-2 and stage-1 tables, residual stream (two buffers:
    // phase A reads 0 and writes 1, phase C the reverse), the off-path q, k, v
    // outputs (added into, zeroed once stored), the program
    int t2, t1, res0, res1, yq, yk, yv, prog;
    // per-unit sums of squares of the residual row steps (kMaxSlots floats)
    int ssslot;
    // cluster reduction of the stage-1 partials, per phase X = A..D: the
    // receive slots of the units this CTA owns (C x 32 floats each,
    // one row per sending rank) and the index of their first mbarrier in ubar
    int slot[4], ubar0[4], ubar, n_ubar;
};

// Steps of the per-CTA program (one per table build or unit loop).
// (*_P2: stage-2 tables straight from the exchange words; *_R: row units,
// stage 2 with the stage-1 tables of its rows; *_S2 / *_S1: stage-2 /
// stage-1 units.)
enum StepId {
    A_P2, A_R, A_S1,
    B_P2, B_R, B_S1, B_S2QKV,
    C_P2, C_R, C_S1,
    D_P2, D_R, D_S1,
    N_STEPS
};

// One program record (8 ints).  Meaning by step kind:
//   poll-table  : tb, n_tab, n_vals, mode, e0, scale, ss_el, job  (e0, ss_el:
//                 exchange word indices in the layer; ss_el < 0: none; job:
//                 the bound entry 0-3 the unit's |z| sum goes to, -1: none)
//   stage-2 unit: U, R, nw, tb, h, out, nrows, -
//   stage-1 unit: V, r, nw, tb, dst, ncols, own, slot  (own: the cluster rank
//                 that sums the unit's partials and sends them; slot: the
//                 unit's receive slot and mbarrier at that rank)
//   row unit    : a header  nseg, n_job, mode | log2(nr) << 8, nrows, res_in,
//                 res_out, slot, -
//                 then per lane group (32 / nr of them) nseg segments
//                 U, R, nw, tb, h, -, -, -
//                 then per table job  tb, g, -, -, -, -, -, -
//                 (offsets of the unit's first row; slot: the unit's
//                 sum-of-squares slot, ROW_RES)
struct Item {
    int f[8];
};
// Poll-table modes.
enum { TAB_PLAIN = 0, TAB_MUL = 8 };
// Row-unit modes: x = A + B;  x = res_in + A + B (stored to res_out, x^2
// added to the sum of squares);  x = silu(A) * B.
enum { ROW_SUM = 0, ROW_RES = 1, ROW_SILU = 2 };

// Warp w runs units [first + wo[w], first + wo[w + 1]) of its step (records,
// for a row step).
struct Step {
    int first;
    int wo[kCW + 1];
    int nslot;  // sum-of-squares slots written by the step (ROW_RES)
};
constexpr int kStepBytes = (int)((N_STEPS * sizeof(Step) + 15) / 16 * 16);
constexpr int kProgBytes = 16384;  // per CTA, in the workspace and in shared memory
constexpr int kMaxItems = (kProgBytes - kStepBytes) / (int)sizeof(Item);
constexpr int kMaxCtas = 255;      // the 8-bit contribution count of the exchange
constexpr int kMaxSlots = 64;      // row units of a residual step
constexpr unsigned kEarlyRead = 30;  // a poll's lanes read this many contributions early
#ifndef LB_ROW_MIN_LNR
#define LB_ROW_MIN_LNR 3
#endif
constexpr int kRowMinLnr = LB_ROW_MIN_LNR;  // smallest row unit: 1 << kRowMinLnr rows

struct Params {
    const LinDesc *lin;  // 7 * n_layers descriptors in the workspace
    const int *prog;     // kProgBytes per CTA in the workspace
    int n_layers, d, dkv, dff, hd;
    int np[7], r[7][2];  // paths and ranks of q, k, v, o, gate, up, down
    const uint16_t *x0;
    float *out, *q_out, *kv_out;
    unsigned *ws_words;
    unsigned long long plan;
    unsigned long long *xacc;  // exchange words, n_layers * acc_layer
    unsigned n_t;              // contributions per t element: one per cluster
    // per layer l (0..n_layers) and phase X, two float4 of constants for the
    // exchange bounds (k_stack_consts): c[0..3], then max|g| of the
    // linears whose stage 1 the phase sends
    const float4 *cst;
    int acc_layer, offA, offQ, offB, offC, offD, lenA, lenQ, lenB, lenC, lenD;
    // largest |scaled contribution| of a t / mean-square element: below
    // 2^55 / contributions, so no complete sum leaves the word
    float lim_t, lim_ss;
    Offsets o;
};

// ---------------------------------------------------------------- small pieces

// Units [w0, w0 + n) of W (32-row words or 8-row octets) owned by CTA c of N.
// In clusters the clusters split the units evenly in whole multiples of the
// cluster size and each member takes an equal share: the members' stage-1
// partials meet in the owner, which would wait for a member with more work.
// (Units not divisible that way are split per CTA.)
__host__ __device__ inline void slice_of(int W, int N, int c, int C, int &w0, int &n) {
    if (C > 1 && W % C == 0 && N % C == 0) {
        const int Wc = W / C, Nc = N / C, k = c / C;
        const int u0 = (int)((long long)k * Wc / Nc), u1 = (int)((long long)(k + 1) * Wc / Nc);
        n = u1 - u0;
        w0 = C * u0 + (c % C) * n;
        return;
    }
    w0 = (int)((long long)c * W / N);
    n = (int)((long long)(c + 1) * W / N) - w0;
}

__device__ __forceinline__ int wordsR(int r) { return (r + 31) >> 5; }

__device__ __forceinline__ float *sm_f(int off) { return reinterpret_cast<float *>(g_smem + off); }
__device__ __forceinline__ const uint32_t *sm_u32(int off) {
    return reinterpret_cast<const uint32_t *>(g_smem + off);
}
__device__ __forceinline__ const uint16_t *sm_u16(int off) {
    return reinterpret_cast<const uint16_t *>(g_smem + off);
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }


// The program lives in shared memory at byte offset prog; step and unit
// records are read with shared-memory loads (the step functions take byte
// offsets, not generic pointers, so the compiler knows the state space).
__device__ __forceinline__ const Step &step_at(int prog, int s) {
    return *reinterpret_cast<const Step *>(g_smem + prog + s * (int)sizeof(Step));
}
__device__ __forceinline__ void item_at(int prog, int u, int4 &a, int4 &b) {
    const unsigned char *p = g_smem + prog + kStepBytes + u * (int)sizeof(Item);
    a = *reinterpret_cast<const int4 *>(p);
    b = *reinterpret_cast<const int4 *>(p + 16);
}

// Row units: nr = 16, 8 or 4 output rows of a stage-2 step summed whole
// inside one warp, then the stage-1 tables of those rows, with no shared
// accumulator and no barrier in between.  Lane l takes row l mod nr and lane
// group l / nr: the groups of lanes 0-15 split the words of the first half
// of the work (path 0, or gate in phase D) and those of lanes 16-31 the
// second (path 1, or up), each group a run of words of one or more segments.
// The two half-warps read the two copies of every table.  Shuffles join the
// groups into x (by the unit's mode; a butterfly, so every lane of a row gets
// the same value).  Table job j then gets the unit's nr / 4 tables, table n
// of v_i = x_i * g_j[i], i = 4n + k.  do_s2 = false takes A = B = 0 (the
// first layer has no previous down); do_tab = false builds no tables (the
// last phase).  ROW_RES units leave the sum of squares of their rows in
// ss[slot] (added in slot order later, so the total does not depend on
// which warp finishes first).
__device__ __noinline__ void run_rows(int prog, int s, bool do_s2, bool do_tab, float *ss) {
    const Step &st = step_at(prog, s);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    const int u1 = st.first + st.wo[warp + 1];
    for (int u = st.first + st.wo[warp]; u < u1;) {
        int4 hd, he;
        item_at(prog, u, hd, he);
        const int nseg = hd.x, njob = hd.y, mode = hd.z & 0xff, lnr = hd.z >> 8, nrows = hd.w;
        const int nr = 1 << lnr, G = 32 >> lnr;
        const int row = min(lane & (nr - 1), nrows - 1);
        const int seg0 = u + 1 + (lane >> lnr) * nseg;
        // the residual input does not depend on the sums: load it first
        const float res = mode == ROW_RES && lane < nrows ? sm_f(he.x)[lane] : 0.f;
        float acc = 0.f;
        if (do_s2) {
#pragma unroll 1
            for (int k = 0; k < nseg; ++k) {
                int4 a, b;
                item_at(prog, seg0 + k, a, b);
                const int nw = a.z;
                const uint32_t *Uw = sm_u32(a.x) + row * a.y;
                const uint32_t tb = (uint32_t)a.w;
                float s0 = 0.f, s1 = 0.f;
                int w = 0;
#pragma unroll 1
                for (; w + 2 <= nw; w += 2) {
                    s0 += lut_word(Uw[w], copy, tb + w * 1024);
                    s1 += lut_word(Uw[w + 1], copy, tb + (w + 1) * 1024);
                }
                if (w < nw) s0 += lut_word(Uw[w], copy, tb + w * 1024);
                if (nw > 0) acc += (s0 + s1) * half_bits_to_float(sm_u16(b.x)[row]);
            }
        }
        float x = acc;
        if (mode == ROW_SILU) {
            // gate in lanes 0-15, up in lanes 16-31
            for (int o = nr; o < 16; o <<= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
            const float other = __shfl_xor_sync(0xffffffffu, x, 16);
            x = silu(x) * other;
        } else {
            for (int o = nr; o < 32; o <<= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
        }
        if (lane >= nrows) x = 0.f;  // also every lane beyond the unit's rows
        if (mode == ROW_RES) {
            float q = 0.f;
            if (lane < nrows) {
                x += res;
                sm_f(he.y)[lane] = x;
                q = x * x;
            }
            for (int o = nr >> 1; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
            if (lane == 0) ss[he.z] = q;
        }
        if (do_tab) {
            const int ltj = lnr - 2;  // log2 of the tables per job
            const int n = lane & ((1 << ltj) - 1);
            const float4 v = make_float4(__shfl_sync(0xffffffffu, x, 4 * n),
                                         __shfl_sync(0xffffffffu, x, 4 * n + 1),
                                         __shfl_sync(0xffffffffu, x, 4 * n + 2),
                                         __shfl_sync(0xffffffffu, x, 4 * n + 3));
#pragma unroll 1
            for (int L = lane; L < (njob << ltj); L += 32) {
                int4 ta, tz;
                item_at(prog, u + 1 + G * nseg + (L >> ltj), ta, tz);
                const uint2 hb = *reinterpret_cast<const uint2 *>(g_smem + ta.y + 8 * n);
                const float4 t =
                    make_float4(v.x * half_bits_to_float((uint16_t)(hb.x & 0xffffu)),
                                v.y * half_bits_to_float((uint16_t)(hb.x >> 16)),
                                v.z * half_bits_to_float((uint16_t)(hb.y & 0xffffu)),
                                v.w * half_bits_to_float((uint16_t)(hb.y >> 16)));
                store_table(g_smem + ta.x + 128 * n, t, lane);
            }
        }
        u += 1 + G * nseg + njob;
    }
}

// Stage-2 units: out[row] += h[row] * sum over the unit's words of the
// +-1 products of U's row with the tabled t (lane = row).
__device__ __noinline__ void run_s2(int prog, int s) {
    const Step &st = step_at(prog, s);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    const int u1 = st.first + st.wo[warp + 1];
    int u = st.first + st.wo[warp];
    // two units per pass: their word loops run side by side (a unit has at
    // least one word; the shorter one re-reads its last word, masked out)
    for (; u + 2 <= u1; u += 2) {
        int4 a, b, c, d;
        item_at(prog, u, a, b);
        item_at(prog, u + 1, c, d);
        const uint32_t *U0 = sm_u32(a.x) + min(lane, b.z - 1) * a.y;
        const uint32_t *U1 = sm_u32(c.x) + min(lane, d.z - 1) * c.y;
        const int nw = max(a.z, c.z);
        float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 1
        for (int w = 0; w < nw; ++w) {
            const int w0 = min(w, a.z - 1), w1 = min(w, c.z - 1);
            const float v0 = lut_word(U0[w0], copy, (uint32_t)a.w + w0 * 1024);
            const float v1 = lut_word(U1[w1], copy, (uint32_t)c.w + w1 * 1024);
            acc0 += w < a.z ? v0 : 0.f;
            acc1 += w < c.z ? v1 : 0.f;
        }
        if (lane < b.z) atomicAdd(sm_f(b.y) + lane, acc0 * half_bits_to_float(sm_u16(b.x)[lane]));
        if (lane < d.z) atomicAdd(sm_f(d.y) + lane, acc1 * half_bits_to_float(sm_u16(d.x)[lane]));
    }
    if (u < u1) {
        int4 a, b;
        item_at(prog, u, a, b);
        const int R = a.y, nw = a.z, nrows = b.z;
        const uint32_t tb = (uint32_t)a.w;
        const int row = min(lane, nrows - 1);
        const uint32_t *Uw = sm_u32(a.x) + row * R;
        float acc0 = 0.f, acc1 = 0.f;
        int w = 0;
#pragma unroll 1
        for (; w + 2 <= nw; w += 2) {
            const uint32_t w0 = Uw[w], w1 = Uw[w + 1];
            acc0 += lut_word(w0, copy, tb + w * 1024);
            acc1 += lut_word(w1, copy, tb + (w + 1) * 1024);
        }
        if (w < nw) acc0 += lut_word(Uw[w], copy, tb + w * 1024);
        if (lane < nrows)
            atomicAdd(sm_f(b.y) + lane, (acc0 + acc1) * half_bits_to_float(sm_u16(b.x)[lane]));
    }
}

__device__ __forceinline__ bool sticky(const unsigned *ws_words) {
    return ld_relaxed_gpu(ws_words + kErrWord) != 0u;
}

__device__ __forceinline__ void record(unsigned *ws_words, lb_status st) {
    atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(st));
}

// Stage-1 units: t[col] partial over the CTA's input slice (lane = column).
// Every CTA has a unit for every column, also when its slice is empty (it
// then contributes zeros).  Without clusters each partial goes straight into
// the exchange words (at scale sc).  With clusters a unit belongs to one rank of the
// cluster: the other ranks store their partials into its receive slot in
// the owner's shared memory (st.async, completing on the slot's mbarrier),
// and the owner adds them to its own in rank order and sends the sum -- one
// contribution per cluster.  A warp runs the units it does not own first.
// Returns false (this warp) when an owner's wait ran out.
template <int C>
__device__ __noinline__ bool run_s1(int prog, int s, unsigned long long *xbase, float sc,
                                    float limit, unsigned *err, int slot0, int ubar0, int ubar,
                                    unsigned par, unsigned rank, unsigned *ws_words) {
    const Step &st = step_at(prog, s);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t copy = (lane >> 4) ? 0x40404040u : 0u;
    const int u0 = st.first + st.wo[warp], u1 = st.first + st.wo[warp + 1];
    auto bar_of = [&](int slot) {
        return reinterpret_cast<unsigned long long *>(g_smem + ubar) + ubar0 + slot;
    };
    if (C > 1 && lane == 0) {
        // arm the mbarriers of this warp's own units for this use
        for (int u = u0; u < u1; ++u) {
            int4 a, b;
            item_at(prog, u, a, b);
            if ((unsigned)b.z == rank)
                mbar_arrive_expect_tx(bar_of(b.w), (unsigned)((C - 1) * 4 * b.y));
        }
    }
    __syncwarp();
    bool ok = true;
    // one finished unit: its partial v of column `lane`
    auto finish = [&](const int4 &b, float v) {
        const int dst = b.x, ncols = b.y;
        if (C == 1) {
            if (lane < ncols) send_fix1(xbase + dst + lane, v, sc, limit, err);
            return;
        }
        const unsigned own = (unsigned)b.z;
        const int slot = b.w;
        if (own != rank) {
            if (lane < ncols) {
                const uint32_t loc =
                    saddr(g_smem + slot0 + (slot * C + (int)rank) * 128 + 4 * lane);
                st_async_f32(mapa(loc, own), v, mapa(saddr(bar_of(slot)), own));
            }
            return;
        }
        // owner: the other ranks' partials, then the sum in rank order
        if (!ok) return;
        unsigned long long *bar = bar_of(slot);
        if (!mbar_try_wait_cluster(bar, par)) {
            const unsigned long long t0 = globaltimer_ns();
            while (!mbar_try_wait_cluster(bar, par)) {
                if (sticky(ws_words) || globaltimer_ns() - t0 > kWaitLimitNs) {
                    record(ws_words, LB_ERR_TIMEOUT);
                    ok = false;
                    return;
                }
            }
        }
        const float *rx = reinterpret_cast<const float *>(g_smem + slot0 + slot * C * 128);
        float sum = 0.f;
#pragma unroll
        for (int k = 0; k < C; ++k) sum += (unsigned)k == rank ? v : rx[32 * k + lane];
        if (lane < ncols) send_fix1(xbase + dst + lane, sum, sc, limit, err);
    };
    int u = u0;
    // two units per pass; a unit whose input slice is empty (no words) reads
    // the first entries of its buffer and table, masked out, and sends zero
    for (; u + 2 <= u1; u += 2) {
        int4 a, b, c, d;
        item_at(prog, u, a, b);
        item_at(prog, u + 1, c, d);
        const uint32_t *V0 = sm_u32(a.x) + min(lane, b.y - 1);
        const uint32_t *V1 = sm_u32(c.x) + min(lane, d.y - 1);
        const int nw = max(a.z, c.z);
        float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 1
        for (int w = 0; w < nw; ++w) {
            const int w0 = max(min(w, a.z - 1), 0), w1 = max(min(w, c.z - 1), 0);
            const float v0 = lut_word(V0[w0 * a.y], copy, (uint32_t)a.w + w0 * 1024);
            const float v1 = lut_word(V1[w1 * c.y], copy, (uint32_t)c.w + w1 * 1024);
            acc0 += w < a.z ? v0 : 0.f;
            acc1 += w < c.z ? v1 : 0.f;
        }
        finish(b, acc0);
        finish(d, acc1);
    }
    if (u < u1) {
        int4 a, b;
        item_at(prog, u, a, b);
        const int r = a.y, nw = a.z, ncols = b.y;
        const uint32_t tb = (uint32_t)a.w;
        const uint32_t *Vw = sm_u32(a.x) + min(lane, ncols - 1);
        float acc0 = 0.f, acc1 = 0.f;
        int w = 0;
#pragma unroll 1
        for (; w + 2 <= nw; w += 2) {
            const uint32_t w0 = Vw[w * r], w1 = Vw[(w + 1) * r];
            acc0 += lut_word(w0, copy, tb + w * 1024);
            acc1 += lut_word(w1, copy, tb + (w + 1) * 1024);
        }
        if (w < nw) acc0 += lut_word(Vw[w * r], copy, tb + w * 1024);
        finish(b, acc0 + acc1);
    }
    return ok;
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

__device__ __forceinline__ void zero_f(float *p, int n) {
    for (int i = threadIdx.x; i < n; i += kCT) p[i] = 0.f;
}

// Exchange regions of a layer, in the order of their stripe bounds.
enum { XR_A = 0, XR_Q, XR_B, XR_C, XR_D, XR_N };

// Zero this CTA's stripe [z[0], z[1]) of an exchange region whose readers are
// all done (the bounds are computed once per launch).
__device__ __forceinline__ void zero_stripe(unsigned long long *region, const int *z) {
    for (int i = z[0] + threadIdx.x; i < z[1]; i += kCT) region[i] = 0ull;
}

// Poll-table units: the stage-2 tables of a phase built straight from the
// exchange words.  Lane n waits until the elements e0 + 4n .. +3 (those below
// n_vals) -- and the element ss_el, for a TAB_MUL unit that has one -- count
// n_t contributions (n_ss for ss_el), decodes them (inverse scales it, and
// iss for ss_el) and builds table n of v_i = t_i * l_i (* inv with TAB_MUL,
// inv = rsqrt(mean square) of element ss_el, or the argument when the unit
// has no ss_el).  A unit with a job adds the sum of its |v_i| (a fixed-order
// warp sum) to zmax[job] by max (fp32 bits of a non-negative value: an
// order-independent result).  Bounded; returns false (to every compute
// thread) on failure.
__device__ __noinline__ bool run_poll_tables(int prog, int s, const unsigned long long *xbase,
                                             unsigned n_t, unsigned n_ss, float inv, float it,
                                             float iss, unsigned *zmax, bool late,
                                             unsigned *ws_words) {
    const Step &st = step_at(prog, s);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int ok = 1;
    const int u1 = st.first + st.wo[warp + 1];
    for (int u = st.first + st.wo[warp]; u < u1 && ok; ++u) {
        int4 a, b;
        item_at(prog, u, a, b);
        const bool have = lane < a.y && a.z - 4 * lane > 0;
        const bool need_ss = have && (a.w & TAB_MUL) && b.z >= 0;
        const unsigned long long *w = xbase + b.x + 4 * lane;
        unsigned long long v0 = 0, v1 = 0, v2 = 0, v3 = 0, vs = 0, t0 = 0;
        auto complete = [&]() {
            return counted1(v0, n_t) && counted1(v1, n_t) && counted1(v2, n_t) &&
                   counted1(v3, n_t) && (!need_ss || counted1(vs, n_ss));
        };
        // late: the step starts when its exchange has usually completed
        // (phase C, behind the off-path q, k, v work), so every lane reads
        // once first -- one round trip to the L2.  (Early, such reads only
        // load the L2 while the contributions arrive.)
        if (late && have) {
            ld_relaxed_v2_u64(w, v0, v1);
            ld_relaxed_v2_u64(w + 2, v2, v3);
            if (need_ss) vs = ld_relaxed_u64(xbase + b.z);
        }
        if (!late || !__all_sync(0xffffffffu, !have || complete())) {
            // lane 0 waits on the unit's last word (its stage-1 column block
            // is sent after those of the unit's other words): one poller per
            // warp keeps the L2 free for the contributions still arriving.
            // It lets the lanes read once all but kEarlyRead contributions
            // are in, so their round trip overlaps the last ones' arrival
            // (against waiting for all of them: 1.513 -> 1.501 ms per token
            // with 152 contributions; 30 to 48 early measured alike).
            if (lane == 0 && a.z > 0) {
                const unsigned long long s0 = globaltimer_ns();
                const unsigned long long *gw = xbase + b.x + (min(a.z, 4 * a.y) - 1);
                for (int spin = 0; (unsigned)(ld_relaxed_u64(gw) & 0xffull) + kEarlyRead < n_t;
                     ++spin)
                    if ((spin & 15) == 15 && globaltimer_ns() - s0 > kWaitLimitNs) break;
            }
            __syncwarp();
            for (int spin = 0; have; ++spin) {
                ld_relaxed_v2_u64(w, v0, v1);
                ld_relaxed_v2_u64(w + 2, v2, v3);
                if (need_ss) vs = ld_relaxed_u64(xbase + b.z);
                if (complete()) break;
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
            // every lane of the warp leaves together (the sum below is warp-wide)
            if (__any_sync(0xffffffffu, !ok)) {
                ok = 0;
                break;
            }
        }
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (have) {
            const uint2 hb = *reinterpret_cast<const uint2 *>(g_smem + b.y + 8 * lane);
            const float m = (a.w & TAB_MUL) ? (need_ss ? rsqrtf(dec_fix1(vs, iss)) : inv) : 1.f;
            x.x = dec_fix1(v0, it) * half_bits_to_float((uint16_t)(hb.x & 0xffffu)) * m;
            x.y = dec_fix1(v1, it) * half_bits_to_float((uint16_t)(hb.x >> 16)) * m;
            x.z = dec_fix1(v2, it) * half_bits_to_float((uint16_t)(hb.y & 0xffffu)) * m;
            x.w = dec_fix1(v3, it) * half_bits_to_float((uint16_t)(hb.y >> 16)) * m;
        }
        if (b.w >= 0) {
            float zs = (fabsf(x.x) + fabsf(x.y)) + (fabsf(x.z) + fabsf(x.w));
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) zs += __shfl_xor_sync(0xffffffffu, zs, o);
            if (lane == 0) atomicMax(zmax + b.w, __float_as_uint(zs));
        }
        if (lane < a.y) store_table(g_smem + a.x + lane * 128, x, lane);
    }
    return csync_and(ok) != 0;
}

// Bounded wait on an mbarrier phase by every compute thread.
__device__ bool wait_full(unsigned long long *bar, unsigned parity, unsigned *ws_words) {
    int ok = 1;
    if (!mbar_try_wait(bar, parity)) {
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(bar, parity)) {
            __nanosleep(32);
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                record(ws_words, LB_ERR_TIMEOUT);
                ok = 0;
                break;
            }
        }
    }
    return csync_and(ok) != 0;
}


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
    // the exchange-bound constants of phase X of layer l
    __device__ void consts(int X, int l, unsigned long long *b) const {
        copy(P->o.cst[X], P->cst + ((size_t)l * 4 + X) * 2, 32u, b);
    }

    // phase A of layer l (0 <= l <= n_layers): down of layer l-1 on R_c rows,
    // stage 1 of q, k, v of layer l on R_c (absent for l = n_layers).
    __device__ void issue_A(int l) const {
        unsigned long long *b = full + 0;
        const Offsets &o = P->o;
        consts(0, l, b);
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
        consts(1, l, b);
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
        consts(2, l, b);
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
        consts(3, l, b);
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
            // the compute warps hold the buffer for most of a layer: poll it
            // gently, so the wait does not take issue slots and shared-memory
            // bandwidth from them
            for (int spin = 0; !mbar_try_wait(empty + b, parity); ++spin) {
                __nanosleep(128);
                if ((spin & 15) == 15) {
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

template <int C>
__global__ void __launch_bounds__(kST, 1) k_stack(const __grid_constant__ Params P) {
    __shared__ __align__(8) unsigned long long full[4], empty[4];
    __shared__ int s_last;
    __shared__ int s_zs[XR_N][2];  // this CTA's stripe of each exchange region
    // per phase, the largest |z| sum of a poll unit of each bound entry; and
    // the largest per-thread share of the L1 norm of x0 (fp32 bits)
    __shared__ unsigned s_zmax[4][4], s_x0max;
    unsigned *err = P.ws_words + kErrWord;
    if (sticky(P.ws_words)) return;
    if (*reinterpret_cast<const volatile unsigned long long *>(P.ws_words + kPlanWord) != P.plan) {
        if (blockIdx.x == 0 && threadIdx.x == 0) record(P.ws_words, LB_ERR_PLAN);
        return;
    }
    // the partials of a cluster meet in its CTAs' shared memory: a launch
    // that did not form clusters of C CTAs (the per-CTA programs
    // assume them) records an error and touches no other CTA's memory
    if (C > 1 && cluster_size() != (unsigned)C) {
        if (threadIdx.x == 0) record(P.ws_words, LB_ERR_UNSUPPORTED);
        return;
    }
    const int N = gridDim.x, c = blockIdx.x;
    const unsigned n_ctas = (unsigned)N, n_t = P.n_t;
    const unsigned rank = C > 1 ? cluster_rank() : 0u;
    Part s;
    {
        int u0, nu;
        slice_of(P.d >> 5, N, c, C, s.dw0, s.nd);
        slice_of(P.dff >> 5, N, c, C, s.fw0, s.nf);
        slice_of(P.dkv >> 3, N, c, C, u0, nu);
        s.k0 = 8 * u0;
        s.nkv = 8 * nu;
    }
    if (threadIdx.x == 0) {
        for (int b = 0; b < 4; ++b) {
            mbar_init(full + b, 1);
            mbar_init(empty + b, 1);
        }
        for (int b = 0; b < P.o.n_ubar; ++b)
            mbar_init(reinterpret_cast<unsigned long long *>(g_smem + P.o.ubar) + b, 1);
        fence_barrier_init();
        for (int k = 0; k < 16; ++k) s_zmax[k >> 2][k & 3] = 0u;
        s_x0max = 0u;
    }
    if (threadIdx.x < XR_N) {
        const int t = threadIdx.x;
        const int n = t == XR_A ? P.lenA : t == XR_Q ? P.lenQ : t == XR_B ? P.lenB
                    : t == XR_C ? P.lenC : P.lenD;
        const long long w = (long long)n;
        s_zs[threadIdx.x][0] = (int)(c * w / N);
        s_zs[threadIdx.x][1] = (int)((c + 1) * w / N);
    }
    __syncthreads();
    // every CTA of the cluster has initialised its mbarriers before any
    // other may complete a transaction on them
    if (C > 1) cluster_sync_all();
    if (threadIdx.x >= kCT) {
        if (threadIdx.x == kCT) producer(Loader{&P, s, full}, empty, P.ws_words);
    } else {

    // ------------------------------------------------------------ compute warps
    const Offsets &o = P.o;
    {
        const int4 *src = reinterpret_cast<const int4 *>(P.prog) + (size_t)c * (kProgBytes / 16);
        int4 *dst = reinterpret_cast<int4 *>(g_smem + o.prog);
        for (int i = threadIdx.x; i < kProgBytes / 16; i += kCT) dst[i] = src[i];
    }
    const int pg = o.prog;
    const int rows_d = 32 * s.nd, nkv = s.nkv;
    float *res0 = sm_f(o.res0), *res1 = sm_f(o.res1), *yq = sm_f(o.yq);
    float *yk = sm_f(o.yk), *yv = sm_f(o.yv);
    float *ssslot = sm_f(o.ssslot);  // per-unit sums of squares (residual row steps)
    for (int i = threadIdx.x; i < rows_d; i += kCT) {
        res0[i] = bf16_bits_to_float(P.x0[32 * s.dw0 + i]);
        yq[i] = 0.f;
    }
    zero_f(yk, nkv);
    zero_f(yv, nkv);
    for (int i = threadIdx.x; i < kMaxSlots; i += kCT) ssslot[i] = 0.f;
    {
        // ||x0||_1 <= kCT x the largest per-thread share (every CTA alike)
        float a = 0.f;
        for (int i = threadIdx.x; i < P.d; i += kCT) a += fabsf(bf16_bits_to_float(P.x0[i]));
        atomicMax(&s_x0max, __float_as_uint(a));
    }
    csync();
    int nr[7];
#pragma unroll
    for (int k = 0; k < 7; ++k) nr[k] = P.r[k][0] + (P.np[k] > 1 ? P.r[k][1] : 0);
    const int ssA_el = nr[LV], ssC_el = nr[LG] + nr[LU];
    const bool lead = threadIdx.x == 0;
    const float inv_d = 1.f / (float)P.d;
    const int n_tc = (int)n_t, n_cc = (int)n_ctas;
    // Exchange bounds (identical in every CTA).  Ba, Bh: L1 norms of a and
    // h; per exchange the scale of its t (sc*) and mean square (ss*) and the
    // inverses its readers decode with (i*).
    float Ba = (float)kCT * __uint_as_float(s_x0max), Bh = 0.f;
    float2 scA = make_float2(1.f, 1.f), ssA = scA, scB = scA, scC = scA, ssC = scA, scD = scA;
    // phase X's constants and largest unit |z| sums
    auto cst = [&](int X, int k) { return reinterpret_cast<const float4 *>(g_smem + o.cst[X])[k]; };
    auto zm = [&](int X, int j) { return __uint_as_float(s_zmax[X][j]); };
    // the first word of region off in the layer at x
    auto at = [](unsigned long long *x, int off) { return x + off; };
    auto release = [&](int b) {
        csync();
        if (lead) mbar_arrive(empty + b);
    };
    // The lead sends this CTA's share of the mean square (sum / d: the row
    // step's slots added in slot order, zero for a CTA without rows) once
    // its own stage-1 units are out, so the sum is off the critical path;
    // the share's bound is B^2 / d for B the L1 norm of the vector.
    auto send_ss = [&](unsigned long long *p, float2 sc, int step) {
        if (lead) {
            const int n = step_at(pg, step).nslot;
            float q = 0.f;
            for (int i = 0; i < n; ++i) q += ssslot[i];
            send_fix1(p, q * inv_d, sc.x, P.lim_ss, err);
        }
    };
    // Threads 0-3 clear a phase's |z| maxima once every compute thread has
    // read them (after the barrier that follows the row step).
    auto clear_z = [&](int X) {
        if (threadIdx.x < 4) s_zmax[X][threadIdx.x] = 0u;
    };
    // a failed wait leaves the layer loop; the CTA still meets its cluster at
    // the end, so no other CTA stores into its shared memory after it exits
#define FAIL_EXIT() goto done

    for (int l = 0; l < P.n_layers; ++l) {
        unsigned long long *xl = P.xacc + (size_t)l * P.acc_layer;
        unsigned long long *xp = xl - P.acc_layer;  // the previous layer's words
        const unsigned par = (unsigned)(l & 1);

        // ================= phase A: a = h + Down_{l-1}(m) on R_c; stage 1 of q, k, v
        if (!wait_full(full + 0, par, P.ws_words)) FAIL_EXIT();
        if (l > 0) {
            if (!run_poll_tables(pg, A_P2, xp, n_t, n_ctas, 1.f, scD.y, 1.f, s_zmax[0], false,
                                 P.ws_words))
                FAIL_EXIT();
            const float4 c = cst(0, 0);
            Ba = Bh + (c.x * zm(0, 0) + c.y * zm(0, 1));  // ||a|| <= ||h|| + ||Down(m)||
        }
        scA = fix1_scale(cst(0, 1).x * Ba, n_tc);  // |t| <= max|g| ||a||
        ssA = fix1_scale(Ba * Ba * inv_d, n_cc);
        run_rows(pg, A_R, l > 0, true, ssslot);  // a = res0 + Down(m) -> res1; tables
        csync();
        clear_z(0);
        {
            const bool ok1 = run_s1<C>(pg, A_S1, xl, scA.x, P.lim_t, err, o.slot[0], o.ubar0[0],
                                    o.ubar, par, rank, P.ws_words);
            send_ss(xl + P.offA + ssA_el, ssA, A_R);
            if (!csync_and(ok1)) FAIL_EXIT();
        }
        // regions C and Q of the previous layer: every CTA has passed the
        // poll that read them (exchange D, polled above, counts all CTAs)
        if (l > 0) {
            zero_stripe(at(xp, P.offC), s_zs[XR_C]);
            zero_stripe(at(xp, P.offQ), s_zs[XR_Q]);
        }
        release(0);

        // ================= phase B: v rows for attention, stage 1 of o; then q, k, v out
        if (!wait_full(full + 1, par, P.ws_words)) FAIL_EXIT();
        // tables of v (critical) and of q, k (region Q, sent with region A)
        if (!run_poll_tables(pg, B_P2, xl, n_t, n_ctas, 1.f, scA.y, ssA.y, s_zmax[1], false,
                             P.ws_words))
            FAIL_EXIT();
        {
            // the attention rows repeat v: ||attn|| <= grp ||v|| (grp in c)
            const float4 c = cst(1, 0);
            scB = fix1_scale(cst(1, 1).x * (c.x * zm(1, 0) + c.y * zm(1, 1)), n_tc);
        }
        run_rows(pg, B_R, true, true, ssslot);  // v on the attention rows; tables of o
        csync();
        clear_z(1);
        if (!csync_and(run_s1<C>(pg, B_S1, xl, scB.x, P.lim_t, err, o.slot[1], o.ubar0[1], o.ubar,
                              par, rank, P.ws_words)))
            FAIL_EXIT();
        if (l > 0) zero_stripe(at(xp, P.offD), s_zs[XR_D]);  // read by phase A's poll
        // ---- off the critical path, while exchange B is in flight: q on R_c,
        //      k and v on K_c (their tables were built with v's)
        run_s2(pg, B_S2QKV);  // -> yq, yk, yv
        csync();
        for (int i = threadIdx.x; i < nkv; i += kCT) {
            if (P.kv_out) {
                P.kv_out[((size_t)l * 2 + 0) * P.dkv + s.k0 + i] = yk[i];
                P.kv_out[((size_t)l * 2 + 1) * P.dkv + s.k0 + i] = yv[i];
            }
            yk[i] = yv[i] = 0.f;
        }
        for (int i = threadIdx.x; i < rows_d; i += kCT) {
            if (P.q_out) P.q_out[(size_t)l * P.d + 32 * s.dw0 + i] = yq[i];
            yq[i] = 0.f;
        }
        release(1);

        // ================= phase C: h = a + O(attn) on R_c; stage 1 of gate, up
        if (!wait_full(full + 2, par, P.ws_words)) FAIL_EXIT();
        if (!run_poll_tables(pg, C_P2, xl, n_t, n_ctas, 1.f, scB.y, 1.f, s_zmax[2], true,
                             P.ws_words))
            FAIL_EXIT();
        {
            const float4 c = cst(2, 0);
            Bh = Ba + (c.x * zm(2, 0) + c.y * zm(2, 1));  // ||h|| <= ||a|| + ||O(attn)||
            scC = fix1_scale(cst(2, 1).x * Bh, n_tc);
            ssC = fix1_scale(Bh * Bh * inv_d, n_cc);
        }
        run_rows(pg, C_R, true, true, ssslot);  // h = res1 + O(attn) -> res0; tables
        csync();
        clear_z(2);
        {
            const bool ok1 = run_s1<C>(pg, C_S1, xl, scC.x, P.lim_t, err, o.slot[2], o.ubar0[2],
                                    o.ubar, par, rank, P.ws_words);
            send_ss(xl + P.offC + ssC_el, ssC, C_R);
            if (!csync_and(ok1)) FAIL_EXIT();
        }
        zero_stripe(at(xl, P.offA), s_zs[XR_A]);  // read by phase B's poll
        release(2);

        // ================= phase D: m = silu(gate) * up on F_c; stage 1 of down
        if (!wait_full(full + 3, par, P.ws_words)) FAIL_EXIT();
        if (!run_poll_tables(pg, D_P2, xl, n_t, n_ctas, 1.f, scC.y, ssC.y, s_zmax[3], false,
                             P.ws_words))
            FAIL_EXIT();
        {
            // ||silu(G) * U|| <= max|G| ||U||
            const float4 c = cst(3, 0);
            const float Bm = (c.x * zm(3, 0) + c.y * zm(3, 1)) * (c.z * zm(3, 2) + c.w * zm(3, 3));
            scD = fix1_scale(cst(3, 1).x * Bm, n_tc);
        }
        run_rows(pg, D_R, true, true, ssslot);  // m = silu(gate) * up; tables of down
        csync();
        clear_z(3);
        if (!csync_and(run_s1<C>(pg, D_S1, xl, scD.x, P.lim_t, err, o.slot[3], o.ubar0[3], o.ubar,
                              par, rank, P.ws_words)))
            FAIL_EXIT();
        zero_stripe(at(xl, P.offB), s_zs[XR_B]);  // read by phase C's poll
        release(3);
    }

    // ================= final: out = h + Down_{L-1}(m) on R_c
    {
        const int l = P.n_layers;
        unsigned long long *xp = P.xacc + (size_t)(l - 1) * P.acc_layer;
        if (!wait_full(full + 0, (unsigned)(l & 1), P.ws_words)) FAIL_EXIT();
        if (!run_poll_tables(pg, A_P2, xp, n_t, n_ctas, 1.f, scD.y, 1.f, s_zmax[0], false,
                             P.ws_words))
            FAIL_EXIT();
        zero_stripe(at(xp, P.offC), s_zs[XR_C]);
        zero_stripe(at(xp, P.offQ), s_zs[XR_Q]);
        run_rows(pg, A_R, true, false, ssslot);  // a = res0 + Down(m) -> res1
        csync();
        for (int i = threadIdx.x; i < rows_d; i += kCT) P.out[32 * s.dw0 + i] = res1[i];
        // The last CTA to finish has seen every other CTA's reads of the final
        // region: it clears that region and the counters for the next launch.
        if (lead) {
            __threadfence();
            s_last = atomicAdd(P.ws_words + kDoneWord, 1u) == n_ctas - 1;
        }
        csync();
        if (s_last) {
            __threadfence();
            for (int i = threadIdx.x; i < P.lenD; i += kCT)
                at(xp, P.offD)[i] = 0ull;
            if (lead) P.ws_words[kDoneWord] = 0u;
        }
    }
    }  // compute warps
done:
    // no CTA leaves while another CTA of its cluster may still store into its
    // shared memory (every wait above is bounded, so every thread gets here)
    if (C > 1) cluster_sync_all();
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

// Exchange elements (one word each) per layer: A = t of v + ss(a); Q = t of
// q, k (read off the critical path); B = t of o; C = t of gate, up + ss(h);
// D = t of down; each region padded to 32 elements.
struct XLayout {
    int acc_layer, offA, offQ, offB, offC, offD, lenA, lenQ, lenB, lenC, lenD;
};

XLayout xlayout(const lb_linear *lin) {
    XLayout X{};
    X.lenA = rsum(lin[LV]) + 1;
    X.lenQ = rsum(lin[LQ]) + rsum(lin[LK]);
    X.lenB = rsum(lin[LO]);
    X.lenC = rsum(lin[LG]) + rsum(lin[LU]) + 1;
    X.lenD = rsum(lin[LD]);
    X.offA = 0;
    X.offQ = X.offA + up(X.lenA, 32);
    X.offB = X.offQ + up(X.lenQ, 32);
    X.offC = X.offB + up(X.lenB, 32);
    X.offD = X.offC + up(X.lenC, 32);
    X.acc_layer = X.offD + up(X.lenD, 32);
    return X;
}

size_t desc_bytes_for(int n_layers) {
    return ((size_t)7 * n_layers * sizeof(LinDesc) + 255) & ~(size_t)255;
}

// One exchange word per element.
size_t xacc_bytes(const XLayout &X, int n_layers) {
    return ((size_t)n_layers * X.acc_layer * sizeof(unsigned long long) + 255) & ~(size_t)255;
}

// Two float4 per phase and layer, layers 0..n_layers.
size_t cst_bytes(int n_layers) { return ((size_t)(n_layers + 1) * 4 * 32 + 255) & ~(size_t)255; }

// 2^55 / n rounded down: n contributions below it sum to less than 2^55.
float fix1_limit(int n) {
    float l = (float)(std::ldexp(1.0, 55) / n);
    while ((double)l * n >= std::ldexp(1.0, 55)) l = std::nextafter(l, 0.f);
    return l;
}

// ---------------------------------------------------------------- bound constants

constexpr int kConstThreads = 1024;

// Block-wide sum and max of |v| over n fp16 values.  Each thread adds its
// k = ceil(n / 1024) terms in fp32 (relative error below k 2^-24: 2^-14 for
// the 70B shapes' n <= 28672), the block adds the threads' sums in fp64, and
// the callers scale the total by (1 + 2^-12) and round it up.  The bound
// only chooses the exchange's scale, which leaves a factor of 2 between the
// bound and the largest contribution it accepts.
__device__ void abs_stats(const uint16_t *v, int n, double &sum, float &mx) {
    __shared__ double s_sum[kConstThreads / 32];
    __shared__ float s_max[kConstThreads / 32];
    float a = 0.f, m = 0.f;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const float x = fabsf(half_bits_to_float(v[i]));
        a += x;
        m = fmaxf(m, x);
    }
    double ad = (double)a;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        ad += __shfl_xor_sync(0xffffffffu, ad, o);
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    }
    __syncthreads();  // the previous call's readers are done
    if ((threadIdx.x & 31) == 0) {
        s_sum[threadIdx.x >> 5] = ad;
        s_max[threadIdx.x >> 5] = m;
    }
    __syncthreads();
    sum = 0.0;
    mx = 0.f;
    for (int w = 0; w < kConstThreads / 32; ++w) {
        sum += s_sum[w];
        mx = fmaxf(mx, s_max[w]);
    }
}

// Constants of the exchange bounds, block l for layer l (0..n_layers).  A
// poll unit covers 128 values of t, so a path of rank r has nu = ceil(r /
// 128) units and sum |z| <= nu x the largest unit sum zmax.  Per phase
// (c[0..3]; then max|g| of the linears whose stage 1 the phase sends):
//   A: ||h_down(l-1),p||_1 nu (p = 0, 1)                  ; q, k, v of layer l
//   B: grp ||h_v,p||_1 nu (attention repeats v grp times) ; o
//   C: ||h_o,p||_1 nu                                     ; gate, up
//   D: max|h_gate,p| nu, ||h_up,p||_1 nu                  ; down
// (sums in fp64, rounded up to fp32).
__global__ void __launch_bounds__(kConstThreads) k_stack_consts(const LinDesc *lin, int n_layers,
                                                                int grp, float4 *cst) {
    const int l = blockIdx.x;
    float c[4][4] = {}, gmax[4] = {};
    auto nu = [](int r) { return (double)((r + 127) / 128); };
    auto hsum = [&](const LinDesc &L, int p, double mul) {
        double s;
        float m;
        abs_stats(L.h[p], L.d_out, s, m);
        return __double2float_ru(s * (1.0 + 0x1p-12) * mul * nu(L.r[p]));
    };
    auto hmax = [&](const LinDesc &L, int p) {
        double s;
        float m;
        abs_stats(L.h[p], L.d_out, s, m);
        return __double2float_ru((double)m * nu(L.r[p]));
    };
    auto gm = [&](const LinDesc &L) {
        float r = 0.f;
        for (int p = 0; p < L.n_paths; ++p) {
            double s;
            float m;
            abs_stats(L.g[p], L.d_in, s, m);
            r = fmaxf(r, m);
        }
        return r;
    };
    if (l > 0) {
        const LinDesc &D = lin[7 * (l - 1) + LD];
        for (int p = 0; p < D.n_paths; ++p) c[0][p] = hsum(D, p, 1.0);
    }
    if (l < n_layers) {
        const LinDesc *L = lin + 7 * l;
        gmax[0] = fmaxf(gm(L[LQ]), fmaxf(gm(L[LK]), gm(L[LV])));
        for (int p = 0; p < L[LV].n_paths; ++p) c[1][p] = hsum(L[LV], p, (double)grp);
        gmax[1] = gm(L[LO]);
        for (int p = 0; p < L[LO].n_paths; ++p) c[2][p] = hsum(L[LO], p, 1.0);
        gmax[2] = fmaxf(gm(L[LG]), gm(L[LU]));
        for (int p = 0; p < L[LG].n_paths; ++p) c[3][p] = hmax(L[LG], p);
        for (int p = 0; p < L[LU].n_paths; ++p) c[3][2 + p] = hsum(L[LU], p, 1.0);
        gmax[3] = gm(L[LD]);
    }
    if (threadIdx.x < 4) {
        const int X = threadIdx.x;
        cst[((size_t)l * 4 + X) * 2 + 0] = make_float4(c[X][0], c[X][1], c[X][2], c[X][3]);
        cst[((size_t)l * 4 + X) * 2 + 1] = make_float4(gmax[X], 0.f, 0.f, 0.f);
    }
}

// Stage-1 units (32-column blocks over every path) of linears k0..k1.
int s1_units(const lb_linear *lin, int k0, int k1) {
    int n = 0;
    for (int k = k0; k <= k1; ++k)
        for (int p = 0; p < lin[k].n_paths; ++p) n += (lin[k].path[p].r + 31) / 32;
    return n;
}

// Shared-memory plan from the largest slices any CTA gets.
struct SmemPlan {
    Offsets o;
    int bytes;
};

SmemPlan smem_plan(const lb_linear *lin, const StackShape &sh, int N, int C) {
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
    o.cst[0] = take(32);
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
    o.cst[1] = take(32);
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
    o.cst[2] = take(32);
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
    o.cst[3] = take(32);
    // nibble tables (1 KB per 32 values): the largest set a phase holds at once
    auto utab = [&](int k, int p0, int p1) {
        int b = 0;
        for (int p = p0; p < std::min(p1, lin[k].n_paths); ++p) b += R(k, p) * 1024;
        return b;
    };
    auto vtab = [&](int k, int nw) { return lin[k].n_paths * nw * 1024; };
    int t2 = utab(LD, 0, 2);
    t2 = std::max(t2, utab(LV, 0, 2) + utab(LQ, 0, 2) + utab(LK, 0, 2));
    t2 = std::max(t2, utab(LO, 0, 2));
    t2 = std::max(t2, utab(LG, 0, 2) + utab(LU, 0, 2));
    int t1 = vtab(LQ, nd) + vtab(LK, nd) + vtab(LV, nd);
    t1 = std::max(t1, vtab(LO, nd));
    t1 = std::max(t1, vtab(LG, nd) + vtab(LU, nd));
    t1 = std::max(t1, vtab(LD, nf));
    at = up(at, 1024);
    o.t2 = at;
    at += up(t2, 1024);
    o.t1 = at;
    at += up(t1, 1024);
    o.res0 = take(4 * 32 * nd);
    o.res1 = take(4 * 32 * nd);
    o.yq = take(4 * 32 * nd);
    o.yk = take(4 * nkv);
    o.yv = take(4 * nkv);
    o.ssslot = take(4 * kMaxSlots);
    o.prog = take(kProgBytes);
    // cluster reduction: per phase, the receive slots and mbarriers of the
    // ceil(units / C) stage-1 units a rank owns at most
    const int units[4] = {s1_units(lin, LQ, LV), s1_units(lin, LO, LO), s1_units(lin, LG, LU),
                          s1_units(lin, LD, LD)};
    o.n_ubar = 0;
    for (int ph = 0; ph < 4; ++ph) {
        const int owned = C > 1 ? (units[ph] + C - 1) / C : 0;
        o.slot[ph] = take(owned * C * 128);
        o.ubar0[ph] = o.n_ubar;
        o.n_ubar += owned;
    }
    at = up(at, 8);
    o.ubar = take(8 * o.n_ubar);
    S.bytes = up(at, 128);
    return S;
}

// ---------------------------------------------------------------- the program

// e0, ss_el: exchange word indices within a layer (ss_el < 0: none); job:
// the bound entry of the unit's |z| sums (-1: none)
Item ptab(int tb, int n_tab, int n_vals, int mode, int e0, int scale, int ss_el, int job) {
    return Item{{tb, n_tab, n_vals, mode, e0, scale, ss_el, job}};
}

struct Costed {
    Item it;
    double cost;
};

// Longest-processing-time assignment of units to the compute warps; returns
// the units grouped by warp (warp-start offsets in wo) and the makespan.
// Longest-processing-time assignment of units to warps [w0, w1): appends
// to the per-warp lists, returns the makespan.
using PerWarp = std::vector<Item>[kCW];
double lpt_into(const std::vector<Costed> &us, int w0, int w1, PerWarp &per) {
    std::vector<int> idx(us.size());
    for (size_t i = 0; i < us.size(); ++i) idx[i] = (int)i;
    std::stable_sort(idx.begin(), idx.end(),
                     [&](int a, int b) { return us[a].cost > us[b].cost; });
    double load[kCW] = {};
    for (int i : idx) {
        int w = w0;
        for (int k = w0 + 1; k < w1; ++k)
            if (load[k] < load[w]) w = k;
        load[w] += us[i].cost;
        per[w].push_back(us[i].it);
    }
    double mk = 0;
    for (int w = w0; w < w1; ++w) mk = std::max(mk, load[w]);
    return mk;
}

// The same over all compute warps, grouped by warp (warp-start offsets in wo).
double lpt(const std::vector<Costed> &us, std::vector<Item> &out, int (&wo)[kCW + 1]) {
    PerWarp per;
    const double mk = lpt_into(us, 0, kCW, per);
    out.clear();
    wo[0] = 0;
    for (int w = 0; w < kCW; ++w) {
        out.insert(out.end(), per[w].begin(), per[w].end());
        wo[w + 1] = (int)out.size();
    }
    return mk;
}

struct S2Job {
    int U, h, R, rows, tb, out;
};
// A row-unit segment at row 0: U rows (R words each, from word 0 of the
// segment), nw words, the stage-2 tables of word 0 and h.  A segment without
// words keeps its partner's offsets (its reads are masked).
struct Seg {
    int U, R, nw, tb, h;
};
// A stage-1 table job of a row step: its table set (128 bytes per 4 rows) and
// its g, at row 0.
struct TabJob {
    int tb, g;
};
struct S1Job {
    int V, r, nw, tb, dst;
};

struct ProgBuild {
    Step step[N_STEPS] = {};
    std::vector<Item> items;
    int min_lnr = kRowMinLnr;  // smallest log2 rows per row unit (4: only the two halves)

    void place(int s, const std::vector<Item> &grouped, const int (&wo)[kCW + 1]) {
        step[s].first = (int)items.size();
        for (int w = 0; w <= kCW; ++w) step[s].wo[w] = wo[w];
        items.insert(items.end(), grouped.begin(), grouped.end());
    }
    void place(int s, const PerWarp &per) {
        step[s].first = (int)items.size();
        step[s].wo[0] = 0;
        for (int w = 0; w < kCW; ++w) {
            items.insert(items.end(), per[w].begin(), per[w].end());
            step[s].wo[w + 1] = (int)items.size() - step[s].first;
        }
    }
    // Row units of a stage-2 step (see run_rows): the work of lanes 0-15 and
    // of lanes 16-31 as segments given at row 0 (half[0], half[1]), the table
    // jobs of the rows, the mode and the residual buffers.  The rows per unit
    // (16, 8 or 4: 2, 4 or 8 lane groups, each half's words split evenly
    // over its groups) minimise the estimated makespan over the warps (in
    // sign words per lane: a fixed cost per unit, the longest group's words,
    // the mode and the table jobs); units go to the warps longest first.
    // Returns false when a residual step needs more than kMaxSlots units.
    bool rows(int s, const std::vector<Seg> (&half)[2], const std::vector<TabJob> &jobs,
              int mode, int res_in, int res_out, int nrows) {
        struct Unit {
            std::vector<Item> it;
            double cost;
        };
        std::vector<Unit> best;
        double best_mk = 1e300;
        for (int lnr = 4; lnr >= min_lnr; --lnr) {
            const int nr = 1 << lnr, G = 32 >> lnr, gh = G / 2;
            // each half's words in gh runs: group g of half h covers words
            // [g W / gh, (g + 1) W / gh) of the half's segments laid end to end
            std::vector<std::vector<Seg>> grp(G);
            int maxw = 0;
            for (int h = 0; h < 2; ++h) {
                int W = 0;
                for (const Seg &g : half[h]) W += g.nw;
                for (int g = 0; g < gh; ++g) {
                    const int w0 = (int)((long long)g * W / gh), w1 = (int)((long long)(g + 1) * W / gh);
                    maxw = std::max(maxw, w1 - w0);
                    int base = 0;
                    for (const Seg &sg : half[h]) {
                        const int a = std::max(w0, base), b = std::min(w1, base + sg.nw);
                        if (a < b)
                            grp[h * gh + g].push_back({sg.U + 4 * (a - base), sg.R, b - a,
                                                       sg.tb + 1024 * (a - base), sg.h});
                        base += sg.nw;
                    }
                }
            }
            size_t nseg = 1;
            for (const auto &g : grp) nseg = std::max(nseg, g.size());
            // pad with segments without words (their reads are never made)
            for (int g = 0; g < G; ++g) {
                const Seg pad = grp[g].empty() ? half[g / gh].front() : grp[g].front();
                while (grp[g].size() < nseg) grp[g].push_back({pad.U, pad.R, 0, pad.tb, pad.h});
            }
            const int ntab = (int)jobs.size() * (nr / 4);
            const double cost = 3.0 + maxw + 0.5 * (double)(nseg - 1) +
                                (mode == ROW_RES ? 1.0 : 0.5) + (ntab > 0 ? 2.0 : 0.0) +
                                (ntab > 32 ? 2.0 : 0.0);
            std::vector<Unit> us;
            int slot = 0;
            for (int r0 = 0; r0 < nrows; r0 += nr, ++slot) {
                Unit U{{}, cost};
                U.it.push_back(Item{{(int)nseg, (int)jobs.size(), mode | (lnr << 8),
                                     std::min(nr, nrows - r0), res_in + 4 * r0, res_out + 4 * r0,
                                     slot, 0}});
                for (int g = 0; g < G; ++g)
                    for (const Seg &sg : grp[g])
                        U.it.push_back(Item{{sg.U + 4 * r0 * sg.R, sg.R, sg.nw, sg.tb,
                                             sg.h + 2 * r0, 0, 0, 0}});
                for (const TabJob &J : jobs)
                    U.it.push_back(Item{{J.tb + 128 * (r0 / 4), J.g + 2 * r0, 0, 0, 0, 0, 0, 0}});
                us.push_back(U);
            }
            const double mk = std::ceil((double)us.size() / kCW) * cost;
            if (mk < best_mk - 1e-9) {
                best_mk = mk;
                best = us;
            }
        }
        if (mode == ROW_RES && (int)best.size() > kMaxSlots) return false;
        PerWarp per;
        double load[kCW] = {};
        for (const Unit &U : best) {
            int w = 0;
            for (int k = 1; k < kCW; ++k)
                if (load[k] < load[w]) w = k;
            load[w] += U.cost;
            per[w].insert(per[w].end(), U.it.begin(), U.it.end());
        }
        place(s, per);
        step[s].nslot = mode == ROW_RES ? (int)best.size() : 0;
        return true;
    }
    // The two halves of one linear summed over its paths: path 0 beside
    // path 1, or one path's words split between the halves.
    static void halves_of(const std::vector<Seg> &g, std::vector<Seg> (&half)[2]) {
        half[0].clear();
        half[1].clear();
        if (g.size() > 1) {
            half[0].push_back(g[0]);
            half[1].push_back(g[1]);
            return;
        }
        Seg a = g[0], b = g[0];
        a.nw = (g[0].nw + 1) / 2;
        b.nw = g[0].nw - a.nw;
        b.U += 4 * a.nw;
        b.tb += 1024 * a.nw;
        half[0].push_back(a);
        if (b.nw > 0) half[1].push_back(b);
        else half[1].push_back({a.U, a.R, 0, a.tb, a.h});
    }
    // Poll-table units: the same split, word indices instead of offsets.
    void ptables(int s, const std::vector<Item> &jobs) {
        std::vector<Costed> us;
        for (const Item &J : jobs) {
            const int nt = J.f[1];
            for (int t0 = 0; t0 < nt; t0 += 32)
                us.push_back({Item{{J.f[0] + 128 * t0, std::min(32, nt - t0), J.f[2] - 4 * t0,
                                    J.f[3], J.f[4] + 4 * t0, J.f[5] + 8 * t0, J.f[6], J.f[7]}},
                              1.0 + std::min(32, nt - t0) / 32.0});
        }
        std::vector<Item> g;
        int wo[kCW + 1];
        lpt(us, g, wo);
        place(s, g, wo);
    }
    // 32-row blocks x runs of words, the run length chosen to balance warps
    // (cost of a unit: its words plus a fixed overhead).
    void s2(int s, const std::vector<S2Job> &jobs) {
        int maxR = 1;
        for (const S2Job &J : jobs) maxR = std::max(maxR, J.R);
        std::vector<Item> best;
        int best_wo[kCW + 1] = {};
        double best_mk = 1e300;
        for (int run = 1; run <= maxR; ++run) {
            std::vector<Costed> us;
            for (const S2Job &J : jobs)
                for (int r0 = 0; r0 < J.rows; r0 += 32)
                    for (int w0 = 0; w0 < J.R; w0 += run) {
                        const int nw = std::min(run, J.R - w0);
                        us.push_back({Item{{J.U + (r0 * J.R + w0) * 4, J.R, nw, J.tb + w0 * 1024,
                                            J.h + 2 * r0, J.out + 4 * r0,
                                            std::min(32, J.rows - r0), 0}},
                                      nw + 1.5});
                    }
            if (us.size() > 160 && run < maxR) continue;
            std::vector<Item> g;
            int wo[kCW + 1];
            const double mk = lpt(us, g, wo);
            if (mk < best_mk - 1e-9) {
                best_mk = mk;
                best = g;
                std::copy(wo, wo + kCW + 1, best_wo);
            }
        }
        place(s, best, best_wo);
    }
    // 32-column blocks over the whole input slice.  Unit g of the phase
    // belongs to cluster rank g % C (its receive slot there: g / C); each
    // warp runs the units its CTA (rank `rank`) does not own
    // first, so their partials are on their way before it waits for its own.
    int C = 1;  // CTAs per cluster
    void s1(int s, const std::vector<S1Job> &jobs, int rank) {
        std::vector<Costed> us;
        int g = 0;
        for (const S1Job &J : jobs)
            for (int c0 = 0; c0 < J.r; c0 += 32, ++g)
                us.push_back({Item{{J.V + 4 * c0, J.r, J.nw, J.tb, J.dst + c0,
                                    std::min(32, J.r - c0), g % C, g / C}},
                              J.nw + 1.0});
        std::vector<Item> grouped;
        int wo[kCW + 1];
        lpt(us, grouped, wo);
        for (int w = 0; w < kCW; ++w)
            std::stable_partition(grouped.begin() + wo[w], grouped.begin() + wo[w + 1],
                                  [rank](const Item &it) { return it.f[6] != rank; });
        place(s, grouped, wo);
    }
};

// The program of CTA c (kProgBytes, zero-padded); false when it does not fit.
// Row units of 8 or 4 rows take more records: a program that does not fit
// with them is built again with 16-row units only.
bool build_program_at(const lb_linear *lin, const StackShape &sh, int N, int C, int c,
                      const Offsets &o, const XLayout &X, int min_lnr,
                      std::vector<int> &prog_out) {
    int dw0, nd, fw0, nf, k0u, nku;
    slice_of(sh.d / 32, N, c, C, dw0, nd);
    slice_of(sh.dff / 32, N, c, C, fw0, nf);
    slice_of(sh.dkv / 8, N, c, C, k0u, nku);
    const int nkv = 8 * nku;
    const int rows_d = 32 * nd, rows_f = 32 * nf;
    auto np = [&](int k) { return lin[k].n_paths; };
    auto rk = [&](int k, int p) { return lin[k].path[p].r; };
    auto Rk = [&](int k, int p) { return (lin[k].path[p].r + 31) / 32; };
    ProgBuild B;
    B.min_lnr = min_lnr;
    B.C = C;
    std::vector<Item> T;
    std::vector<S2Job> U;
    std::vector<S1Job> V;
    auto flush_p = [&](int s) {
        B.ptables(s, T);
        T.clear();
    };
    auto flush_u = [&](int s) {
        B.s2(s, U);
        U.clear();
    };
    const int rank = c % C;  // cluster rank of CTA c (1-D clusters of C)
    auto flush_v = [&](int s) {
        B.s1(s, V, rank);
        V.clear();
    };
    std::vector<Seg> hv[2];
    // phase A: stage 2 of down (previous layer) in row units, a = res0 +
    // Down(m) written to res1, the stage-1 tables of q, k, v; stage 1 of q, k, v
    {
        int tb = o.t2, off = X.offD;  // words of the previous layer
        std::vector<Seg> g;
        for (int p = 0; p < np(LD); ++p) {
            T.push_back(ptab(tb, 8 * Rk(LD, p), rk(LD, p), TAB_PLAIN, off, o.a_ld[p], -1, p));
            g.push_back({o.a_Ud[p], Rk(LD, p), Rk(LD, p), tb, o.a_hd[p]});
            tb += Rk(LD, p) * 1024;
            off += rk(LD, p);
        }
        flush_p(A_P2);
        // q, k -> region Q; v -> region A
        std::vector<TabJob> tj;
        int tb1 = o.t1, dq = X.offQ, dv = X.offA;
        for (int k = 0; k < 3; ++k)
            for (int p = 0; p < np(k); ++p) {
                tj.push_back({tb1, o.a_g[k][p]});
                int &dst = k == LV ? dv : dq;
                V.push_back({o.a_V[k][p], rk(k, p), nd, tb1, dst});
                tb1 += nd * 1024;
                dst += rk(k, p);
            }
        ProgBuild::halves_of(g, hv);
        if (!B.rows(A_R, hv, tj, ROW_RES, o.res0, o.res1, rows_d)) return false;
        flush_v(A_S1);
    }
    // phase B: tables of v, q, k (scaled by the rms factor of a); v on the
    // attention rows of R_c in row units with the tables of o; stage 1 of o;
    // then q -> yq, k -> yk and v on K_c -> yv
    {
        const int ssA = X.offA + rsum(lin[LV]);
        int tb = o.t2, tbv[2] = {0, 0}, off = X.offA;
        std::vector<Seg> g;
        for (int p = 0; p < np(LV); ++p) {
            T.push_back(ptab(tb, 8 * Rk(LV, p), rk(LV, p), TAB_PLAIN | TAB_MUL, off, o.b_lv[p],
                             ssA, p));
            g.push_back({o.b_Uat[p], Rk(LV, p), Rk(LV, p), tb, o.b_hat[p]});
            tbv[p] = tb;
            tb += Rk(LV, p) * 1024;
            off += rk(LV, p);
        }
        std::vector<S2Job> Uqkv;
        off = X.offQ;
        for (int p = 0; p < np(LQ); ++p) {
            T.push_back(ptab(tb, 8 * Rk(LQ, p), rk(LQ, p), TAB_PLAIN | TAB_MUL, off, o.b_lq[p],
                             ssA, -1));
            Uqkv.push_back({o.b_Uq[p], o.b_hq[p], Rk(LQ, p), rows_d, tb, o.yq});
            tb += Rk(LQ, p) * 1024;
            off += rk(LQ, p);
        }
        for (int p = 0; p < np(LK); ++p) {
            T.push_back(ptab(tb, 8 * Rk(LK, p), rk(LK, p), TAB_PLAIN | TAB_MUL, off, o.b_lk[p],
                             ssA, -1));
            Uqkv.push_back({o.b_Uk[p], o.b_hk[p], Rk(LK, p), nkv, tb, o.yk});
            tb += Rk(LK, p) * 1024;
            off += rk(LK, p);
        }
        for (int p = 0; p < np(LV); ++p)
            Uqkv.push_back({o.b_Uvk[p], o.b_hvk[p], Rk(LV, p), nkv, tbv[p], o.yv});
        flush_p(B_P2);
        std::vector<TabJob> tj;
        int tb1 = o.t1, dst = X.offB;
        for (int p = 0; p < np(LO); ++p) {
            tj.push_back({tb1, o.b_go[p]});
            V.push_back({o.b_Vo[p], rk(LO, p), nd, tb1, dst});
            tb1 += nd * 1024;
            dst += rk(LO, p);
        }
        ProgBuild::halves_of(g, hv);
        B.rows(B_R, hv, tj, ROW_SUM, 0, 0, rows_d);
        flush_v(B_S1);
        U = Uqkv;
        flush_u(B_S2QKV);
    }
    // phase C: stage 2 of o in row units, h = res1 + O(attn) written to res0,
    // the tables of gate, up; stage 1 of gate, up
    {
        int tb = o.t2, off = X.offB;
        std::vector<Seg> g;
        for (int p = 0; p < np(LO); ++p) {
            T.push_back(ptab(tb, 8 * Rk(LO, p), rk(LO, p), TAB_PLAIN, off, o.c_lo[p], -1, p));
            g.push_back({o.c_Uo[p], Rk(LO, p), Rk(LO, p), tb, o.c_ho[p]});
            tb += Rk(LO, p) * 1024;
            off += rk(LO, p);
        }
        flush_p(C_P2);
        std::vector<TabJob> tj;
        int tb1 = o.t1, dst = X.offC;
        for (int k = LG; k <= LU; ++k)
            for (int p = 0; p < np(k); ++p) {
                tj.push_back({tb1, k == LG ? o.c_gg[p] : o.c_gu[p]});
                V.push_back({k == LG ? o.c_Vg[p] : o.c_Vu[p], rk(k, p), nd, tb1, dst});
                tb1 += nd * 1024;
                dst += rk(k, p);
            }
        ProgBuild::halves_of(g, hv);
        if (!B.rows(C_R, hv, tj, ROW_RES, o.res1, o.res0, rows_d)) return false;
        flush_v(C_S1);
    }
    // phase D: stage 2 of gate (lanes 0-15) and up (lanes 16-31) in row
    // units, m = silu(gate) * up, the tables of down; stage 1 of down
    {
        const int ssC = X.offC + rsum(lin[LG]) + rsum(lin[LU]);
        int tb = o.t2, off = X.offC;
        std::vector<Seg> gs[2];
        for (int k = LG; k <= LU; ++k)
            for (int p = 0; p < np(k); ++p) {
                T.push_back(ptab(tb, 8 * Rk(k, p), rk(k, p), TAB_PLAIN | TAB_MUL, off,
                                 k == LG ? o.d_lg[p] : o.d_lu[p], ssC, 2 * (k - LG) + p));
                gs[k - LG].push_back({k == LG ? o.d_Ug[p] : o.d_Uu[p], Rk(k, p), Rk(k, p), tb,
                                      k == LG ? o.d_hg[p] : o.d_hu[p]});
                tb += Rk(k, p) * 1024;
                off += rk(k, p);
            }
        flush_p(D_P2);
        std::vector<TabJob> tj;
        int tb1 = o.t1, dst = X.offD;
        for (int p = 0; p < np(LD); ++p) {
            tj.push_back({tb1, o.d_gd[p]});
            V.push_back({o.d_Vd[p], rk(LD, p), nf, tb1, dst});
            tb1 += nf * 1024;
            dst += rk(LD, p);
        }
        B.rows(D_R, gs, tj, ROW_SILU, 0, 0, rows_f);
        flush_v(D_S1);
    }
    if ((int)B.items.size() > kMaxItems) return false;
    prog_out.assign(kProgBytes / 4, 0);
    std::memcpy(prog_out.data(), B.step, sizeof(B.step));
    std::memcpy(prog_out.data() + kStepBytes / 4, B.items.data(), B.items.size() * sizeof(Item));
    return true;
}

bool build_program(const lb_linear *lin, const StackShape &sh, int N, int C, int c,
                   const Offsets &o, const XLayout &X, std::vector<int> &prog_out) {
    return build_program_at(lin, sh, N, C, c, o, X, kRowMinLnr, prog_out) ||
           build_program_at(lin, sh, N, C, c, o, X, 4, prog_out);
}

bool build_programs(const lb_linear *lin, const StackShape &sh, int N, int C,
                    std::vector<int> &all) {
    const SmemPlan S = smem_plan(lin, sh, N, C);
    const XLayout X = xlayout(lin);
    all.assign((size_t)N * (kProgBytes / 4), 0);
    std::vector<int> one;
    for (int c = 0; c < N; ++c) {
        if (!build_program(lin, sh, N, C, c, S.o, X, one)) return false;
        std::copy(one.begin(), one.end(), all.begin() + (size_t)c * (kProgBytes / 4));
    }
    return true;
}

bool smem_fits(const lb_linear *lin, const StackShape &sh, int num_sms, int C) {
    const SmemPlan S = smem_plan(lin, sh, num_sms, C);
    int max_optin = 0, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess)
        return false;
    return S.bytes + 1024 <= max_optin;
}

bool shapes_ok(const lb_linear *lin, const StackShape &sh, int num_sms, int C) {
    if (C < 1 || C > kMaxCluster || num_sms % C != 0) return false;
    for (int k = 0; k < 7; ++k)
        for (int p = 0; p < lin[k].n_paths; ++p)
            if (lin[k].path[p].r % 8 != 0) return false;
    return sh.head_dim % 32 == 0 && sh.dkv % 8 == 0 && num_sms >= 1 && num_sms <= kMaxCtas;
}

}  // namespace

static_assert(sizeof(LinDesc) % sizeof(uint32_t) == 0, "descriptor is copied as words");

// Workspace after the header: descriptors, exchange words, bound constants,
// programs.
size_t stack_ws_bytes_after_header(const lb_linear *lin, int n_layers) {
    const XLayout X = xlayout(lin);
    return desc_bytes_for(n_layers) + xacc_bytes(X, n_layers) + cst_bytes(n_layers) +
           (size_t)kMaxCtas * kProgBytes;
}

namespace {
char *xacc_at(int n_layers, char *ws_after_header) {
    return ws_after_header + desc_bytes_for(n_layers);
}
float4 *cst_at(const lb_linear *lin, int n_layers, char *ws_after_header) {
    return reinterpret_cast<float4 *>(xacc_at(n_layers, ws_after_header) +
                                      xacc_bytes(xlayout(lin), n_layers));
}
char *programs_at(const lb_linear *lin, int n_layers, char *ws_after_header) {
    return reinterpret_cast<char *>(cst_at(lin, n_layers, ws_after_header)) + cst_bytes(n_layers);
}
}  // namespace

cudaError_t launch_stack_prepare(const lb_linear *lin, int n_layers, const StackShape &sh,
                                 int num_sms, int cluster, unsigned long long plan,
                                 unsigned *ws_words, char *ws_after_header, cudaStream_t s) {
    if (!shapes_ok(lin, sh, num_sms, cluster) || !smem_fits(lin, sh, num_sms, cluster))
        return cudaErrorNotSupported;
    std::vector<int> progs;
    if (!build_programs(lin, sh, num_sms, cluster, progs)) return cudaErrorNotSupported;
    const XLayout X = xlayout(lin);
    LinDesc *desc = reinterpret_cast<LinDesc *>(ws_after_header);
    char *xacc = xacc_at(n_layers, ws_after_header);
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, 2 * sizeof(unsigned), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(xacc, 0, xacc_bytes(X, n_layers), s);
    // pageable source: the call returns once the data is staged
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(programs_at(lin, n_layers, ws_after_header), progs.data(),
                            progs.size() * sizeof(int), cudaMemcpyHostToDevice, s);
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
    k_stack_consts<<<n_layers + 1, kConstThreads, 0, s>>>(desc, n_layers, sh.d / sh.dkv,
                                                         cst_at(lin, n_layers, ws_after_header));
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_set_plan<<<1, 1, 0, s>>>(ws_words, plan);
    return cudaGetLastError();
}

bool stack_supported(const lb_linear *lin, const StackShape &sh, int num_sms, int cluster) {
    return shapes_ok(lin, sh, num_sms, cluster) && smem_fits(lin, sh, num_sms, cluster);
}

int stack_grid_ctas(const lb_linear *lin, const StackShape &sh, int num_sms, int cluster) {
    if (cluster == 1) return num_sms;
    if (cluster != 2) return 0;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    // the plan of the full grid bounds the shared memory from below (smaller
    // grids give each CTA larger slices); clusters need not fill every SM
    const int smem = smem_plan(lin, sh, num_sms, cluster).bytes;
    static std::mutex mu;
    static int cached_dev = -1, cached_smem = -1, cached_sms = -1, cached_n = 0;
    std::lock_guard<std::mutex> lock(mu);
    if (dev == cached_dev && smem == cached_smem && num_sms == cached_sms) return cached_n;
    const void *fn = (const void *)k_stack<2>;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
        return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster, 1, 1);
    cfg.blockDim = dim3(kST, 1, 1);
    cfg.dynamicSmemBytes = (size_t)smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = cluster;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n_cl = 0;
    if (cudaOccupancyMaxActiveClusters(&n_cl, fn, &cfg) != cudaSuccess || n_cl <= 0) return 0;
    const int n = std::min(num_sms / cluster, n_cl) * cluster;
    // the larger slices of the smaller grid must still fit
    if (!smem_fits(lin, sh, n, cluster)) return 0;
    cached_dev = dev;
    cached_smem = smem;
    cached_sms = num_sms;
    cached_n = n;
    return n;
}

cudaError_t launch_stack(const lb_linear *lin, int n_layers, const StackShape &sh,
                         unsigned long long plan, const uint16_t *x0, float *out, float *q_out,
                         float *kv_out, unsigned *ws_words, char *ws_after_header, int num_sms,
                         int cluster, cudaStream_t s) {
    if (cluster < 1 || cluster > kMaxCluster || num_sms % cluster != 0)
        return cudaErrorInvalidConfiguration;
    const XLayout X = xlayout(lin);
    const SmemPlan S = smem_plan(lin, sh, num_sms, cluster);
    Params P{};
    P.lin = reinterpret_cast<const LinDesc *>(ws_after_header);
    P.prog = reinterpret_cast<const int *>(programs_at(lin, n_layers, ws_after_header));
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
    P.xacc = reinterpret_cast<unsigned long long *>(xacc_at(n_layers, ws_after_header));
    P.cst = cst_at(lin, n_layers, ws_after_header);
    P.acc_layer = X.acc_layer;
    P.offA = X.offA;
    P.offQ = X.offQ;
    P.lenQ = X.lenQ;
    P.offB = X.offB;
    P.offC = X.offC;
    P.offD = X.offD;
    P.lenA = X.lenA;
    P.lenB = X.lenB;
    P.lenC = X.lenC;
    P.lenD = X.lenD;
    P.n_t = (unsigned)(num_sms / cluster);
    P.lim_t = fix1_limit((int)P.n_t);
    P.lim_ss = fix1_limit(num_sms);
    P.o = S.o;
    const size_t smem = (size_t)S.bytes;
    const void *fn = cluster == 2 ? (const void *)k_stack<2> : (const void *)k_stack<1>;
    cudaError_t e =
        cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kST, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorCooperativeLaunchTooLarge;
    // cooperative: the grid is launched only if every CTA is co-resident (the
    // kernel's waits need that); clusters of `cluster` consecutive CTAs
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(num_sms, 1, 1);
    cfg.blockDim = dim3(kST, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeCooperative;
    at[0].val.cooperative = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cluster;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cluster == 2 ? cudaLaunchKernelEx(&cfg, k_stack<2>, P)
                        : cudaLaunchKernelEx(&cfg, k_stack<1>, P);
}

}  // namespace lb
