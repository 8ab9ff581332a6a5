// lb_persistent.cu -- single-launch decode (T = 1) of one LittleBit linear and
// of the seven-linear-per-layer stack, as persistent kernels with one CTA per
// SM and bounded grid-wide waits.
//
// Prop. 1 (LittleBit, arXiv 2506.13771) splits each linear into a +-1
// reduction over d_in (stage 1, rank-r result t) and a +-1 reduction over r
// (stage 2).  Every CTA owns a slice of the input words: it forms the partial
// t of its slice and red.adds it into an fp32 accumulator in the workspace.
// After one grid-wide wait every CTA holds the full t and produces its own
// slice of output rows.  In the stack, a CTA's output-row slice of one linear
// is the input slice of the next, so stage 2 of linear n and stage 1 of
// linear n+1 run back to back on the same CTA with no exchange in between;
// the only exchange is the rank-r all-reduce of t (plus one sum of squares
// for the rms normalisation, folded into stage 2 by homogeneity:
// L(v / rms(v)) = L(v) / rms(v)).
#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kThreads = 512;
constexpr int kMaxJobs = 6;

int round_up32(int n) { return (n + 31) & ~31; }

// ---------------------------------------------------------------- building blocks

// One stage-1 partial: all columns of one (linear, path) over the CTA's slice.
struct VJob {
    const uint32_t *V;  // full V words of the path, [d_in/32][r]
    const uint16_t *g;  // full column scale
    float *acc;         // global accumulator of this path's t, r floats
    int r;
};

// One stage-2 row block: rows of one (linear, path), accumulated into ys.
struct UJob {
    const uint32_t *U;  // full U words, [d_out][ceil(r/32)]
    const uint16_t *h;  // full row scale
    const float *z;     // l . t / rms, in shared memory, r floats
    float *ys;          // shared output rows
    int r;
    // Row map: output row o reads U row ((o / hd) / grp) * hd + o % hd.  With
    // grp = 1 this is the identity; with grp = query heads per kv head it
    // gathers, for a slice of attention-output rows, the v rows they read.
    int hd, grp;
};

__device__ __forceinline__ int map_row(int o, int hd, int grp) {
    if (grp == 1) return o;
    const int head = o / hd;
    return (head / grp) * hd + (o - head * hd);
}

// Stage 1 over input words [w0, w0 + nw): for every job column j,
//   acc[j] += sum_{i in slice} V_sign[i][j] * g[i] * xs[i - 32 w0].
// s_a: shared scratch of njobs * nw * 32 floats.
__device__ void v_partials(const VJob *jobs, int njobs, const float *xs, int w0, int nw,
                           float *s_a) {
    if (nw <= 0) return;
    const int n_in = nw * 32;
    for (int e = threadIdx.x; e < njobs * n_in; e += blockDim.x) {
        const int jb = e / n_in, i = e - jb * n_in;
        s_a[e] = xs[i] * half_bits_to_float(jobs[jb].g[w0 * 32 + i]);
    }
    __syncthreads();
    int total = 0;
    for (int jb = 0; jb < njobs; ++jb) total += jobs[jb].r;
    for (int col = threadIdx.x; col < total; col += blockDim.x) {
        int c = col, jb = 0;
        while (c >= jobs[jb].r) {
            c -= jobs[jb].r;
            ++jb;
        }
        const int r = jobs[jb].r;
        const uint32_t *V = jobs[jb].V + (size_t)w0 * r + c;
        const float *a = s_a + jb * n_in;
        float acc = 0.f;
        for (int w = 0; w < nw; ++w) {
            const uint32_t word = __ldg(V + (size_t)w * r);
            const float *aw = a + w * 32;
#pragma unroll
            for (int k = 0; k < 32; ++k) acc += apply_sign(aw[k], word, k);
        }
        red_add_f32(jobs[jb].acc + c, acc);
    }
}

// Stage 2 over rows [o0, o0 + nrows): ys[row] += h[o] * sum_j U_sign[o][j] z[j].
// Work items are (row, word) pairs; consecutive lanes take consecutive words
// of a row, and each lane starts its 32 bits at a different offset so the
// z reads of one warp fall in distinct shared-memory banks.
__device__ void u_rows(const UJob *jobs, int njobs, int o0, int nrows) {
    if (nrows <= 0) return;
    for (int jb = 0; jb < njobs; ++jb) {
        const int r = jobs[jb].r;
        const int R = (r + 31) >> 5;
        const int hd = jobs[jb].hd, grp = jobs[jb].grp;
        const int items = nrows * R;
        for (int it = threadIdx.x; it < items; it += blockDim.x) {
            const int row = it / R, w = it - row * R;
            const int urow = map_row(o0 + row, hd, grp);
            const uint32_t word = __ldg(jobs[jb].U + (size_t)urow * R + w);
            const float *zw = jobs[jb].z + 32 * w;
            const int nb = min(32, r - 32 * w);
            float acc = 0.f;
            if (nb == 32) {
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                    const int kk = (k + w) & 31;
                    acc += apply_sign(zw[kk], word, kk);
                }
            } else {
                for (int k = 0; k < nb; ++k) acc += apply_sign(zw[k], word, k);
            }
            atomicAdd(jobs[jb].ys + row, acc * half_bits_to_float(jobs[jb].h[urow]));
        }
    }
}

// z_p[j] = l_p[j] * t_p[j] * inv_rms for every path of L; t read from the
// global accumulator (L2 only: it was produced by red.add of other CTAs).
__device__ void load_z(const LinDesc &L, const float *acc, float inv_rms, float *zs) {
    int off = 0;
    for (int p = 0; p < L.n_paths; ++p) {
        const int r = L.r[p];
        for (int j = threadIdx.x; j < r; j += blockDim.x)
            zs[off + j] = half_bits_to_float(L.l[p][j]) * __ldcg(acc + off + j) * inv_rms;
        off += r;
    }
}

__device__ int rank_sum(const LinDesc &L) {
    int s = 0;
    for (int p = 0; p < L.n_paths; ++p) s += L.r[p];
    return s;
}

__device__ void zero_shared(float *p, int n) {
    for (int i = threadIdx.x; i < n; i += blockDim.x) p[i] = 0.f;
}

// Sum of squares of xs[0..n) added to *dst (one red.add per CTA).
__device__ void add_sumsq(const float *xs, int n, float *dst) {
    float s = 0.f;
    for (int i = threadIdx.x; i < n; i += blockDim.x) s += xs[i] * xs[i];
    s = block_sum(s);
    if (threadIdx.x == 0 && n > 0) red_add_f32(dst, s);
}

// Append the stage-1 jobs of every path of L; acc points at this linear's t.
__device__ int push_vjobs(VJob *jobs, int nj, const LinDesc &L, float *acc) {
    int off = 0;
    for (int p = 0; p < L.n_paths; ++p) {
        jobs[nj++] = VJob{L.v[p], L.g[p], acc + off, L.r[p]};
        off += L.r[p];
    }
    return nj;
}

__device__ int push_ujobs(UJob *jobs, int nj, const LinDesc &L, const float *zs, float *ys,
                          int hd = 1, int grp = 1) {
    int off = 0;
    for (int p = 0; p < L.n_paths; ++p) {
        jobs[nj++] = UJob{L.u[p], L.h[p], zs + off, ys, L.r[p], hd, grp};
        off += L.r[p];
    }
    return nj;
}

__device__ __forceinline__ bool sticky_error(const unsigned *ws_words) {
    return ld_relaxed_gpu(ws_words + kErrWord) != 0u;
}

// ---------------------------------------------------------------- single linear

struct DecodeParams {
    LinDesc L;
    const uint16_t *x;
    void *y;
    int y_fp32;
    unsigned *ws_words;
    float *acc;
    int sm_xs, sm_a, sm_z, sm_y;  // shared-memory offsets in floats
};

__global__ void __launch_bounds__(kThreads, 1) k_linear_decode(const DecodeParams P) {
    extern __shared__ float smem[];
    if (sticky_error(P.ws_words)) return;
    float *xs = smem + P.sm_xs, *s_a = smem + P.sm_a, *zs = smem + P.sm_z, *ys = smem + P.sm_y;
    const int N = gridDim.x, c = blockIdx.x;
    const LinDesc &L = P.L;
    const int W = L.d_in >> 5;
    const int w0 = (int)((long long)c * W / N), w1 = (int)((long long)(c + 1) * W / N);
    const int nw = w1 - w0;
    for (int i = threadIdx.x; i < nw * 32; i += blockDim.x)
        xs[i] = bf16_bits_to_float(P.x[w0 * 32 + i]);
    __syncthreads();
    VJob vj[2];
    const int nv = push_vjobs(vj, 0, L, P.acc);
    v_partials(vj, nv, xs, w0, nw, s_a);
    if (!grid_barrier(P.ws_words, (unsigned)N)) return;
    load_z(L, P.acc, 1.f, zs);
    const int o0 = (int)((long long)c * L.d_out / N), o1 = (int)((long long)(c + 1) * L.d_out / N);
    zero_shared(ys, o1 - o0);
    __syncthreads();
    UJob uj[2];
    const int nu = push_ujobs(uj, 0, L, zs, ys);
    u_rows(uj, nu, o0, o1 - o0);
    __syncthreads();
    for (int i = threadIdx.x; i < o1 - o0; i += blockDim.x) {
        if (P.y_fp32)
            static_cast<float *>(P.y)[o0 + i] = ys[i];
        else
            static_cast<uint16_t *>(P.y)[o0 + i] = float_to_bf16_bits(ys[i]);
    }
}

// ---------------------------------------------------------------- stack

// Decode step at sequence position 0 of n_layers Llama-shaped blocks:
//   n = rho(a); q, k, v = Q, K, V(n); attn = v broadcast over each kv head's
//   query heads (softmax over one position is 1); h = a + O(attn);
//   n = rho(h); m = silu(Gate(n)) * Up(n); a = h + Down(m).
// CTA c owns d-rows R_c (whole 32-row words), f-rows F_c and kv-rows K_c.
// The residual stream slice a/h on R_c stays in shared memory across the
// whole launch.  Per layer, four rank-r all-reduces:
//   A: stage 1 of q, k, v on a(R_c)                  (+ sum of squares of a)
//   B: stage 2 of q (R_c), k, v (K_c) and of v on the rows attn(R_c) reads;
//      stage 1 of o on attn(R_c)
//   C: stage 2 of o -> h(R_c) = a + o; stage 1 of gate, up on h(R_c) (+ ss of h)
//   D: stage 2 of gate, up (F_c) -> m; stage 1 of down on m(F_c)
// and the next layer's A begins with stage 2 of down: a(R_c) = h + down.
struct StackParams {
    const LinDesc *lin;  // device, 7 * n_layers
    int n_layers, d, dkv, dff, head_dim;
    const uint16_t *x0;
    float *out, *q_out, *kv_out;
    unsigned *ws_words;
    unsigned long long plan;                // fingerprint the workspace must hold
    float *acc;
    int acc_layer, offA, offB, offC, offD;  // floats
    int lenA, lenB, lenC, lenD;             // used floats of each region
    int sm_res, sm_xs, sm_a, sm_z, sm_y;    // shared-memory offsets in floats
};

// Zero this CTA's stripe of an accumulator region whose last readers have
// all passed a later grid barrier: the launch leaves the workspace zeroed
// for the next one.
__device__ __forceinline__ void zero_stripe(float *region, int len) {
    const int a = (int)((long long)blockIdx.x * len / gridDim.x);
    const int b = (int)((long long)(blockIdx.x + 1) * len / gridDim.x);
    for (int i = a + threadIdx.x; i < b; i += blockDim.x) region[i] = 0.f;
}

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }

__global__ void __launch_bounds__(kThreads, 1) k_stack_decode(const StackParams P) {
    extern __shared__ float smem[];
    if (sticky_error(P.ws_words)) return;
    {
        const unsigned long long plan =
            *reinterpret_cast<const volatile unsigned long long *>(P.ws_words + kPlanWord);
        if (plan != P.plan) {
            if (blockIdx.x == 0 && threadIdx.x == 0)
                atomicCAS(P.ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_PLAN));
            return;
        }
    }
    float *res = smem + P.sm_res, *xs = smem + P.sm_xs, *s_a = smem + P.sm_a;
    float *zs = smem + P.sm_z, *ys = smem + P.sm_y;
    const int N = gridDim.x, c = blockIdx.x;
    const int Wd = P.d >> 5, Wf = P.dff >> 5;
    const int dw0 = (int)((long long)c * Wd / N), dw1 = (int)((long long)(c + 1) * Wd / N);
    const int fw0 = (int)((long long)c * Wf / N), fw1 = (int)((long long)(c + 1) * Wf / N);
    const int k0 = (int)((long long)c * P.dkv / N), k1 = (int)((long long)(c + 1) * P.dkv / N);
    const int nd = dw1 - dw0, nf = fw1 - fw0, nkv = k1 - k0;
    const int rows_d = nd * 32, rows_f = nf * 32;
    const int grp = P.d / P.dkv;
    unsigned barrier_no = 0;
    VJob vj[kMaxJobs];
    UJob uj[kMaxJobs];

    for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
        res[i] = bf16_bits_to_float(P.x0[dw0 * 32 + i]);

    for (int l = 0; l < P.n_layers; ++l) {
        const LinDesc *Ly = P.lin + 7 * l;
        float *accA = P.acc + (size_t)l * P.acc_layer + P.offA;
        float *accB = P.acc + (size_t)l * P.acc_layer + P.offB;
        float *accC = P.acc + (size_t)l * P.acc_layer + P.offC;
        float *accD = P.acc + (size_t)l * P.acc_layer + P.offD;
        const int rq = rank_sum(Ly[0]), rk = rank_sum(Ly[1]), rv = rank_sum(Ly[2]);
        const int rg = rank_sum(Ly[4]), ru = rank_sum(Ly[5]);
        const int ssA = rq + rk + rv, ssC = rg + ru;

        // ---- phase A: a = h + Down_{l-1}(m) on R_c; stage 1 of q, k, v
        if (l > 0) {
            const LinDesc &Dn = P.lin[7 * (l - 1) + 6];
            const float *accDp = P.acc + (size_t)(l - 1) * P.acc_layer + P.offD;
            // every CTA read the previous layer's C region before barrier D
            zero_stripe(P.acc + (size_t)(l - 1) * P.acc_layer + P.offC, P.lenC);
            load_z(Dn, accDp, 1.f, zs);
            zero_shared(ys, rows_d);
            __syncthreads();
            const int nu = push_ujobs(uj, 0, Dn, zs, ys);
            u_rows(uj, nu, dw0 * 32, rows_d);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_d; i += blockDim.x) res[i] += ys[i];
        }
        __syncthreads();
        add_sumsq(res, rows_d, accA + ssA);
        {
            int nv = push_vjobs(vj, 0, Ly[0], accA);
            nv = push_vjobs(vj, nv, Ly[1], accA + rq);
            nv = push_vjobs(vj, nv, Ly[2], accA + rq + rk);
            v_partials(vj, nv, res, dw0, nd, s_a);
        }
        if (!grid_barrier(P.ws_words, (unsigned)N * ++barrier_no)) return;

        // ---- phase B: q on R_c, k and v on K_c, v on the rows attn(R_c)
        //      reads; stage 1 of o on attn(R_c)
        {
            if (l > 0) zero_stripe(P.acc + (size_t)(l - 1) * P.acc_layer + P.offD, P.lenD);
            const float inv = rsqrtf(__ldcg(accA + ssA) / (float)P.d);
            load_z(Ly[0], accA, inv, zs);
            load_z(Ly[1], accA + rq, inv, zs + rq);
            load_z(Ly[2], accA + rq + rk, inv, zs + rq + rk);
            float *yq = ys, *yk = ys + rows_d, *yv = yk + nkv, *attn = xs;
            zero_shared(ys, rows_d + 2 * nkv);
            zero_shared(attn, rows_d);
            __syncthreads();
            int nu = push_ujobs(uj, 0, Ly[0], zs, yq);
            u_rows(uj, nu, dw0 * 32, rows_d);
            nu = push_ujobs(uj, 0, Ly[1], zs + rq, yk);
            nu = push_ujobs(uj, nu, Ly[2], zs + rq + rk, yv);
            u_rows(uj, nu, k0, nkv);
            nu = push_ujobs(uj, 0, Ly[2], zs + rq + rk, attn, P.head_dim, grp);
            u_rows(uj, nu, dw0 * 32, rows_d);
            __syncthreads();
            if (P.q_out)
                for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
                    P.q_out[(size_t)l * P.d + dw0 * 32 + i] = yq[i];
            if (P.kv_out)
                for (int i = threadIdx.x; i < nkv; i += blockDim.x) {
                    P.kv_out[((size_t)l * 2 + 0) * P.dkv + k0 + i] = yk[i];
                    P.kv_out[((size_t)l * 2 + 1) * P.dkv + k0 + i] = yv[i];
                }
            const int nv = push_vjobs(vj, 0, Ly[3], accB);
            v_partials(vj, nv, attn, dw0, nd, s_a);
        }
        if (!grid_barrier(P.ws_words, (unsigned)N * ++barrier_no)) return;

        // ---- phase C: h = a + O(attn) on R_c; stage 1 of gate, up on h
        {
            zero_stripe(accA, P.lenA);
            load_z(Ly[3], accB, 1.f, zs);
            zero_shared(ys, rows_d);
            __syncthreads();
            const int nu = push_ujobs(uj, 0, Ly[3], zs, ys);
            u_rows(uj, nu, dw0 * 32, rows_d);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_d; i += blockDim.x) res[i] += ys[i];
            __syncthreads();
            add_sumsq(res, rows_d, accC + ssC);
            int nv = push_vjobs(vj, 0, Ly[4], accC);
            nv = push_vjobs(vj, nv, Ly[5], accC + rg);
            v_partials(vj, nv, res, dw0, nd, s_a);
        }
        if (!grid_barrier(P.ws_words, (unsigned)N * ++barrier_no)) return;

        // ---- phase D: m = silu(gate) * up on F_c; stage 1 of down on m
        {
            zero_stripe(accB, P.lenB);
            const float inv = rsqrtf(__ldcg(accC + ssC) / (float)P.d);
            load_z(Ly[4], accC, inv, zs);
            load_z(Ly[5], accC + rg, inv, zs + rg);
            float *yg = ys, *yu = ys + rows_f;
            zero_shared(ys, 2 * rows_f);
            __syncthreads();
            int nu = push_ujobs(uj, 0, Ly[4], zs, yg);
            nu = push_ujobs(uj, nu, Ly[5], zs + rg, yu);
            u_rows(uj, nu, fw0 * 32, rows_f);
            __syncthreads();
            for (int i = threadIdx.x; i < rows_f; i += blockDim.x) xs[i] = silu(yg[i]) * yu[i];
            __syncthreads();
            const int nv = push_vjobs(vj, 0, Ly[6], accD);
            v_partials(vj, nv, xs, fw0, nf, s_a);
        }
        if (!grid_barrier(P.ws_words, (unsigned)N * ++barrier_no)) return;
        (void)ru;
    }

    // ---- final: out = h + Down_{L-1}(m) on R_c
    {
        const int l = P.n_layers - 1;
        const LinDesc &Dn = P.lin[7 * l + 6];
        float *accD = P.acc + (size_t)l * P.acc_layer + P.offD;
        zero_stripe(P.acc + (size_t)l * P.acc_layer + P.offC, P.lenC);
        load_z(Dn, accD, 1.f, zs);
        zero_shared(ys, rows_d);
        __syncthreads();
        const int nu = push_ujobs(uj, 0, Dn, zs, ys);
        u_rows(uj, nu, dw0 * 32, rows_d);
        __syncthreads();
        for (int i = threadIdx.x; i < rows_d; i += blockDim.x)
            P.out[dw0 * 32 + i] = res[i] + ys[i];
        // The last CTA to finish has seen every other CTA's reads of the final
        // region: it clears that region and the counters for the next launch.
        __shared__ int s_last;
        if (threadIdx.x == 0) {
            __threadfence();
            s_last = atomicAdd(P.ws_words + kDoneWord, 1u) == (unsigned)N - 1;
        }
        __syncthreads();
        if (s_last) {
            __threadfence();
            for (int i = threadIdx.x; i < P.lenD; i += blockDim.x) accD[i] = 0.f;
            if (threadIdx.x == 0) {
                P.ws_words[kCounterWord] = 0u;
                P.ws_words[kDoneWord] = 0u;
            }
        }
    }
}

// One CTA waits at a grid barrier that needs two arrivals: only its own comes,
// so the bounded wait must run out and record LB_ERR_TIMEOUT.
__global__ void k_wait_timeout(unsigned *ws_words) {
    if (sticky_error(ws_words)) return;
    if (!grid_barrier(ws_words, 2u)) return;
}

// Copies linear descriptors from kernel-parameter space into the workspace, so
// the host array reaches the device with the launch itself (no staging copy).
constexpr int kDescChunk = 256;
struct DescChunk {
    int count;
    LinDesc d[kDescChunk];
};

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

int rank_sum_host(const lb_linear &L) {
    int s = 0;
    for (int p = 0; p < L.n_paths; ++p) s += L.path[p].r;
    return s;
}

cudaError_t cooperative_launch(const void *fn, int grid, size_t smem, void **args,
                               cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorCooperativeLaunchTooLarge;
    return cudaLaunchCooperativeKernel(fn, dim3(grid), dim3(kThreads), args, smem, s);
}

}  // namespace

static_assert(sizeof(LinDesc) % sizeof(uint32_t) == 0, "descriptor is copied as words");

size_t decode_ws_floats(const lb_linear &L) { return (size_t)round_up32(rank_sum_host(L)); }

cudaError_t launch_decode(const lb_linear &L, const uint16_t *x, void *y, int y_fp32,
                          unsigned *ws_words, float *acc, int num_sms, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, sizeof(unsigned), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(acc, 0, decode_ws_floats(L) * sizeof(float), s);
    if (e != cudaSuccess) return e;
    DecodeParams P{};
    P.L = make_desc(L);
    P.x = x;
    P.y = y;
    P.y_fp32 = y_fp32;
    P.ws_words = ws_words;
    P.acc = acc;
    const int N = num_sms;
    const int nw = (L.d_in / 32 + N - 1) / N;
    const int nrows = (L.d_out + N - 1) / N;
    P.sm_xs = 0;
    P.sm_a = P.sm_xs + round_up32(nw * 32);
    P.sm_z = P.sm_a + round_up32(L.n_paths * nw * 32);
    P.sm_y = P.sm_z + round_up32(rank_sum_host(L));
    const size_t smem = (size_t)(P.sm_y + round_up32(nrows)) * sizeof(float);
    void *args[] = {&P};
    return cooperative_launch((const void *)k_linear_decode, N, smem, args, s);
}

namespace {
struct StackLayout {
    int acc_layer, offA, offB, offC, offD, lenA, lenB, lenC, lenD;
};

// Accumulator floats of one layer: A = t of q, k, v + ss(a); B = t of o;
// C = t of gate, up + ss(h); D = t of down.  Each region padded to 128 bytes.
StackLayout stack_layout(const lb_linear *lin) {
    StackLayout S{};
    const int A = rank_sum_host(lin[0]) + rank_sum_host(lin[1]) + rank_sum_host(lin[2]) + 1;
    const int B = rank_sum_host(lin[3]);
    const int C = rank_sum_host(lin[4]) + rank_sum_host(lin[5]) + 1;
    const int D = rank_sum_host(lin[6]);
    S.lenA = A;
    S.lenB = B;
    S.lenC = C;
    S.lenD = D;
    S.offA = 0;
    S.offB = S.offA + round_up32(A);
    S.offC = S.offB + round_up32(B);
    S.offD = S.offC + round_up32(C);
    S.acc_layer = S.offD + round_up32(D);
    return S;
}

size_t desc_bytes_for(int n_layers) {
    return ((size_t)7 * n_layers * sizeof(LinDesc) + 255) & ~(size_t)255;
}
}  // namespace

size_t stack_ws_bytes_after_header(const lb_linear *lin, int n_layers) {
    const StackLayout S = stack_layout(lin);
    return desc_bytes_for(n_layers) + (size_t)n_layers * S.acc_layer * sizeof(float);
}

cudaError_t launch_stack_prepare(const lb_linear *lin, int n_layers, unsigned long long plan,
                                 unsigned *ws_words, char *ws_after_header, cudaStream_t s) {
    const StackLayout S = stack_layout(lin);
    LinDesc *desc = reinterpret_cast<LinDesc *>(ws_after_header);
    float *acc = reinterpret_cast<float *>(ws_after_header + desc_bytes_for(n_layers));
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, 2 * sizeof(unsigned), s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(acc, 0, (size_t)n_layers * S.acc_layer * sizeof(float), s);
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

cudaError_t launch_stack(const lb_linear *lin, int n_layers, const StackShape &shape,
                         unsigned long long plan, const uint16_t *x0, float *out, float *q_out,
                         float *kv_out, unsigned *ws_words, char *ws_after_header, int num_sms,
                         cudaStream_t s) {
    const StackLayout S = stack_layout(lin);
    StackParams P{};
    P.lin = reinterpret_cast<const LinDesc *>(ws_after_header);
    P.acc = reinterpret_cast<float *>(ws_after_header + desc_bytes_for(n_layers));
    P.plan = plan;
    P.n_layers = n_layers;
    P.d = shape.d;
    P.dkv = shape.dkv;
    P.dff = shape.dff;
    P.head_dim = shape.head_dim;
    P.x0 = x0;
    P.out = out;
    P.q_out = q_out;
    P.kv_out = kv_out;
    P.ws_words = ws_words;
    P.acc_layer = S.acc_layer;
    P.offA = S.offA;
    P.offB = S.offB;
    P.offC = S.offC;
    P.offD = S.offD;
    P.lenA = S.lenA;
    P.lenB = S.lenB;
    P.lenC = S.lenC;
    P.lenD = S.lenD;
    const int N = num_sms;
    const int nd = (shape.d / 32 + N - 1) / N, nf = (shape.dff / 32 + N - 1) / N;
    const int nkv = (shape.dkv + N - 1) / N;
    const int rq = rank_sum_host(lin[0]), rk = rank_sum_host(lin[1]), rv = rank_sum_host(lin[2]);
    const int ro = rank_sum_host(lin[3]), rg = rank_sum_host(lin[4]), ru = rank_sum_host(lin[5]);
    const int rd = rank_sum_host(lin[6]);
    const int res_n = 32 * nd;
    const int xs_n = 32 * (nd > nf ? nd : nf);                 // attn (d rows) or m (f rows)
    int a_n = 6 * 32 * nd;                                       // stage-1 jobs x slice inputs
    if (2 * 32 * nf > a_n) a_n = 2 * 32 * nf;
    int z_n = rq + rk + rv;
    if (ro > z_n) z_n = ro;
    if (rg + ru > z_n) z_n = rg + ru;
    if (rd > z_n) z_n = rd;
    int y_n = 32 * nd + 2 * nkv;
    if (2 * 32 * nf > y_n) y_n = 2 * 32 * nf;
    P.sm_res = 0;
    P.sm_xs = P.sm_res + round_up32(res_n);
    P.sm_a = P.sm_xs + round_up32(xs_n);
    P.sm_z = P.sm_a + round_up32(a_n);
    P.sm_y = P.sm_z + round_up32(z_n);
    const size_t smem = (size_t)(P.sm_y + round_up32(y_n)) * sizeof(float);
    void *args[] = {&P};
    return cooperative_launch((const void *)k_stack_decode, N, smem, args, s);
}

cudaError_t launch_wait_timeout(unsigned *ws_words, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
    k_wait_timeout<<<1, 32, 0, s>>>(ws_words);
    return cudaGetLastError();
}

}  // namespace lb
