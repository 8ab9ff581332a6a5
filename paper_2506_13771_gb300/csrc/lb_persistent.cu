// lb_persistent.cu -- single-launch decode (T = 1) of one LittleBit linear as a
// persistent kernel with one CTA per SM and a bounded grid-wide wait.
//
// Prop. 1 (LittleBit, arXiv 2506.13771) splits each linear into a +-1
// reduction over d_in (stage 1, rank-r result t) and a +-1 reduction over r
// (stage 2).  Every CTA owns a slice of the input words: it forms the partial
// t of its slice and red.adds it into an fp32 accumulator in the workspace.
// After one grid-wide wait every CTA holds the full t and produces its own
// slice of output rows.
#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kThreads = 512;

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

__device__ void zero_shared(float *p, int n) {
    for (int i = threadIdx.x; i < n; i += blockDim.x) p[i] = 0.f;
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

// One CTA waits at a grid barrier that needs two arrivals: only its own comes,
// so the bounded wait must run out and record LB_ERR_TIMEOUT.
__global__ void k_wait_timeout(unsigned *ws_words) {
    if (sticky_error(ws_words)) return;
    if (!grid_barrier(ws_words, 2u)) return;
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

cudaError_t launch_wait_timeout(unsigned *ws_words, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(ws_words + kCounterWord, 0, sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
    k_wait_timeout<<<1, 32, 0, s>>>(ws_words);
    return cudaGetLastError();
}

}  // namespace lb
