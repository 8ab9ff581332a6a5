// lb_generic.cu -- any-T LittleBit forward on CUDA cores, two launches.
//
// Prop. 1 (LittleBit, arXiv 2506.13771), per path p:
//   stage 1  t_p[tok][j] = sum_i V_p,sign[i][j] * g_p[i] * X[tok][i]
//   stage 2  Y[tok][o]  += h_p[o] * sum_j U_p,sign[o][j] * l_p[j] * t_p[tok][j]
// and Eq. 6 sums the paths.  Stage 1 splits d_in over blocks and reduces into
// the fp32 workspace with red.add; stage 2 reads the finished t.  This is the
// path for token counts the decode and tensor-core kernels do not take.
#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kGenThreads = 256;
constexpr int kVTok = 8;   // tokens per stage-1 block
constexpr int kUTok = 4;   // tokens per stage-2 block

// grid: (word chunks of d_in, token tiles, paths)
__global__ void __launch_bounds__(kGenThreads)
k_stage1_generic(LinDesc L, const uint16_t *__restrict__ x, int T, int chunk_words,
                 float *__restrict__ t_acc, int t_off1) {
    extern __shared__ float s_a[];  // [kVTok][chunk_words*32]
    const int p = blockIdx.z;
    const int r = L.r[p];
    const int W = L.d_in >> 5;
    const int w0 = blockIdx.x * chunk_words;
    const int nw = min(chunk_words, W - w0);
    const int tok0 = blockIdx.y * kVTok;
    const int ntok = min(kVTok, T - tok0);
    const int n_in = nw * 32;
    const uint16_t *g = L.g[p];
    for (int e = threadIdx.x; e < kVTok * n_in; e += blockDim.x) {
        const int tt = e / n_in, i = e - tt * n_in;
        float a = 0.f;
        if (tt < ntok) {
            const int gi = w0 * 32 + i;
            a = bf16_bits_to_float(x[(size_t)(tok0 + tt) * L.d_in + gi]) *
                half_bits_to_float(g[gi]);
        }
        s_a[tt * n_in + i] = a;
    }
    __syncthreads();
    float *t_p = t_acc + (p == 0 ? 0 : t_off1);
    const uint32_t *V = L.v[p];
    for (int j = threadIdx.x; j < r; j += blockDim.x) {
        float acc[kVTok];
#pragma unroll
        for (int tt = 0; tt < kVTok; ++tt) acc[tt] = 0.f;
        for (int w = 0; w < nw; ++w) {
            const uint32_t word = __ldg(V + (size_t)(w0 + w) * r + j);
            const float *aw = s_a + w * 32;
#pragma unroll 8
            for (int k = 0; k < 32; ++k) {
#pragma unroll
                for (int tt = 0; tt < kVTok; ++tt)
                    acc[tt] += apply_sign(aw[tt * n_in + k], word, k);
            }
        }
        for (int tt = 0; tt < ntok; ++tt) red_add_f32(t_p + (size_t)(tok0 + tt) * r + j, acc[tt]);
    }
}

// grid: (row blocks of d_out, token tiles)
__global__ void __launch_bounds__(kGenThreads)
k_stage2_generic(LinDesc L, int T, const float *__restrict__ t_acc, int t_off1, void *y,
                 int y_fp32) {
    extern __shared__ float s_z[];  // [paths][kUTok][r_p]
    const int tok0 = blockIdx.y * kUTok;
    const int ntok = min(kUTok, T - tok0);
    int zoff[2] = {0, kUTok * L.r[0]};
    for (int p = 0; p < L.n_paths; ++p) {
        const int r = L.r[p];
        const float *t_p = t_acc + (p == 0 ? 0 : t_off1);
        for (int e = threadIdx.x; e < kUTok * r; e += blockDim.x) {
            const int tt = e / r, j = e - tt * r;
            s_z[zoff[p] + e] =
                tt < ntok ? __ldcg(t_p + (size_t)(tok0 + tt) * r + j) * half_bits_to_float(L.l[p][j])
                          : 0.f;
        }
    }
    __syncthreads();
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= L.d_out) return;
    float y_acc[kUTok];
#pragma unroll
    for (int tt = 0; tt < kUTok; ++tt) y_acc[tt] = 0.f;
    for (int p = 0; p < L.n_paths; ++p) {
        const int r = L.r[p];
        const int R = (r + 31) >> 5;
        const uint32_t *U = L.u[p] + (size_t)o * R;
        float acc[kUTok];
#pragma unroll
        for (int tt = 0; tt < kUTok; ++tt) acc[tt] = 0.f;
        for (int w = 0; w < R; ++w) {
            const uint32_t word = __ldg(U + w);
            const int nb = min(32, r - 32 * w);
            const float *zw = s_z + zoff[p] + 32 * w;
            for (int k = 0; k < nb; ++k) {
#pragma unroll
                for (int tt = 0; tt < kUTok; ++tt) acc[tt] += apply_sign(zw[tt * r + k], word, k);
            }
        }
        const float hp = half_bits_to_float(L.h[p][o]);
#pragma unroll
        for (int tt = 0; tt < kUTok; ++tt) y_acc[tt] += hp * acc[tt];
    }
    for (int tt = 0; tt < ntok; ++tt) {
        const size_t idx = (size_t)(tok0 + tt) * L.d_out + o;
        if (y_fp32)
            static_cast<float *>(y)[idx] = y_acc[tt];
        else
            static_cast<uint16_t *>(y)[idx] = float_to_bf16_bits(y_acc[tt]);
    }
}

}  // namespace

size_t generic_ws_floats(const lb_linear &L, int64_t T) {
    size_t n = 0;
    for (int p = 0; p < L.n_paths; ++p) n += (size_t)T * L.path[p].r;
    return n;
}

cudaError_t launch_generic(const lb_linear &L, const uint16_t *x, int64_t T, void *y, int y_fp32,
                           float *t_acc, int num_sms, cudaStream_t s) {
    LinDesc D = make_desc(L);
    const int t_off1 = (int)((size_t)T * L.path[0].r);
    cudaError_t e = cudaMemsetAsync(t_acc, 0, generic_ws_floats(L, T) * sizeof(float), s);
    if (e != cudaSuccess) return e;
    const int W = L.d_in / 32;
    const int tok_tiles1 = (int)((T + kVTok - 1) / kVTok);
    // enough blocks to fill the GPU, at most 8 words (256 inputs) per block
    int chunk = 8;
    while (chunk > 1 && (long long)((W + chunk - 1) / chunk) * tok_tiles1 * L.n_paths < 2LL * num_sms)
        chunk >>= 1;
    dim3 g1((W + chunk - 1) / chunk, tok_tiles1, L.n_paths);
    size_t sm1 = (size_t)kVTok * chunk * 32 * sizeof(float);
    k_stage1_generic<<<g1, kGenThreads, sm1, s>>>(D, x, (int)T, chunk, t_acc, t_off1);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 g2((L.d_out + kGenThreads - 1) / kGenThreads, (unsigned)((T + kUTok - 1) / kUTok));
    size_t sm2 = 0;
    for (int p = 0; p < L.n_paths; ++p) sm2 += (size_t)kUTok * L.path[p].r * sizeof(float);
    k_stage2_generic<<<g2, kGenThreads, sm2, s>>>(D, (int)T, t_acc, t_off1, y, y_fp32);
    return cudaGetLastError();
}

}  // namespace lb
