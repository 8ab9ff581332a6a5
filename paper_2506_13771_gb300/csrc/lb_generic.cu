// lb_generic.cu -- any-T LittleBit forward on CUDA cores, two launches.
//
// Prop. 1 (LittleBit, arXiv 2506.13771), per path p:
//   stage 1  z_p[tok][j] = l_p[j] * sum_i V_p,sign[i][j] * g_p[i] * X[tok][i]
//   stage 2  Y[tok][o]  += h_p[o] * sum_j U_p,sign[o][j] * z_p[tok][j]
// and Eq. 6 sums the paths.  z is the latent state of Sec. 5 (KV cache
// compression), kept as [T][r_0 + r_1] with path 1 after path 0.  Stage 1
// splits d_in over blocks and reduces into an fp32 z with red.add (l folded
// into each partial sum); stage 2 reads a finished z, fp32 or fp16.  This is
// the path for token counts the decode and tensor-core kernels do not take,
// and the latent / expansion entry points use the two stages on their own.
#include "lb_common.cuh"
#include "lb_kernels.h"

#include <algorithm>

namespace lb {

namespace {

constexpr int kGenThreads = 256;
constexpr int kVTok = 8;   // tokens per stage-1 block
constexpr int kUTok = 4;   // tokens per stage-2 block

// grid: (word chunks of d_in, token tiles, paths).  z: fp32 [T][n1], zeroed.
__global__ void __launch_bounds__(kGenThreads)
k_stage1_generic(LinDesc L, const uint16_t *__restrict__ x, int T, int chunk_words,
                 float *__restrict__ z, int n1) {
    extern __shared__ float s_a[];  // [kVTok][chunk_words*32]
    const int p = blockIdx.z;
    const int r = p == 0 ? L.r[0] : L.r[1];
    const int W = L.d_in >> 5;
    const int w0 = blockIdx.x * chunk_words;
    const int nw = min(chunk_words, W - w0);
    const int tok0 = blockIdx.y * kVTok;
    const int ntok = min(kVTok, T - tok0);
    const int n_in = nw * 32;
    const uint16_t *g = p == 0 ? L.g[0] : L.g[1];
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
    float *z_p = z + (p == 0 ? 0 : L.r[0]);
    const uint32_t *V = p == 0 ? L.v[0] : L.v[1];
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
        const float lj = half_bits_to_float((p == 0 ? L.l[0] : L.l[1])[j]);
#pragma unroll
        for (int tt = 0; tt < kVTok; ++tt)
            if (tt < ntok) red_add_f32(z_p + (size_t)(tok0 + tt) * n1 + j, lj * acc[tt]);
    }
}

// grid: (row blocks of d_out, token tiles).  z: [T][n1], fp32 or fp16 (z_half).
__global__ void __launch_bounds__(kGenThreads)
k_stage2_generic(LinDesc L, int T, const void *__restrict__ z, int z_half, int n1, void *y,
                 int y_fp32) {
    extern __shared__ float s_z[];  // [paths][kUTok][r_p]
    const int tok0 = blockIdx.y * kUTok;
    const int ntok = min(kUTok, T - tok0);
    for (int p = 0; p < L.n_paths; ++p) {
        const int r = p == 0 ? L.r[0] : L.r[1];
        const int c0 = p == 0 ? 0 : L.r[0];
        float *s_zp = s_z + (p == 0 ? 0 : kUTok * L.r[0]);
        for (int e = threadIdx.x; e < kUTok * r; e += blockDim.x) {
            const int tt = e / r, j = e - tt * r;
            float v = 0.f;
            if (tt < ntok) {
                const size_t idx = (size_t)(tok0 + tt) * n1 + c0 + j;
                v = z_half ? half_bits_to_float(static_cast<const uint16_t *>(z)[idx])
                           : __ldcg(static_cast<const float *>(z) + idx);
            }
            s_zp[e] = v;
        }
    }
    __syncthreads();
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= L.d_out) return;
    float y_acc[kUTok];
#pragma unroll
    for (int tt = 0; tt < kUTok; ++tt) y_acc[tt] = 0.f;
    for (int p = 0; p < L.n_paths; ++p) {
        const int r = p == 0 ? L.r[0] : L.r[1];
        const int R = (r + 31) >> 5;
        const uint32_t *U = (p == 0 ? L.u[0] : L.u[1]) + (size_t)o * R;
        float acc[kUTok];
#pragma unroll
        for (int tt = 0; tt < kUTok; ++tt) acc[tt] = 0.f;
        for (int w = 0; w < R; ++w) {
            const uint32_t word = __ldg(U + w);
            const int nb = min(32, r - 32 * w);
            const float *zw = s_z + (p == 0 ? 0 : kUTok * L.r[0]) + 32 * w;
            for (int k = 0; k < nb; ++k) {
#pragma unroll
                for (int tt = 0; tt < kUTok; ++tt) acc[tt] += apply_sign(zw[tt * r + k], word, k);
            }
        }
        const float hp = half_bits_to_float((p == 0 ? L.h[0] : L.h[1])[o]);
#pragma unroll
        for (int tt = 0; tt < kUTok; ++tt) y_acc[tt] += hp * acc[tt];
    }
#pragma unroll
    for (int tt = 0; tt < kUTok; ++tt) {
        if (tt >= ntok) break;
        const size_t idx = (size_t)(tok0 + tt) * L.d_out + o;
        if (y_fp32)
            static_cast<float *>(y)[idx] = y_acc[tt];
        else
            static_cast<uint16_t *>(y)[idx] = float_to_bf16_bits(y_acc[tt]);
    }
}

// z16[i] = fp16(z32[i]), round to nearest even.
__global__ void k_to_half(const float *__restrict__ z32, uint16_t *__restrict__ z16, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x)
        z16[i] = __half_as_ushort(__float2half_rn(z32[i]));
}

int n1_of(const lb_linear &L) {
    int n1 = 0;
    for (int p = 0; p < L.n_paths; ++p) n1 += L.path[p].r;
    return n1;
}

}  // namespace

size_t generic_ws_floats(const lb_linear &L, int64_t T) { return (size_t)T * n1_of(L); }

cudaError_t launch_latent_generic(const lb_linear &L, const uint16_t *x, int64_t T, float *z32,
                                  int num_sms, cudaStream_t s) {
    LinDesc D = make_desc(L);
    const int n1 = n1_of(L);
    cudaError_t e = cudaMemsetAsync(z32, 0, (size_t)T * n1 * sizeof(float), s);
    if (e != cudaSuccess) return e;
    const int W = L.d_in / 32;
    const int tok_tiles1 = (int)((T + kVTok - 1) / kVTok);
    // enough blocks to fill the GPU, at most 8 words (256 inputs) per block
    int chunk = 8;
    while (chunk > 1 && (long long)((W + chunk - 1) / chunk) * tok_tiles1 * L.n_paths < 2LL * num_sms)
        chunk >>= 1;
    dim3 g1((W + chunk - 1) / chunk, tok_tiles1, L.n_paths);
    size_t sm1 = (size_t)kVTok * chunk * 32 * sizeof(float);
    k_stage1_generic<<<g1, kGenThreads, sm1, s>>>(D, x, (int)T, chunk, z32, n1);
    return cudaGetLastError();
}

cudaError_t launch_expand_generic(const lb_linear &L, const void *z, int z_half, int64_t T,
                                  void *y, int y_fp32, cudaStream_t s) {
    LinDesc D = make_desc(L);
    dim3 g2((L.d_out + kGenThreads - 1) / kGenThreads, (unsigned)((T + kUTok - 1) / kUTok));
    size_t sm2 = 0;
    for (int p = 0; p < L.n_paths; ++p) sm2 += (size_t)kUTok * L.path[p].r * sizeof(float);
    k_stage2_generic<<<g2, kGenThreads, sm2, s>>>(D, (int)T, z, z_half, n1_of(L), y, y_fp32);
    return cudaGetLastError();
}

cudaError_t launch_to_half(const float *z32, uint16_t *z16, long long n, cudaStream_t s) {
    const int blocks = (int)std::min<long long>((n + 255) / 256, 148 * 8);
    k_to_half<<<blocks, 256, 0, s>>>(z32, z16, n);
    return cudaGetLastError();
}

cudaError_t launch_generic(const lb_linear &L, const uint16_t *x, int64_t T, void *y, int y_fp32,
                           float *z_ws, int num_sms, cudaStream_t s) {
    cudaError_t e = launch_latent_generic(L, x, T, z_ws, num_sms, s);
    if (e != cudaSuccess) return e;
    return launch_expand_generic(L, z_ws, 0, T, y, y_fp32, s);
}

}  // namespace lb
