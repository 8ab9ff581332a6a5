// lb_qat.cu -- QAT forward and backward of a LittleBit linear on latent
// factors, with SmoothSign (sign in the forward; d tanh(k x)/dx, k = 100, in
// the backward), as the paper trains it (Sec. 4 settings; App. SmoothSign).
//
// Per path, with S the sign (+1 for x >= 0), a = X . g, t = a S(V),
// z = t . l, y = (z S(U)^T) . h, and dY the gradient of the output:
//   forward   t = X Vg,  Vg = diag(g) S(V)          (GEMM)
//             Y += z Uh^T, Uh = diag(h) S(U)          (GEMM)
//   backward  dYz = dY^T z                            (GEMM)
//             dh_o = sum_j S(U)_oj dYz_oj,  dU = h_o dYz_oj k (1 - tanh^2(k U_oj))
//             dz = dY Uh                               (GEMM)
//             dl_j = sum_t dz_tj t_tj,  dt = dz . l
//             XTdt = X^T dt                            (GEMM)
//             dg_i = sum_j S(V)_ij XTdt_ij,  dV = g_i XTdt_ij k (1 - tanh^2(k V_ij))
//             dX += dt Vg^T                            (GEMM)
// The GEMMs run on the tensor cores through cuBLAS (TF32 inputs, fp32
// accumulation: the +-1 factors are exact in TF32, the other operand is
// rounded to 10 mantissa bits); the sign folds, the scalings and the fused
// row / column gradient reductions are the kernels below.
#include <cublas_v2.h>

#include <algorithm>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

__device__ __forceinline__ float sgn(float x) { return x < 0.f ? -1.f : 1.f; }

// Uh[o][j] = h_o S(U_oj) (d_out x r) and Vg[i][j] = g_i S(V_ij) (d_in x r).
__global__ void k_fold_signs(const float *U, const float *V, const float *h, const float *g,
                             int d_out, int d_in, int r, float *Uh, float *Vg) {
    const long long nu = (long long)d_out * r, nv = (long long)d_in * r;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < nu + nv;
         idx += (long long)gridDim.x * blockDim.x) {
        if (idx < nu) Uh[idx] = h[idx / r] * sgn(U[idx]);
        else Vg[idx - nu] = g[(idx - nu) / r] * sgn(V[idx - nu]);
    }
}

// z[t][j] = t[t][j] l_j.
__global__ void k_scale_cols(const float *t, const float *l, long long n, int r, float *z) {
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x)
        z[idx] = t[idx] * l[idx % r];
}

// One warp per row of M (rows x r): out_row[row] = sum_j S(lat_rj) M_rj and
// grad[row][j] = scale_row M_rj k (1 - tanh^2(k lat_rj)).
__global__ void k_grad_rows(const float *M, const float *lat, const float *scale, int rows, int r,
                            float k, float *out_row, float *grad) {
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    const int nw = (gridDim.x * blockDim.x) >> 5;
    for (int row = warp; row < rows; row += nw) {
        const float sc = scale[row];
        float acc = 0.f;
        for (int j = lane; j < r; j += 32) {
            const size_t e = (size_t)row * r + j;
            const float m = M[e], x = lat[e];
            acc += sgn(x) * m;
            const float th = tanhf(k * x);
            grad[e] = sc * m * k * (1.f - th * th);
        }
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) out_row[row] = acc;
    }
}

// dl_j = sum_t dz[t][j] t[t][j] (fp32 partials added with red.add into dl,
// zeroed by the caller), then dz <- dz . l in place.  Threads walk the T x r
// elements; each block adds its column partials once.
__global__ void k_dl_dt(float *dz, const float *t, const float *l, int T, int r, float *dl) {
    extern __shared__ float s_part[];  // [r]
    for (int j = threadIdx.x; j < r; j += blockDim.x) s_part[j] = 0.f;
    __syncthreads();
    const long long n = (long long)T * r;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int j = (int)(idx % r);
        const float d = dz[idx];
        atomicAdd(&s_part[j], d * t[idx]);
        dz[idx] = d * l[j];
    }
    __syncthreads();
    for (int j = threadIdx.x; j < r; j += blockDim.x) red_add_f32(dl + j, s_part[j]);
}

int blocks_for(long long n) { return (int)std::min<long long>((n + 255) / 256, 152 * 8); }

// Row-major C[M][N] = op(A) op(B) (beta C): the column-major GEMM of the
// transposes, C^T = op(B)^T op(A)^T, on TF32 tensor cores.
bool rm_gemm(cublasHandle_t H, bool ta, bool tb, int M, int N, int K, const float *A, int lda,
             const float *B, int ldb, float beta, float *C, int ldc) {
    const float alpha = 1.f;
    return cublasGemmEx(H, tb ? CUBLAS_OP_T : CUBLAS_OP_N, ta ? CUBLAS_OP_T : CUBLAS_OP_N, N, M, K,
                        &alpha, B, CUDA_R_32F, ldb, A, CUDA_R_32F, lda, &beta, C, CUDA_R_32F, ldc,
                        CUBLAS_COMPUTE_32F_FAST_TF32, CUBLAS_GEMM_DEFAULT) == CUBLAS_STATUS_SUCCESS;
}

struct QatBuf {
    float *Uh, *Vg, *t, *z, *dz, *dYz, *XTdt;
};

QatBuf carve(void *ws, int d_in, int d_out, int rmax, long long T) {
    char *p = static_cast<char *>(ws);
    auto take = [&](size_t n) {
        float *r = reinterpret_cast<float *>(p);
        p += (n * sizeof(float) + 255) & ~(size_t)255;
        return r;
    };
    QatBuf b;
    b.Uh = take((size_t)d_out * rmax);
    b.Vg = take((size_t)d_in * rmax);
    b.t = take((size_t)T * rmax);
    b.z = take((size_t)T * rmax);
    b.dz = take((size_t)T * rmax);
    b.dYz = take((size_t)d_out * rmax);
    b.XTdt = take((size_t)d_in * rmax);
    return b;
}

}  // namespace

size_t qat_ws_bytes(int d_in, int d_out, int rmax, long long T) {
    auto sz = [](size_t n) { return (n * sizeof(float) + 255) & ~(size_t)255; };
    return sz((size_t)d_out * rmax) + sz((size_t)d_in * rmax) + 3 * sz((size_t)T * rmax) +
           sz((size_t)d_out * rmax) + sz((size_t)d_in * rmax) + 256;
}

cudaError_t launch_train_forward(const lb_train_linear &L, const float *x, long long T, float *y,
                                 void *ws, cudaStream_t s) {
    cublasHandle_t H = blas_handle();
    if (!H || cublasSetStream(H, s) != CUBLAS_STATUS_SUCCESS) return cudaErrorNotSupported;
    int rmax = 0;
    for (int p = 0; p < L.n_paths; ++p) rmax = std::max(rmax, (int)L.path[p].r);
    QatBuf b = carve(ws, L.d_in, L.d_out, rmax, T);
    bool ok = true;
    for (int p = 0; p < L.n_paths && ok; ++p) {
        const lb_train_path &P = L.path[p];
        const int r = P.r;
        k_fold_signs<<<blocks_for((long long)(L.d_out + L.d_in) * r), 256, 0, s>>>(
            P.u, P.v, P.h, P.g, L.d_out, L.d_in, r, b.Uh, b.Vg);
        ok = ok && rm_gemm(H, false, false, (int)T, r, L.d_in, x, L.d_in, b.Vg, r, 0.f, b.t, r);
        k_scale_cols<<<blocks_for(T * r), 256, 0, s>>>(b.t, P.l, T * r, r, b.z);
        // Y (+)= z Uh^T
        ok = ok && rm_gemm(H, false, true, (int)T, L.d_out, r, b.z, r, b.Uh, r, p ? 1.f : 0.f, y,
                           L.d_out);
    }
    const cudaError_t e = cudaGetLastError();
    return e != cudaSuccess ? e : (ok ? cudaSuccess : cudaErrorUnknown);
}

cudaError_t launch_train_backward(const lb_train_linear &L, const float *x, const float *dy,
                                  long long T, float k, const lb_train_grad *G, float *dx, void *ws,
                                  cudaStream_t s) {
    cublasHandle_t H = blas_handle();
    if (!H || cublasSetStream(H, s) != CUBLAS_STATUS_SUCCESS) return cudaErrorNotSupported;
    int rmax = 0;
    for (int p = 0; p < L.n_paths; ++p) rmax = std::max(rmax, (int)L.path[p].r);
    QatBuf b = carve(ws, L.d_in, L.d_out, rmax, T);
    bool ok = true;
    for (int p = 0; p < L.n_paths && ok; ++p) {
        const lb_train_path &P = L.path[p];
        const lb_train_grad &D = G[p];
        const int r = P.r;
        k_fold_signs<<<blocks_for((long long)(L.d_out + L.d_in) * r), 256, 0, s>>>(
            P.u, P.v, P.h, P.g, L.d_out, L.d_in, r, b.Uh, b.Vg);
        // forward intermediates t = X Vg, z = t . l
        ok = ok && rm_gemm(H, false, false, (int)T, r, L.d_in, x, L.d_in, b.Vg, r, 0.f, b.t, r);
        k_scale_cols<<<blocks_for(T * r), 256, 0, s>>>(b.t, P.l, T * r, r, b.z);
        // dYz = dY^T z -> dh, dU
        ok = ok && rm_gemm(H, true, false, L.d_out, r, (int)T, dy, L.d_out, b.z, r, 0.f, b.dYz, r);
        k_grad_rows<<<blocks_for((long long)L.d_out * 32), 256, 0, s>>>(b.dYz, P.u, P.h, L.d_out, r,
                                                                        k, D.dh, D.du);
        // dz = dY Uh -> dl, dt (in dz)
        ok = ok && rm_gemm(H, false, false, (int)T, r, L.d_out, dy, L.d_out, b.Uh, r, 0.f, b.dz, r);
        cudaMemsetAsync(D.dl, 0, (size_t)r * sizeof(float), s);
        k_dl_dt<<<blocks_for(T * r), 256, (size_t)r * sizeof(float), s>>>(b.dz, b.t, P.l, (int)T,
                                                                           r, D.dl);
        // XTdt = X^T dt -> dg, dV
        ok = ok && rm_gemm(H, true, false, L.d_in, r, (int)T, x, L.d_in, b.dz, r, 0.f, b.XTdt, r);
        k_grad_rows<<<blocks_for((long long)L.d_in * 32), 256, 0, s>>>(b.XTdt, P.v, P.g, L.d_in, r,
                                                                       k, D.dg, D.dv);
        // dX (+)= dt Vg^T
        if (dx)
            ok = ok && rm_gemm(H, false, true, (int)T, L.d_in, r, b.dz, r, b.Vg, r, p ? 1.f : 0.f,
                               dx, L.d_in);
    }
    const cudaError_t e = cudaGetLastError();
    return e != cudaSuccess ? e : (ok ? cudaSuccess : cudaErrorUnknown);
}

}  // namespace lb
