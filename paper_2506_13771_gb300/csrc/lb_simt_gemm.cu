// lb_simt_gemm.cu -- column-major C = alpha op(A) op(B) + beta C in fp32 or
// fp64 on the CUDA cores (FMA, the precision of the type), for the Dual-SVID
// initialisation (lb_svid.cu): its subspace iteration, Gram matrices,
// Cholesky updates and Ritz rotations need full fp32 / fp64 products, which
// the tensor cores do not give (FP64 and TF32 fall short), and they run once
// per weight, offline.
//
// op(A) is M x K: A[m + k lda] (no transpose) or A[k + m lda] (transpose);
// op(B) is K x N likewise; C[m + n ldc].  One CTA computes a 64 x 64 tile of
// C with 256 threads (4 x 4 outputs each), staging 16-deep K slices of op(A)
// and op(B) in shared memory; alpha and beta are host scalars (beta = 0 does
// not read C).  When the tiles of C are too few for the SMs and K is long
// (the Gram matrices and Cholesky updates: k x k over thousands of rows), K
// is split over blockIdx.z: C is scaled by beta first and every slice adds
// alpha times its partial with atomics (the order of those additions, and so
// the last bits of C, may vary from run to run).
#include <algorithm>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int ST = 64;  // tile
constexpr int SK = 16;  // K slice

template <typename T>
__global__ void __launch_bounds__(256) k_gemm_simt(int M, int N, int K, T alpha, const T *A,
                                                   long long lda, int ta, const T *B,
                                                   long long ldb, int tb, T beta, T *C,
                                                   long long ldc, int split) {
    __shared__ T As[SK][ST + 1];  // As[k][m]
    __shared__ T Bs[SK][ST + 1];  // Bs[k][n]
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int m0 = blockIdx.x * ST, n0 = blockIdx.y * ST;
    T acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = T(0);
    // this slice's K range, in whole SK steps
    const int ks = (K + SK - 1) / SK;
    const int kb = (int)((long long)blockIdx.z * ks / split) * SK;
    const int ke = min(K, (int)((long long)(blockIdx.z + 1) * ks / split) * SK);
    for (int k0 = kb; k0 < ke; k0 += SK) {
        // 64 x 16 elements of each operand, 4 per thread; consecutive threads
        // walk the operand's contiguous dimension
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int idx = tid + 256 * q;
            if (!ta) {  // A[m + k lda]: m contiguous
                const int mm = idx & 63, kk = idx >> 6;
                const int gm = m0 + mm, gk = k0 + kk;
                As[kk][mm] = gm < M && gk < ke ? A[gm + (long long)gk * lda] : T(0);
            } else {    // A[k + m lda]: k contiguous
                const int kk = idx & 15, mm = idx >> 4;
                const int gm = m0 + mm, gk = k0 + kk;
                As[kk][mm] = gm < M && gk < ke ? A[gk + (long long)gm * lda] : T(0);
            }
            if (!tb) {  // B[k + n ldb]: k contiguous
                const int kk = idx & 15, nn = idx >> 4;
                const int gn = n0 + nn, gk = k0 + kk;
                Bs[kk][nn] = gn < N && gk < ke ? B[gk + (long long)gn * ldb] : T(0);
            } else {    // B[n + k ldb]: n contiguous
                const int nn = idx & 63, kk = idx >> 6;
                const int gn = n0 + nn, gk = k0 + kk;
                Bs[kk][nn] = gn < N && gk < ke ? B[gn + (long long)gk * ldb] : T(0);
            }
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < SK; ++kk) {
            T a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][tx + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][ty + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fma(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int gn = n0 + ty + 16 * j;
        if (gn >= N) continue;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int gm = m0 + tx + 16 * i;
            if (gm >= M) continue;
            T *c = C + gm + (long long)gn * ldc;
            if (split > 1)
                atomicAdd(c, alpha * acc[i][j]);  // C already holds beta C
            else
                *c = beta == T(0) ? alpha * acc[i][j] : fma(alpha, acc[i][j], beta * *c);
        }
    }
}

// C = beta C (M x N at ldc).
template <typename T>
__global__ void k_scale_c(int M, int N, T beta, T *C, long long ldc) {
    const long long n = (long long)M * N;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const long long col = i / M;
        T *c = C + (i - col * M) + col * ldc;
        *c = beta == T(0) ? T(0) : beta * *c;
    }
}

template <typename T>
cudaError_t gemm_simt_t(bool ta, bool tb, int M, int N, int K, T alpha, const T *A, long long lda,
                        const T *B, long long ldb, T beta, T *C, long long ldc, cudaStream_t s) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    const int gx = (M + ST - 1) / ST, gy = (N + ST - 1) / ST;
    // slices of at least 256 K each, until about two CTAs per SM
    const int target = 2 * 152;
    int split = 1;
    if (gx * gy < target) split = std::max(1, std::min(target / (gx * gy), K / 256));
    if (split > 1) {
        const long long n = (long long)M * N;
        k_scale_c<T><<<(int)std::min<long long>((n + 255) / 256, 152 * 8), 256, 0, s>>>(M, N, beta,
                                                                                       C, ldc);
    }
    const dim3 grid((unsigned)gx, (unsigned)gy, (unsigned)split);
    k_gemm_simt<T><<<grid, 256, 0, s>>>(M, N, K, alpha, A, lda, ta ? 1 : 0, B, ldb, tb ? 1 : 0,
                                         beta, C, ldc, split);
    return cudaGetLastError();
}

}  // namespace

cudaError_t gemm_simt(bool ta, bool tb, int M, int N, int K, float alpha, const float *A,
                      long long lda, const float *B, long long ldb, float beta, float *C,
                      long long ldc, cudaStream_t s) {
    return gemm_simt_t<float>(ta, tb, M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, s);
}

cudaError_t gemm_simt(bool ta, bool tb, int M, int N, int K, double alpha, const double *A,
                      long long lda, const double *B, long long ldb, double beta, double *C,
                      long long ldc, cudaStream_t s) {
    return gemm_simt_t<double>(ta, tb, M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, s);
}

}  // namespace lb
