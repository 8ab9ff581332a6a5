// lb_svid.cu -- Dual-SVID initialisation (Sec. 3.2) with Residual
// Compensation (Sec. 3.3) on the GPU.
//
// Per path p (rank r), from the residual R (path 0: W; path p: W minus the
// W_hat of the paths before it, with their scales as stored in fp16):
//   (1) truncated SVD R ~ U_r diag(s) V_r^T by subspace iteration: Q (d_in x k,
//       k = r + oversampling) starts random; each iteration Y = R Q, Y = orth(Y),
//       Q = R^T Y, Q = orth(Q), orth being Cholesky QR (X <- X L^{-T}, G = X^T X
//       = L L^T) with the Gram matrix in fp64 followed by a second pass in
//       fp32; then Rayleigh-Ritz: B = R Q,
//       B = Y' L^T (L the Cholesky factor of B^T B), L^T = U_C diag(s) E^T by
//       one-sided Jacobi (fp32, no squaring of the spectrum), V_r = Q E_r,
//       U_r = B E_r diag(1/s).
//       Sign convention: each v_j has its largest-magnitude entry positive.
//   (2) U' = U_r diag(sqrt s), V' = V_r diag(sqrt s); U_sign = sign(U'),
//       V_sign = sign(V') (sign(0) = +1), packed in the lb_path layouts.
//   (3) |U'| ~ h l_u^T, |V'| ~ g l_v^T, the leading singular pair of each
//       nonnegative matrix by power iteration (fp64, 50 steps), the singular value split
//       evenly; l = l_u . l_v.  h, g, l are rounded to fp16 (nearest even).
// The GEMMs are the library's CUDA-core GEMM (lb_simt_gemm.cu: fp32 / fp64
// FMA, column-major like the matrices here); the Cholesky factor of
// a k x k Gram matrix and the triangular solve with it are blocked (64-wide
// diagonal blocks in one CTA each, rows below by many CTAs, updates by GEMM);
// the k x k Jacobi SVD runs in one CTA; the rest are elementwise / reduction
// kernels below.
#include <algorithm>
#include <cmath>
#include <mutex>
#include <vector>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kOversample = 8;
constexpr int kPowerIters = 50;  // rank-1 power iterations on |U'|, |V'|
constexpr int kJacobiSweeps = 40;
constexpr int kSmallThreads = 1024;
constexpr int kMaxK = 1024 + 16;  // rank + oversampling

// Sum of v over the block, returned to every thread (blockDim.x <= 1024).
__device__ double block_sum_d(double v) {
    __shared__ double s_part[32];
    __shared__ double s_total;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) s_part[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const int nw = (blockDim.x + 31) >> 5;
        double t = lane < nw ? s_part[lane] : 0.0;
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) s_total = t;
    }
    __syncthreads();
    const double total = s_total;
    __syncthreads();
    return total;
}

// ---------------------------------------------------------------- random start

// Q[i] uniform in [-1, 1) from a 64-bit counter hash (splitmix64 finaliser).
__global__ void k_rand(float *Q, long long n, unsigned long long seed) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        unsigned long long z = seed + 0x9E3779B97F4A7C15ull * (unsigned long long)(i + 1);
        z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
        z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
        z ^= z >> 31;
        Q[i] = (float)((double)(z >> 11) * (1.0 / 9007199254740992.0) * 2.0 - 1.0);
    }
}

__global__ void k_to_f64(const float *a, double *b, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x)
        b[i] = (double)a[i];
}

// ---------------------------------------------------------------- Cholesky QR

// ---------------------------------------------------------------- blocked Cholesky

constexpr int kNB = 64;  // block width of the blocked Cholesky / triangular solve

// floor = eps_rel * trace(G) / k (one block): pivots at or below it count as zero.
template <typename T>
__global__ void k_pivot_floor(const T *G, int k, T eps_rel, T *floor_out) {
    T acc = 0;
    for (int j = threadIdx.x; j < k; j += blockDim.x) acc += G[(size_t)j * k + j];
    __shared__ T s_part[32];
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        T t = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += s_part[w];
        *floor_out = eps_rel * (t > 0 ? t : 0) / k;
    }
}

// Factor the diagonal block G[jb:jb+b, jb:jb+b] (already updated by the
// blocks to its left) in place, lower triangle, in shared memory; one CTA of
// kNB threads.  A pivot at or below *floor becomes 0, and so does the column
// below it.
template <typename T>
__global__ void __launch_bounds__(kNB) k_potrf_diag(T *G, int k, int jb, int b, const T *floor_p) {
    __shared__ T a[kNB][kNB + 1];
    const int c = threadIdx.x;
    for (int i = 0; i < b; ++i)
        if (c < b) a[i][c] = G[(size_t)(jb + c) * k + jb + i];
    __syncthreads();
    const T fl = *floor_p;
    for (int j = 0; j < b; ++j) {
        if (c == 0) {
            T d = a[j][j];
            for (int p = 0; p < j; ++p) d -= a[j][p] * a[j][p];
            a[j][j] = d > fl && d > 0 ? sqrt(d) : 0;
        }
        __syncthreads();
        const T piv = a[j][j];
        if (c > j && c < b) {
            T v = a[c][j];
            for (int p = 0; p < j; ++p) v -= a[c][p] * a[j][p];
            a[c][j] = piv > 0 ? v / piv : 0;
        }
        __syncthreads();
    }
    for (int i = 0; i < b; ++i)
        if (c < b && c <= i) G[(size_t)(jb + c) * k + jb + i] = a[i][c];
}

// Panel rows i in [jb+b, k): L[i, jb:jb+b] = G[i, jb:jb+b] L_jj^{-T}, one
// thread per row, L_jj in shared memory (column-major G).
template <typename T>
__global__ void k_trsm_panel(T *G, int k, int jb, int b) {
    __shared__ T l[kNB][kNB + 1];
    for (int idx = threadIdx.x; idx < b * b; idx += blockDim.x) {
        const int i = idx / b, j = idx % b;
        l[i][j] = j <= i ? G[(size_t)(jb + j) * k + jb + i] : 0;
    }
    __syncthreads();
    const int i = jb + b + blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= k) return;
    T x[kNB];
#pragma unroll 4
    for (int j = 0; j < kNB; ++j) {
        if (j >= b) break;
        T v = G[(size_t)(jb + j) * k + i];
        for (int p = 0; p < j; ++p) v -= x[p] * l[j][p];
        x[j] = l[j][j] > 0 ? v / l[j][j] : 0;
        G[(size_t)(jb + j) * k + i] = x[j];
    }
}

// In-place rows of X (rows x k column-major, fp32): columns jb:jb+b solved
// against L_jj^T, x L_jj^T = y, one thread per row (the columns left of jb
// have been subtracted by a GEMM already).  L is fp32 column-major k x k.
__global__ void k_trsm_cols(float *X, int rows, const float *L, int k, int jb, int b) {
    __shared__ float l[kNB][kNB + 1];
    for (int idx = threadIdx.x; idx < b * b; idx += blockDim.x) {
        const int i = idx / b, j = idx % b;
        l[i][j] = j <= i ? L[(size_t)(jb + j) * k + jb + i] : 0.f;
    }
    __syncthreads();
    const int row = blockIdx.x * blockDim.x + threadIdx.x;
    if (row >= rows) return;
    float x[kNB];
#pragma unroll 4
    for (int j = 0; j < kNB; ++j) {
        if (j >= b) break;
        float v = X[(size_t)(jb + j) * rows + row];
        for (int p = 0; p < j; ++p) v -= x[p] * l[j][p];
        x[j] = l[j][j] > 0.f ? v / l[j][j] : 0.f;
        X[(size_t)(jb + j) * rows + row] = x[j];
    }
}

// fp32 copy of the lower triangle of G (zeros above), column-major; with
// transpose, Lt = L^T instead.
template <typename T>
__global__ void k_lower_f32(const T *G, int k, float *L, int transpose) {
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < (long long)k * k;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx / k), i = (int)(idx % k);  // column c, row i of the output
        const int gi = transpose ? c : i, gc = transpose ? i : c;  // element (gi, gc) of L
        L[idx] = gi >= gc ? (float)G[(size_t)gc * k + gi] : 0.f;
    }
}

// ---------------------------------------------------------------- Jacobi eigen

// SVD of a small square A (k x k, fp32, column-major, overwritten) by
// one-sided Jacobi: plane rotations of column pairs until the columns are
// mutually orthogonal (A V = U diag(s), the rotations accumulated in V).
// Round-robin pairing: each round rotates k/2 disjoint pairs, one warp per
// pair, so the rounds need one CTA barrier each.  For columns x, y with
// alpha = |x|^2, beta = |y|^2, gamma = x.y, t is the smaller root of
// t^2 + 2 zeta t - 1 = 0, zeta = (beta - alpha) / (2 gamma), and
// x' = c x - s y, y' = s x + c y.  Outputs s (k, decreasing, fp64) and the
// right singular vectors E (fp32, k x k column-major, column j for s[j]).
// Pairs within 1e-6 of orthogonal are left alone; sweeps stop when no pair
// of a sweep is more than 4e-6 from orthogonal (fp32 dot products of length
// k carry ~sqrt(k) 6e-8 of noise) or after kJacobiSweeps.  One CTA; V is fp32 scratch (k x k).
__global__ void __launch_bounds__(kSmallThreads) k_svd_jacobi(float *A, float *V, int k, double *sv,
                                                              float *E) {
    __shared__ float s_off[32];
    __shared__ int s_done;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    const int kk = (k + 1) & ~1;  // even count: index k is a dummy when k is odd
    for (int idx = threadIdx.x; idx < k * k; idx += blockDim.x)
        V[idx] = (idx / k == idx % k) ? 1.f : 0.f;
    __syncthreads();
    for (int sweep = 0; sweep < kJacobiSweeps; ++sweep) {
        float off = 0.f;
        for (int round = 0; round < kk - 1; ++round) {
            for (int t = warp; t < kk / 2; t += nwarps) {
                int a = t == 0 ? 0 : 1 + (t - 1 + round) % (kk - 1);
                int b = 1 + (kk - 2 - t + round) % (kk - 1);
                if (a > b) { const int x = a; a = b; b = x; }
                if (b >= k) continue;
                float *xa = A + (size_t)a * k, *xb = A + (size_t)b * k;
                float al = 0.f, be = 0.f, ga = 0.f;
                for (int i = lane; i < k; i += 32) {
                    al += xa[i] * xa[i];
                    be += xb[i] * xb[i];
                    ga += xa[i] * xb[i];
                }
                for (int o = 16; o > 0; o >>= 1) {
                    al += __shfl_xor_sync(0xffffffffu, al, o);
                    be += __shfl_xor_sync(0xffffffffu, be, o);
                    ga += __shfl_xor_sync(0xffffffffu, ga, o);
                }
                const float rel = (al > 0.f && be > 0.f) ? fabsf(ga) / sqrtf(al * be) : 0.f;
                off = fmaxf(off, rel);
                if (rel <= 1e-6f) continue;
                const float zeta = (be - al) / (2.f * ga);
                const float tt = (zeta >= 0.f ? 1.f : -1.f) / (fabsf(zeta) + sqrtf(1.f + zeta * zeta));
                const float c = 1.f / sqrtf(1.f + tt * tt), sn = c * tt;
                for (int i = lane; i < k; i += 32) {
                    const float x = xa[i], y = xb[i];
                    xa[i] = c * x - sn * y;
                    xb[i] = sn * x + c * y;
                    const float vx = V[(size_t)a * k + i], vy = V[(size_t)b * k + i];
                    V[(size_t)a * k + i] = c * vx - sn * vy;
                    V[(size_t)b * k + i] = sn * vx + c * vy;
                }
            }
            __syncthreads();
        }
        for (int o = 16; o > 0; o >>= 1) off = fmaxf(off, __shfl_xor_sync(0xffffffffu, off, o));
        if (lane == 0) s_off[warp] = off;
        __syncthreads();
        if (threadIdx.x == 0) {
            float m = 0.f;
            for (int w = 0; w < nwarps; ++w) m = fmaxf(m, s_off[w]);
            s_done = m <= 4e-6f;
        }
        __syncthreads();
        if (s_done) break;
    }
    // singular values (column norms), sorted by rank (ties by index)
    __shared__ double s_norm[kMaxK];
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        double ss = 0.0;
        for (int i = 0; i < k; ++i) ss += (double)A[(size_t)j * k + i] * A[(size_t)j * k + i];
        s_norm[j] = sqrt(ss);
    }
    __syncthreads();
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        const double sj = s_norm[j];
        int rank = 0;
        for (int i = 0; i < k; ++i) {
            const double si = s_norm[i];
            rank += (si > sj) || (si == sj && i < j);
        }
        sv[rank] = sj;
        for (int i = 0; i < k; ++i) E[(size_t)rank * k + i] = V[(size_t)j * k + i];
    }
}

// ---------------------------------------------------------------- Ritz vectors

// U (m x r, column-major) /= s_j (0 where s_j = 0).
__global__ void k_ritz_scale(const double *s, float *U, int m, int r) {
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < (long long)m * r;
         idx += (long long)gridDim.x * blockDim.x) {
        const double sj = s[idx / m];
        U[idx] = sj > 0.0 ? (float)((double)U[idx] / sj) : 0.0f;
    }
}

// Sign convention and the even split: for column j, the entry of V (n x r)
// of largest magnitude (first on a tie) decides a joint sign; then
// U' = sign * U * sqrt(s_j), V' = sign * V * sqrt(s_j).  One block per column.
__global__ void k_sign_split(float *U, float *V, int m, int n, const double *s) {
    const int j = blockIdx.x;
    __shared__ float s_v[32];
    __shared__ int s_i[32];
    float best = -1.f;
    int bi = 0x7fffffff;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const float a = fabsf(V[(size_t)j * n + i]);
        if (a > best || (a == best && i < bi)) {
            best = a;
            bi = i;
        }
    }
    for (int o = 16; o > 0; o >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ob > best || (ob == best && oi < bi)) {
            best = ob;
            bi = oi;
        }
    }
    if ((threadIdx.x & 31) == 0) {
        s_v[threadIdx.x >> 5] = best;
        s_i[threadIdx.x >> 5] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
            if (s_v[w] > s_v[0] || (s_v[w] == s_v[0] && s_i[w] < s_i[0])) {
                s_v[0] = s_v[w];
                s_i[0] = s_i[w];
            }
    }
    __syncthreads();
    const int imax = s_i[0];
    const float sg = (imax < n && V[(size_t)j * n + imax] < 0.f) ? -1.f : 1.f;
    __syncthreads();
    const float f = sg * (float)sqrt(s[j]);
    for (int i = threadIdx.x; i < n; i += blockDim.x) V[(size_t)j * n + i] *= f;
    for (int i = threadIdx.x; i < m; i += blockDim.x) U[(size_t)j * m + i] *= f;
}

// ---------------------------------------------------------------- signs

// u_bits[o][w] from U' (d_out x r, column-major): bit k = U'(o, 32w + k) < 0.
__global__ void k_pack_u_cm(const float *U, int d_out, int r, uint32_t *u_bits) {
    const int R = (r + 31) >> 5;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < (long long)d_out * R;
         idx += (long long)gridDim.x * blockDim.x) {
        const int o = (int)(idx / R), w = (int)(idx % R);
        uint32_t word = 0;
        for (int b = 0; b < 32 && 32 * w + b < r; ++b)
            if (U[(size_t)(32 * w + b) * d_out + o] < 0.f) word |= 1u << b;
        u_bits[idx] = word;
    }
}

// v_bits[w][j] from V' (d_in x r, column-major): bit k = V'(32w + k, j) < 0.
__global__ void k_pack_v_cm(const float *V, int d_in, int r, uint32_t *v_bits) {
    const int W = (d_in + 31) >> 5;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < (long long)W * r;
         idx += (long long)gridDim.x * blockDim.x) {
        const int w = (int)(idx / r), j = (int)(idx % r);
        uint32_t word = 0;
        for (int b = 0; b < 32 && 32 * w + b < d_in; ++b)
            if (V[(size_t)j * d_in + 32 * w + b] < 0.f) word |= 1u << b;
        v_bits[idx] = word;
    }
}

// ---------------------------------------------------------------- rank-1 of |M|

// y[i] = sum_j |M(i, j)| x[j], M rows x cols column-major; one thread per row.
__global__ void k_abs_mv(const float *M, int rows, int cols, const double *x, double *y) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < rows; i += gridDim.x * blockDim.x) {
        double acc = 0.0;
        for (int j = 0; j < cols; ++j) acc += fabs((double)M[(size_t)j * rows + i]) * x[j];
        y[i] = acc;
    }
}

// x[j] = sum_i |M(i, j)| y[i]; one block per column.
__global__ void k_abs_mtv(const float *M, int rows, const double *y, double *x) {
    const int j = blockIdx.x;
    double acc = 0.0;
    for (int i = threadIdx.x; i < rows; i += blockDim.x)
        acc += fabs((double)M[(size_t)j * rows + i]) * y[i];
    acc = block_sum_d(acc);
    if (threadIdx.x == 0) x[j] = acc;
}

// v <- v / |v| (one block); the norm goes to *nrm.
__global__ void k_normalize(double *v, int n, double *nrm) {
    double ss = 0.0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) ss += v[i] * v[i];
    ss = block_sum_d(ss);
    const double nv = sqrt(ss);
    for (int i = threadIdx.x; i < n; i += blockDim.x) v[i] = nv > 0.0 ? v[i] / nv : 0.0;
    if (threadIdx.x == 0) *nrm = nv;
}

__global__ void k_fill(double *v, int n, double val) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) v[i] = val;
}

// a = sqrt(sigma) u as fp16 (a zero sigma gives zeros); optionally keep the
// fp64 values in keep[] as well.
__global__ void k_split_half(const double *u, int n, const double *sigma, uint16_t *out,
                             double *keep) {
    const double sq = sqrt(fmax(*sigma, 0.0));
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const double a = *sigma > 0.0 ? sq * u[i] : 0.0;
        if (keep) keep[i] = a;
        else out[i] = __half_as_ushort(__double2half(a));
    }
}

// l = l_u . l_v as fp16.
__global__ void k_latent_half(const double *lu, const double *lv, int r, uint16_t *l) {
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < r; j += gridDim.x * blockDim.x)
        l[j] = __half_as_ushort(__double2half(lu[j] * lv[j]));
}

// ---------------------------------------------------------------- residual

// A1 (d_out x r, cm) = h_o * sign(U'(o, j)) * l_j, B1 (d_in x r, cm) =
// g_i * sign(V'(i, j)), from the stored fp16 scales, so that
// W_hat = A1 B1^T (Eq. 4).
__global__ void k_what_factors(const float *U, const float *V, int d_out, int d_in, int r,
                               const uint16_t *h, const uint16_t *g, const uint16_t *l, float *A1,
                               float *B1) {
    const long long na = (long long)d_out * r, nb = (long long)d_in * r;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < na + nb;
         idx += (long long)gridDim.x * blockDim.x) {
        if (idx < na) {
            const int j = (int)(idx / d_out), o = (int)(idx % d_out);
            const float sg = U[idx] < 0.f ? -1.f : 1.f;
            A1[idx] = half_bits_to_float(h[o]) * sg * half_bits_to_float(l[j]);
        } else {
            const long long e = idx - na;
            const int i = (int)(e % d_in);
            const float sg = V[e] < 0.f ? -1.f : 1.f;
            B1[e] = half_bits_to_float(g[i]) * sg;
        }
    }
}

// ---------------------------------------------------------------- the driver

int grid_for(long long n) { return (int)std::min<long long>((n + 255) / 256, 152 * 8); }

struct Buf {
    char *p;
    size_t off = 0;
    template <class T>
    T *take(size_t n) {
        T *r = reinterpret_cast<T *>(p + off);
        off += (n * sizeof(T) + 255) & ~(size_t)255;
        return r;
    }
};

}  // namespace

int svid_k(int r, int d_out, int d_in) { return std::min(r + kOversample, std::min(d_out, d_in)); }

size_t svid_ws_bytes(int d_out, int d_in, const int *ranks, int n_paths) {
    int kmax = 0;
    for (int p = 0; p < n_paths; ++p) kmax = std::max(kmax, svid_k(ranks[p], d_out, d_in));
    Buf b{nullptr};
    const size_t m = (size_t)d_out, n = (size_t)d_in, k = (size_t)kmax;
    b.take<float>(m * n);                  // R (residual, column-major n x m = row-major W)
    b.take<float>(n * k);                  // Q
    b.take<float>(n * k);                  // Q2
    b.take<float>(m * k);                  // Y
    b.take<float>(m * k);                  // Y2
    b.take<double>(std::max(m, n) * k);    // fp64 copy for the Gram matrix
    b.take<double>(k * k);                 // G (fp64 Gram)
    b.take<float>(k * k);                  // G32 (fp32 Gram / L^T)
    b.take<float>(k * k);                  // fp32 scratch (Jacobi V)
    b.take<float>(k * k);                  // L (fp32) / E
    b.take<double>(k);                     // s
    b.take<double>(m + n);                 // power iteration y
    b.take<double>(2 * k);                 // x, l_u / l_v (fp64)
    b.take<double>(4);                     // norms
    return b.off + 256;
}

cudaError_t launch_dual_svid(const float *W, int d_out, int d_in, int n_paths, const int *ranks,
                             uint32_t *const *v_bits, uint32_t *const *u_bits, uint16_t *const *g,
                             uint16_t *const *l, uint16_t *const *h, int iters, void *ws,
                             cudaStream_t s) {
    const int m = d_out, n = d_in;
    int kmax = 0;
    for (int p = 0; p < n_paths; ++p) kmax = std::max(kmax, svid_k(ranks[p], d_out, d_in));
    Buf b{static_cast<char *>(ws)};
    float *R = b.take<float>((size_t)m * n);
    float *Q = b.take<float>((size_t)n * kmax);
    float *Q2 = b.take<float>((size_t)n * kmax);
    float *Y = b.take<float>((size_t)m * kmax);
    float *Y2 = b.take<float>((size_t)m * kmax);
    double *D = b.take<double>((size_t)std::max(m, n) * kmax);
    double *G = b.take<double>((size_t)kmax * kmax);
    float *G32 = b.take<float>((size_t)kmax * kmax);
    float *JV32 = b.take<float>((size_t)kmax * kmax);
    float *Lt = b.take<float>((size_t)kmax * kmax);
    double *sv = b.take<double>(kmax);
    double *py = b.take<double>((size_t)m + n);
    double *px = b.take<double>(2 * (size_t)kmax);
    double *nrm = b.take<double>(4);
    // R = W (row-major m x n is the column-major n x m matrix R^T)
    cudaError_t e = cudaMemcpyAsync(R, W, (size_t)m * n * sizeof(float), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
    const float one = 1.f, zero = 0.f, minus = -1.f;
    (void)G32;
    const double done = 1.0, dzero = 0.0;
    bool blas_ok = true;
    constexpr bool N_ = false, T_ = true;  // op(X) = X, op(X) = X^T
    auto gemm = [&](bool ta, bool tb, int mm, int nn, int kk, const float *A, int lda,
                    const float *B, int ldb, const float *beta, float *C, int ldc,
                    const float *alpha) {
        blas_ok = blas_ok &&
                  gemm_simt(ta, tb, mm, nn, kk, *alpha, A, lda, B, ldb, *beta, C, ldc, s) ==
                      cudaSuccess;
    };
    // blocked Cholesky of the k x k Gram matrix Gm (lower, in place): per
    // 64-wide block, the diagonal block in one CTA, the rows below it by a
    // triangular solve, the trailing matrix by a GEMM
    double *dfloor = reinterpret_cast<double *>(nrm + 2);
    float *ffloor = reinterpret_cast<float *>(nrm + 3);
    auto chol64 = [&](double *Gm, int k) {
        k_pivot_floor<double><<<1, 256, 0, s>>>(Gm, k, 1e-14, dfloor);
        for (int jb = 0; jb < k; jb += kNB) {
            const int bw = std::min(kNB, k - jb), rest = k - jb - bw;
            k_potrf_diag<double><<<1, kNB, 0, s>>>(Gm, k, jb, bw, dfloor);
            if (rest > 0) {
                k_trsm_panel<double><<<(rest + 127) / 128, 128, 0, s>>>(Gm, k, jb, bw);
                blas_ok = blas_ok &&
                          gemm_simt(N_, T_, rest, rest, bw, -1.0, Gm + (size_t)jb * k + jb + bw, k,
                                    Gm + (size_t)jb * k + jb + bw, k, done,
                                    Gm + (size_t)(jb + bw) * k + jb + bw, k, s) == cudaSuccess;
            }
        }
    };
    auto chol32 = [&](float *Gm, int k) {
        k_pivot_floor<float><<<1, 256, 0, s>>>(Gm, k, 1e-6f, ffloor);
        for (int jb = 0; jb < k; jb += kNB) {
            const int bw = std::min(kNB, k - jb), rest = k - jb - bw;
            k_potrf_diag<float><<<1, kNB, 0, s>>>(Gm, k, jb, bw, ffloor);
            if (rest > 0) {
                k_trsm_panel<float><<<(rest + 127) / 128, 128, 0, s>>>(Gm, k, jb, bw);
                gemm(N_, T_, rest, rest, bw, Gm + (size_t)jb * k + jb + bw, k,
                     Gm + (size_t)jb * k + jb + bw, k, &one, Gm + (size_t)(jb + bw) * k + jb + bw,
                     k, &minus);
            }
        }
    };
    // X (rows x k) <- X L^{-T} in place, block column by block column
    auto trsm_right = [&](float *X, int rows, const float *L32, int k) {
        for (int jb = 0; jb < k; jb += kNB) {
            const int bw = std::min(kNB, k - jb);
            if (jb > 0)
                gemm(N_, T_, rows, bw, jb, X, rows, L32 + jb, k, &one,
                     X + (size_t)jb * rows, rows, &minus);
            k_trsm_cols<<<(rows + 127) / 128, 128, 0, s>>>(X, rows, L32, k, jb, bw);
        }
    };
    // orthonormalise the columns of X (rows x k, column-major) in place:
    // Cholesky QR with the Gram matrix in fp64 (the pass that copes with the
    // conditioning of X), then once more in fp32 on the nearly orthonormal
    // result
    auto orth = [&](float *X, float *, int rows, int k) {
        k_to_f64<<<grid_for((long long)rows * k), 256, 0, s>>>(X, D, (long long)rows * k);
        blas_ok = blas_ok &&
                  gemm_simt(T_, N_, k, k, rows, done, D, rows, D, rows, dzero, G, k, s) ==
                      cudaSuccess;
        chol64(G, k);
        k_lower_f32<double><<<grid_for((long long)k * k), 256, 0, s>>>(G, k, Lt, 0);
        trsm_right(X, rows, Lt, k);
        gemm(T_, N_, k, k, rows, X, rows, X, rows, &zero, G32, k, &one);
        chol32(G32, k);
        k_lower_f32<float><<<grid_for((long long)k * k), 256, 0, s>>>(G32, k, Lt, 0);
        trsm_right(X, rows, Lt, k);
    };
    for (int p = 0; p < n_paths && blas_ok; ++p) {
        const int r = ranks[p], k = svid_k(r, m, n);
        k_rand<<<grid_for((long long)n * k), 256, 0, s>>>(Q, (long long)n * k,
                                                          0x5EEDull + 7919ull * (unsigned)p);
        orth(Q, Q2, n, k);
        for (int it = 0; it < iters; ++it) {
            // Y = R Q  (R is n x m column-major: op T gives m x n)
            gemm(T_, N_, m, k, n, R, n, Q, n, &zero, Y, m, &one);
            orth(Y, Y2, m, k);
            // Q = R^T Y
            gemm(N_, N_, n, k, m, R, n, Y, m, &zero, Q, n, &one);
            orth(Q, Q2, n, k);
        }
        // Rayleigh-Ritz: B = R Q (in Y); B = Y' L^T with L the Cholesky factor
        // of B^T B (fp64); the SVD of the k x k L^T (one-sided Jacobi) gives
        // B's singular values and right vectors E: V_r = Q E_r, U_r = B E_r / s
        gemm(T_, N_, m, k, n, R, n, Q, n, &zero, Y, m, &one);
        k_to_f64<<<grid_for((long long)m * k), 256, 0, s>>>(Y, D, (long long)m * k);
        blas_ok = blas_ok &&
                  gemm_simt(T_, N_, k, k, m, done, D, m, D, m, dzero, G, k, s) == cudaSuccess;
        chol64(G, k);
        k_lower_f32<double><<<grid_for((long long)k * k), 256, 0, s>>>(G, k, G32, 1);
        k_svd_jacobi<<<1, kSmallThreads, 0, s>>>(G32, JV32, k, sv, Lt);
        gemm(N_, N_, n, r, k, Q, n, Lt, k, &zero, Q2, n, &one);
        gemm(N_, N_, m, r, k, Y, m, Lt, k, &zero, Y2, m, &one);
        k_ritz_scale<<<grid_for((long long)m * r), 256, 0, s>>>(sv, Y2, m, r);
        k_sign_split<<<r, 256, 0, s>>>(Y2, Q2, m, n, sv);
        k_pack_u_cm<<<grid_for((long long)m * ((r + 31) / 32)), 256, 0, s>>>(Y2, m, r, u_bits[p]);
        k_pack_v_cm<<<grid_for((long long)((n + 31) / 32) * r), 256, 0, s>>>(Q2, n, r, v_bits[p]);
        // rank-1 of |U'| (m x r) and |V'| (n x r): power iteration from x = 1
        double *lu = px, *lv = px + kmax;
        for (int side = 0; side < 2; ++side) {
            const float *M = side == 0 ? Y2 : Q2;
            const int rows = side == 0 ? m : n;
            k_fill<<<1, 256, 0, s>>>(px + side * kmax, r, 1.0 / sqrt((double)r));
            double *x = px + side * kmax;
            for (int it = 0; it < kPowerIters; ++it) {
                k_abs_mv<<<grid_for(rows), 256, 0, s>>>(M, rows, r, x, py);
                k_normalize<<<1, 1024, 0, s>>>(py, rows, nrm);
                k_abs_mtv<<<r, 256, 0, s>>>(M, rows, py, x);
                k_normalize<<<1, 1024, 0, s>>>(x, r, nrm + 1);
            }
            // x = v (unit), py = u (unit), sigma = |M^T u| in nrm[1]
            if (side == 0) {
                k_split_half<<<grid_for(rows), 256, 0, s>>>(py, rows, nrm + 1, h[p], nullptr);
                k_split_half<<<1, 256, 0, s>>>(x, r, nrm + 1, nullptr, lu);
            } else {
                k_split_half<<<grid_for(rows), 256, 0, s>>>(py, rows, nrm + 1, g[p], nullptr);
                k_split_half<<<1, 256, 0, s>>>(x, r, nrm + 1, nullptr, lv);
            }
        }
        k_latent_half<<<1, 256, 0, s>>>(lu, lv, r, l[p]);
        if (p + 1 < n_paths) {
            // R <- R - W_hat_p: R^T (n x m) -= B1 A1^T with A1 = h.U_sign.l, B1 = g.V_sign
            float *A1 = Y, *B1 = Q;
            k_what_factors<<<grid_for((long long)(m + n) * r), 256, 0, s>>>(Y2, Q2, m, n, r, h[p],
                                                                             g[p], l[p], A1, B1);
            gemm(N_, T_, n, m, r, B1, n, A1, m, &one, R, n, &minus);
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return blas_ok ? cudaSuccess : cudaErrorUnknown;
}

}  // namespace lb
