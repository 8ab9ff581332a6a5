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
// Every GEMM runs on the library's own tcgen05 kernel (lb_gemm.cu: TF32
// operands, fp32 accumulation in TMEM; the +-1 factors are exact in TF32, the
// other operand keeps 10 mantissa bits), as C (+)= A B^T with both operands
// K-major.  The sign folds write Uh and Vg in both orientations; the
// products that contract over the tokens (dY^T z, X^T dt) read token-major
// copies of dY, X, z and dt (transposed here); an operand whose rows are not
// 16-byte aligned is copied with a padded leading dimension.  The scalings
// and the fused row / column gradient reductions are the kernels below.
// Workspace: a 256-byte header (its first word is the error word a bounded
// wait records LB_ERR_TIMEOUT in; each call clears it first), then the
// buffers of carve().
#include <algorithm>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

__device__ __forceinline__ float sgn(float x) { return x < 0.f ? -1.f : 1.f; }

// Uh[o][j] = h_o S(U_oj) at ld_r, UhT[j][o] = Uh[o][j] at ld_o, Vg[i][j] =
// g_i S(V_ij) at ld_r and VgT[j][i] at ld_i.
__global__ void k_fold_signs(const float *U, const float *V, const float *h, const float *g,
                             int d_out, int d_in, int r, int ld_r, int ld_o, int ld_i, float *Uh,
                             float *UhT, float *Vg, float *VgT) {
    const long long nu = (long long)d_out * r, nv = (long long)d_in * r;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < nu + nv;
         idx += (long long)gridDim.x * blockDim.x) {
        if (idx < nu) {
            const int o = (int)(idx / r), j = (int)(idx - (long long)o * r);
            const float w = h[o] * sgn(U[idx]);
            Uh[(size_t)o * ld_r + j] = w;
            UhT[(size_t)j * ld_o + o] = w;
        } else {
            const long long q = idx - nu;
            const int i = (int)(q / r), j = (int)(q - (long long)i * r);
            const float w = g[i] * sgn(V[q]);
            Vg[(size_t)i * ld_r + j] = w;
            VgT[(size_t)j * ld_i + i] = w;
        }
    }
}

// dst = src ([rows][cols] at lds) or its transpose ([cols][rows]), at ldd.
// 32 x 32 tiles through shared memory, so both sides move whole rows.
__global__ void k_copy_t(const float *src, int rows, int cols, long long lds, int transpose,
                         float *dst, long long ldd) {
    __shared__ float tile[32][33];
    const int tr = (rows + 31) / 32, tc = (cols + 31) / 32;
    for (long long b = blockIdx.x; b < (long long)tr * tc; b += gridDim.x) {
        const int r0 = (int)(b / tc) * 32, c0 = (int)(b % tc) * 32;
        for (int k = threadIdx.y; k < 32; k += blockDim.y) {
            const int r = r0 + k, c = c0 + threadIdx.x;
            if (r < rows && c < cols) tile[k][threadIdx.x] = src[(size_t)r * lds + c];
        }
        __syncthreads();
        for (int k = threadIdx.y; k < 32; k += blockDim.y) {
            if (transpose) {
                const int c = c0 + k, r = r0 + threadIdx.x;
                if (r < rows && c < cols) dst[(size_t)c * ldd + r] = tile[threadIdx.x][k];
            } else {
                const int r = r0 + k, c = c0 + threadIdx.x;
                if (r < rows && c < cols) dst[(size_t)r * ldd + c] = tile[k][threadIdx.x];
            }
        }
        __syncthreads();
    }
}

// z[t][j] (at ld_z) = t[t][j] l_j, t dense [T][r].
__global__ void k_scale_cols(const float *t, const float *l, long long T, int r, float *z,
                             int ld_z) {
    const long long n = T * r;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long row = idx / r;
        const int j = (int)(idx - row * r);
        z[(size_t)row * ld_z + j] = t[idx] * l[j];
    }
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
long long pad4(long long n) { return (n + 3) & ~3LL; }

// Workspace carve-up (sizes in floats, each buffer 256-byte aligned).
struct QatBuf {
    unsigned *err;
    float *Uh, *UhT, *Vg, *VgT, *t, *z, *zT, *dz, *dtp, *dtT, *dYz, *XTdt, *XT, *dYT, *Xp, *dYp,
        *part;
    size_t part_floats;
    int ldr, ldo, ldi, ldT;
};

struct Carver {
    char *p;
    size_t total = 0;
    float *take(size_t n) {
        float *r = p ? reinterpret_cast<float *>(p + total) : nullptr;
        total += (n * sizeof(float) + 255) & ~(size_t)255;
        return r;
    }
};

QatBuf carve(void *ws, int d_in, int d_out, int rmax, long long T, size_t *bytes) {
    QatBuf b{};
    Carver c{static_cast<char *>(ws)};
    c.total = kWsHeader;
    b.err = ws ? static_cast<unsigned *>(ws) + kErrWord : nullptr;
    b.ldr = (int)pad4(rmax);
    b.ldo = (int)pad4(d_out);
    b.ldi = (int)pad4(d_in);
    b.ldT = (int)pad4(T);
    b.Uh = c.take((size_t)d_out * b.ldr);
    b.UhT = c.take((size_t)rmax * b.ldo);
    b.Vg = c.take((size_t)d_in * b.ldr);
    b.VgT = c.take((size_t)rmax * b.ldi);
    b.t = c.take((size_t)T * rmax);
    b.z = c.take((size_t)T * b.ldr);
    b.zT = c.take((size_t)rmax * b.ldT);
    b.dz = c.take((size_t)T * rmax);
    b.dtp = c.take((size_t)T * b.ldr);
    b.dtT = c.take((size_t)rmax * b.ldT);
    b.dYz = c.take((size_t)d_out * rmax);
    b.XTdt = c.take((size_t)d_in * rmax);
    b.XT = c.take((size_t)d_in * b.ldT);
    b.dYT = c.take((size_t)d_out * b.ldT);
    b.Xp = c.take(d_in % 4 ? (size_t)T * b.ldi : 0);
    b.dYp = c.take(d_out % 4 ? (size_t)T * b.ldo : 0);
    // split-K partials of the largest product (ranks up to rmax)
    const int Ti = (int)T, r = rmax;
    size_t pf = 0;
    pf = std::max(pf, gemm_part_floats(Ti, r, d_in));   // t = X Vg
    pf = std::max(pf, gemm_part_floats(Ti, d_out, r));  // Y = z Uh^T
    pf = std::max(pf, gemm_part_floats(d_out, r, Ti));  // dY^T z
    pf = std::max(pf, gemm_part_floats(Ti, r, d_out));  // dY Uh
    pf = std::max(pf, gemm_part_floats(d_in, r, Ti));   // X^T dt
    pf = std::max(pf, gemm_part_floats(Ti, d_in, r));   // dt Vg^T
    b.part = c.take(pf);
    b.part_floats = pf;
    if (bytes) *bytes = c.total + 256;
    return b;
}

int rmax_of(const lb_train_linear &L) {
    int r = 0;
    for (int p = 0; p < L.n_paths; ++p) r = std::max(r, (int)L.path[p].r);
    return r;
}

cudaError_t copy_t(const float *src, int rows, int cols, long long lds, bool transpose, float *dst,
                   long long ldd, cudaStream_t s) {
    const long long tiles = (long long)((rows + 31) / 32) * ((cols + 31) / 32);
    k_copy_t<<<(int)std::min<long long>(tiles, 152 * 16), dim3(32, 8), 0, s>>>(
        src, rows, cols, lds, transpose ? 1 : 0, dst, ldd);
    return cudaGetLastError();
}

// The operand X (or dY) of the products that contract over its columns: the
// caller's array when its rows are 16-byte aligned, else a padded copy.
cudaError_t k_major(const float *a, int rows, int cols, float *pad, int ldp, GemmOperand *out,
                    cudaStream_t s) {
    if (cols % 4 == 0) {
        *out = GemmOperand{a, rows, cols, cols};
        return cudaSuccess;
    }
    *out = GemmOperand{pad, rows, cols, ldp};
    return copy_t(a, rows, cols, cols, false, pad, ldp, s);
}

// The per-path forward products: t = X Vg, z = t . l, Y (+)= z Uh^T.
cudaError_t path_forward(const lb_train_linear &L, const lb_train_path &P, const GemmOperand &Xk,
                         long long T, float *y, bool accumulate, const QatBuf &b, cudaStream_t s) {
    const int r = P.r;
    k_fold_signs<<<blocks_for((long long)(L.d_out + L.d_in) * r), 256, 0, s>>>(
        P.u, P.v, P.h, P.g, L.d_out, L.d_in, r, b.ldr, b.ldo, b.ldi, b.Uh, b.UhT, b.Vg, b.VgT);
    cudaError_t e = gemm_tf32(Xk, GemmOperand{b.VgT, r, L.d_in, b.ldi}, b.t, r, false, b.part,
                              b.part_floats, b.err, s);
    if (e != cudaSuccess) return e;
    k_scale_cols<<<blocks_for(T * r), 256, 0, s>>>(b.t, P.l, T, r, b.z, b.ldr);
    if (!y) return cudaGetLastError();
    return gemm_tf32(GemmOperand{b.z, (int)T, r, b.ldr}, GemmOperand{b.Uh, L.d_out, r, b.ldr}, y,
                     L.d_out, accumulate, b.part, b.part_floats, b.err, s);
}

}  // namespace

size_t qat_ws_bytes(int d_in, int d_out, int rmax, long long T) {
    size_t bytes = 0;
    carve(nullptr, d_in, d_out, rmax, T, &bytes);
    return bytes;
}

cudaError_t launch_train_forward(const lb_train_linear &L, const float *x, long long T, float *y,
                                 void *ws, cudaStream_t s) {
    QatBuf b = carve(ws, L.d_in, L.d_out, rmax_of(L), T, nullptr);
    cudaError_t e = cudaMemsetAsync(b.err, 0, sizeof(unsigned), s);
    GemmOperand Xk;
    if (e == cudaSuccess) e = k_major(x, (int)T, L.d_in, b.Xp, b.ldi, &Xk, s);
    for (int p = 0; p < L.n_paths && e == cudaSuccess; ++p)
        e = path_forward(L, L.path[p], Xk, T, y, p > 0, b, s);
    return e;
}

cudaError_t launch_train_backward(const lb_train_linear &L, const float *x, const float *dy,
                                  long long T, float k, const lb_train_grad *G, float *dx, void *ws,
                                  cudaStream_t s) {
    QatBuf b = carve(ws, L.d_in, L.d_out, rmax_of(L), T, nullptr);
    const int Ti = (int)T;
    cudaError_t e = cudaMemsetAsync(b.err, 0, sizeof(unsigned), s);
    // the forward's operand, and the token-major copies of X and dY
    GemmOperand Xk, dYk;
    if (e == cudaSuccess) e = k_major(x, Ti, L.d_in, b.Xp, b.ldi, &Xk, s);
    if (e == cudaSuccess) e = k_major(dy, Ti, L.d_out, b.dYp, b.ldo, &dYk, s);
    if (e == cudaSuccess) e = copy_t(x, Ti, L.d_in, L.d_in, true, b.XT, b.ldT, s);
    if (e == cudaSuccess) e = copy_t(dy, Ti, L.d_out, L.d_out, true, b.dYT, b.ldT, s);
    for (int p = 0; p < L.n_paths && e == cudaSuccess; ++p) {
        const lb_train_path &P = L.path[p];
        const lb_train_grad &D = G[p];
        const int r = P.r;
        // forward intermediates t = X Vg, z = t . l (and the fold of this path)
        e = path_forward(L, P, Xk, T, nullptr, false, b, s);
        // dYz = dY^T z -> dh, dU
        if (e == cudaSuccess) e = copy_t(b.z, Ti, r, b.ldr, true, b.zT, b.ldT, s);
        if (e == cudaSuccess)
            e = gemm_tf32(GemmOperand{b.dYT, L.d_out, Ti, b.ldT}, GemmOperand{b.zT, r, Ti, b.ldT},
                          b.dYz, r, false, b.part, b.part_floats, b.err, s);
        if (e != cudaSuccess) break;
        k_grad_rows<<<blocks_for((long long)L.d_out * 32), 256, 0, s>>>(b.dYz, P.u, P.h, L.d_out,
                                                                        r, k, D.dh, D.du);
        // dz = dY Uh -> dl, dt (in dz)
        e = gemm_tf32(dYk, GemmOperand{b.UhT, r, L.d_out, b.ldo}, b.dz, r, false, b.part,
                      b.part_floats, b.err, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(D.dl, 0, (size_t)r * sizeof(float), s);
        if (e != cudaSuccess) break;
        k_dl_dt<<<blocks_for(T * r), 256, (size_t)r * sizeof(float), s>>>(b.dz, b.t, P.l, Ti, r,
                                                                           D.dl);
        // XTdt = X^T dt -> dg, dV
        e = copy_t(b.dz, Ti, r, r, true, b.dtT, b.ldT, s);
        if (e == cudaSuccess)
            e = gemm_tf32(GemmOperand{b.XT, L.d_in, Ti, b.ldT}, GemmOperand{b.dtT, r, Ti, b.ldT},
                          b.XTdt, r, false, b.part, b.part_floats, b.err, s);
        if (e != cudaSuccess) break;
        k_grad_rows<<<blocks_for((long long)L.d_in * 32), 256, 0, s>>>(b.XTdt, P.v, P.g, L.d_in,
                                                                       r, k, D.dg, D.dv);
        // dX (+)= dt Vg^T
        if (dx) {
            GemmOperand dtk{b.dz, Ti, r, r};
            if (r % 4 != 0) {
                e = copy_t(b.dz, Ti, r, r, false, b.dtp, b.ldr, s);
                dtk = GemmOperand{b.dtp, Ti, r, b.ldr};
            }
            if (e == cudaSuccess)
                e = gemm_tf32(dtk, GemmOperand{b.Vg, L.d_in, r, b.ldr}, dx, L.d_in, p > 0, b.part,
                              b.part_floats, b.err, s);
        }
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace lb
