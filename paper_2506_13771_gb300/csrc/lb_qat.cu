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

// Columns [c0, c0 + r) of one path-concatenated sign factor: F[i][c0 + j] =
// s_i S(L_ij) at ld (L the latent [rows][r], s the row scale) and its
// transpose FT[c0 + j][i] at ldt, in 64 x 64 tiles through shared memory so
// that every read and both writes move whole rows.
__global__ void __launch_bounds__(256) k_fold_signs(const float *Lat, const float *sc, int rows,
                                                     int r, int c0, int ld, int ldt, float *F,
                                                     float *FT) {
    __shared__ float tile[64][65];
    const int tx = threadIdx.x & 63, ty = threadIdx.x >> 6;  // 64 x 4
    const int tr = (rows + 63) / 64, tc = (r + 63) / 64;
    for (long long b = blockIdx.x; b < (long long)tr * tc; b += gridDim.x) {
        const int i0 = (int)(b / tc) * 64, j0 = (int)(b % tc) * 64;
#pragma unroll 4
        for (int k = ty; k < 64; k += 4) {
            const int i = i0 + k, j = j0 + tx;
            if (i < rows && j < r) {
                const float w = sc[i] * sgn(Lat[(size_t)i * r + j]);
                F[(size_t)i * ld + c0 + j] = w;
                tile[k][tx] = w;
            }
        }
        __syncthreads();
#pragma unroll 4
        for (int k = ty; k < 64; k += 4) {
            const int j = j0 + k, i = i0 + tx;
            if (i < rows && j < r) FT[(size_t)(c0 + j) * ldt + i] = tile[tx][k];
        }
        __syncthreads();
    }
}

// dst = src ([rows][cols] at lds) or its transpose ([cols][rows]), at ldd.
// 64 x 64 tiles through shared memory, so both sides move whole rows.
__global__ void __launch_bounds__(256) k_copy_t(const float *src, int rows, int cols,
                                                 long long lds, int transpose, float *dst,
                                                 long long ldd) {
    __shared__ float tile[64][65];
    const int tx = threadIdx.x & 63, ty = threadIdx.x >> 6;  // 64 x 4
    const int tr = (rows + 63) / 64, tc = (cols + 63) / 64;
    for (long long b = blockIdx.x; b < (long long)tr * tc; b += gridDim.x) {
        const int r0 = (int)(b / tc) * 64, c0 = (int)(b % tc) * 64;
#pragma unroll 4
        for (int k = ty; k < 64; k += 4) {
            const int rr = r0 + k, c = c0 + tx;
            if (rr < rows && c < cols) tile[k][tx] = src[(size_t)rr * lds + c];
        }
        __syncthreads();
#pragma unroll 4
        for (int k = ty; k < 64; k += 4) {
            if (transpose) {
                const int c = c0 + k, rr = r0 + tx;
                if (rr < rows && c < cols) dst[(size_t)c * ldd + rr] = tile[tx][k];
            } else {
                const int rr = r0 + k, c = c0 + tx;
                if (rr < rows && c < cols) dst[(size_t)rr * ldd + c] = tile[k][tx];
            }
        }
        __syncthreads();
    }
}

// One warp per row of M's columns [c0, c0 + r) (M: rows x R, dense): the
// path's out_row[row] = sum_j S(lat_rj) M_r,c0+j and grad[row][j] = scale_row
// M_r,c0+j k (1 - tanh^2(k lat_rj)) (lat, grad: rows x r).  Four columns per
// lane in flight.
__global__ void __launch_bounds__(256) k_grad_rows(const float *M, int R, int c0,
                                                   const float *lat, const float *scale, int rows,
                                                   int r, float k, float *out_row, float *grad) {
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    const int nw = (gridDim.x * blockDim.x) >> 5;
    for (int row = warp; row < rows; row += nw) {
        const float sc = scale[row];
        const float *Mr = M + (size_t)row * R + c0;
        const float *Lr = lat + (size_t)row * r;
        float *Gr = grad + (size_t)row * r;
        float acc = 0.f;
#pragma unroll 4
        for (int j = lane; j < r; j += 32) {
            const float m = Mr[j], x = Lr[j];
            acc += sgn(x) * m;
            const float th = tanhf(k * x);
            Gr[j] = sc * m * k * (1.f - th * th);
        }
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) out_row[row] = acc;
    }
}

// dl_j = sum_t dz[t][j] t[t][j] over the concatenated columns: thread j of a
// block sums its column over the block's run of rows in a register and adds
// it to dl (zeroed by the caller) once.
__global__ void __launch_bounds__(256) k_dl(const float *dz, const float *t, int T, int R,
                                            int rows_per, float *dl) {
    const int j = blockIdx.x * 256 + threadIdx.x;
    if (j >= R) return;
    const int t0 = blockIdx.y * rows_per, t1 = min(T, t0 + rows_per);
    float acc = 0.f;
#pragma unroll 4
    for (int q = t0; q < t1; ++q) acc += dz[(size_t)q * R + j] * t[(size_t)q * R + j];
    red_add_f32(dl + j, acc);
}

int blocks_for(long long n) { return (int)std::min<long long>((n + 255) / 256, 152 * 8); }
long long pad4(long long n) { return (n + 3) & ~3LL; }

// Workspace carve-up (each buffer 256-byte aligned).  R = the paths' ranks
// concatenated (Eq. 6 sums the paths, so both GEMMs of a product take the
// paths side by side: the path sum is their K dimension, or their outputs
// sit side by side).
struct QatBuf {
    unsigned *err;
    float *Uh, *UhT, *Vg, *VgT, *lc, *dlc, *t, *z, *zT, *dz, *dt, *dtT, *dYz, *XTdt, *XT, *dYT,
        *Xp, *dYp, *part;
    size_t part_floats;
    int R, ldr, ldo, ldi, ldT;
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

QatBuf carve(void *ws, int d_in, int d_out, int R, long long T, size_t *bytes) {
    QatBuf b{};
    Carver c{static_cast<char *>(ws)};
    c.total = kWsHeader;
    b.err = ws ? static_cast<unsigned *>(ws) + kErrWord : nullptr;
    b.R = R;
    b.ldr = (int)pad4(R);
    b.ldo = (int)pad4(d_out);
    b.ldi = (int)pad4(d_in);
    b.ldT = (int)pad4(T);
    b.Uh = c.take((size_t)d_out * b.ldr);
    b.UhT = c.take((size_t)R * b.ldo);
    b.Vg = c.take((size_t)d_in * b.ldr);
    b.VgT = c.take((size_t)R * b.ldi);
    b.lc = c.take((size_t)R);
    b.dlc = c.take((size_t)R);
    b.t = c.take((size_t)T * R);
    b.z = c.take((size_t)T * b.ldr);
    b.zT = c.take((size_t)R * b.ldT);
    b.dz = c.take((size_t)T * R);
    b.dt = c.take((size_t)T * b.ldr);
    b.dtT = c.take((size_t)R * b.ldT);
    b.dYz = c.take((size_t)d_out * R);
    b.XTdt = c.take((size_t)d_in * R);
    b.XT = c.take((size_t)d_in * b.ldT);
    b.dYT = c.take((size_t)d_out * b.ldT);
    b.Xp = c.take(d_in % 4 ? (size_t)T * b.ldi : 0);
    b.dYp = c.take(d_out % 4 ? (size_t)T * b.ldo : 0);
    // split-K partials of the largest product
    const int Ti = (int)T;
    size_t pf = 0;
    pf = std::max(pf, gemm_part_floats(Ti, R, d_in));   // t = X Vg
    pf = std::max(pf, gemm_part_floats(Ti, d_out, R));  // Y = z Uh^T
    pf = std::max(pf, gemm_part_floats(d_out, R, Ti));  // dY^T z
    pf = std::max(pf, gemm_part_floats(Ti, R, d_out));  // dY Uh
    pf = std::max(pf, gemm_part_floats(d_in, R, Ti));   // X^T dt
    pf = std::max(pf, gemm_part_floats(Ti, d_in, R));   // dt Vg^T
    b.part = c.take(pf);
    b.part_floats = pf;
    if (bytes) *bytes = c.total + 256;
    return b;
}

int rsum_of(const lb_train_linear &L) {
    int r = 0;
    for (int p = 0; p < L.n_paths; ++p) r += (int)L.path[p].r;
    return r;
}

cudaError_t copy_t(const float *src, int rows, int cols, long long lds, bool transpose, float *dst,
                   long long ldd, cudaStream_t s) {
    const long long tiles = (long long)((rows + 63) / 64) * ((cols + 63) / 64);
    k_copy_t<<<(int)std::min<long long>(tiles, 152 * 8), 256, 0, s>>>(
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

// The sign folds of every path side by side (Uh and UhT, Vg and VgT) and the
// concatenated l; then t = X Vg and z = t . l.
cudaError_t forward_latent(const lb_train_linear &L, const GemmOperand &Xk, long long T,
                           const QatBuf &b, cudaStream_t s) {
    int c0 = 0;
    cudaError_t e = cudaSuccess;
    for (int p = 0; p < L.n_paths && e == cudaSuccess; ++p) {
        const lb_train_path &P = L.path[p];
        const int tu = ((L.d_out + 63) / 64) * ((P.r + 63) / 64);
        const int tv = ((L.d_in + 63) / 64) * ((P.r + 63) / 64);
        k_fold_signs<<<std::min(tu, 152 * 8), 256, 0, s>>>(P.u, P.h, L.d_out, P.r, c0, b.ldr,
                                                           b.ldo, b.Uh, b.UhT);
        k_fold_signs<<<std::min(tv, 152 * 8), 256, 0, s>>>(P.v, P.g, L.d_in, P.r, c0, b.ldr,
                                                           b.ldi, b.Vg, b.VgT);
        e = cudaMemcpyAsync(b.lc + c0, P.l, (size_t)P.r * sizeof(float), cudaMemcpyDeviceToDevice,
                            s);
        c0 += P.r;
    }
    // t = X Vg, and z = t . l beside it
    if (e == cudaSuccess)
        e = gemm_tf32(Xk, GemmOperand{b.VgT, b.R, L.d_in, b.ldi}, b.t, b.R, false, b.part,
                      b.part_floats, b.err, s, b.z, b.lc, b.ldr);
    return e;
}

// The workspace's record of the forward it holds (header words kPlanWord ..
// + 1): written by a forward, compared by a backward that reuses its state
// (a mismatch records LB_ERR_PLAN).
__global__ void k_qat_tag(unsigned *ws_words, unsigned long long tag, int check) {
    unsigned long long *w = reinterpret_cast<unsigned long long *>(ws_words + kPlanWord);
    if (!check)
        *w = tag;
    else if (*w != tag)
        atomicCAS(ws_words + kErrWord, 0u, static_cast<unsigned>(LB_ERR_PLAN));
}

}  // namespace

size_t qat_ws_bytes(int d_in, int d_out, int rsum, long long T) {
    size_t bytes = 0;
    carve(nullptr, d_in, d_out, rsum, T, &bytes);
    return bytes;
}

cudaError_t launch_train_forward(const lb_train_linear &L, const float *x, long long T, float *y,
                                 void *ws, unsigned long long tag, cudaStream_t s) {
    QatBuf b = carve(ws, L.d_in, L.d_out, rsum_of(L), T, nullptr);
    cudaError_t e = cudaMemsetAsync(b.err, 0, sizeof(unsigned), s);
    GemmOperand Xk;
    if (e == cudaSuccess) e = k_major(x, (int)T, L.d_in, b.Xp, b.ldi, &Xk, s);
    if (e == cudaSuccess) e = forward_latent(L, Xk, T, b, s);
    // Y = z Uh^T: both paths in one product (Eq. 6's sum is its K dimension)
    if (e == cudaSuccess)
        e = gemm_tf32(GemmOperand{b.z, (int)T, b.R, b.ldr}, GemmOperand{b.Uh, L.d_out, b.R, b.ldr},
                      y, L.d_out, false, b.part, b.part_floats, b.err, s);
    // the folds, l, t and z stay in the workspace for a backward that reuses them
    if (e == cudaSuccess) {
        k_qat_tag<<<1, 1, 0, s>>>(static_cast<unsigned *>(ws), tag, 0);
        e = cudaGetLastError();
    }
    return e;
}

cudaError_t launch_train_backward(const lb_train_linear &L, const float *x, const float *dy,
                                  long long T, float k, const lb_train_grad *G, float *dx, void *ws,
                                  bool saved, unsigned long long tag, cudaStream_t s) {
    QatBuf b = carve(ws, L.d_in, L.d_out, rsum_of(L), T, nullptr);
    const int Ti = (int)T, R = b.R;
    cudaError_t e = cudaMemsetAsync(b.err, 0, sizeof(unsigned), s);
    // the forward's operand, the token-major copies of X and dY, t and z
    GemmOperand Xk, dYk;
    if (e == cudaSuccess) e = k_major(x, Ti, L.d_in, b.Xp, b.ldi, &Xk, s);
    if (e == cudaSuccess) e = k_major(dy, Ti, L.d_out, b.dYp, b.ldo, &dYk, s);
    if (e == cudaSuccess) e = copy_t(x, Ti, L.d_in, L.d_in, true, b.XT, b.ldT, s);
    if (e == cudaSuccess) e = copy_t(dy, Ti, L.d_out, L.d_out, true, b.dYT, b.ldT, s);
    if (e == cudaSuccess) {
        if (saved) {
            // the forward's folds, l, t and z, if the workspace holds this forward
            k_qat_tag<<<1, 1, 0, s>>>(static_cast<unsigned *>(ws), tag, 1);
            e = cudaGetLastError();
        } else {
            e = forward_latent(L, Xk, T, b, s);
        }
    }
    // dYz = dY^T z -> dh, dU per path
    if (e == cudaSuccess) e = copy_t(b.z, Ti, R, b.ldr, true, b.zT, b.ldT, s);
    if (e == cudaSuccess)
        e = gemm_tf32(GemmOperand{b.dYT, L.d_out, Ti, b.ldT}, GemmOperand{b.zT, R, Ti, b.ldT},
                      b.dYz, R, false, b.part, b.part_floats, b.err, s);
    if (e != cudaSuccess) return e;
    for (int p = 0, c0 = 0; p < L.n_paths; c0 += L.path[p].r, ++p)
        k_grad_rows<<<blocks_for((long long)L.d_out * 32), 256, 0, s>>>(
            b.dYz, R, c0, L.path[p].u, L.path[p].h, L.d_out, L.path[p].r, k, G[p].dh, G[p].du);
    // dz = dY Uh and dt = dz . l beside it -> dl
    e = gemm_tf32(dYk, GemmOperand{b.UhT, R, L.d_out, b.ldo}, b.dz, R, false, b.part,
                  b.part_floats, b.err, s, b.dt, b.lc, b.ldr);
    if (e == cudaSuccess) e = cudaMemsetAsync(b.dlc, 0, (size_t)R * sizeof(float), s);
    if (e != cudaSuccess) return e;
    {
        const int rows_per = 64;
        k_dl<<<dim3((R + 255) / 256, (Ti + rows_per - 1) / rows_per), 256, 0, s>>>(
            b.dz, b.t, Ti, R, rows_per, b.dlc);
    }
    for (int p = 0, c0 = 0; p < L.n_paths && e == cudaSuccess; c0 += L.path[p].r, ++p)
        e = cudaMemcpyAsync(G[p].dl, b.dlc + c0, (size_t)L.path[p].r * sizeof(float),
                            cudaMemcpyDeviceToDevice, s);
    // XTdt = X^T dt -> dg, dV per path
    if (e == cudaSuccess) e = copy_t(b.dt, Ti, R, b.ldr, true, b.dtT, b.ldT, s);
    if (e == cudaSuccess)
        e = gemm_tf32(GemmOperand{b.XT, L.d_in, Ti, b.ldT}, GemmOperand{b.dtT, R, Ti, b.ldT},
                      b.XTdt, R, false, b.part, b.part_floats, b.err, s);
    if (e != cudaSuccess) return e;
    for (int p = 0, c0 = 0; p < L.n_paths; c0 += L.path[p].r, ++p)
        k_grad_rows<<<blocks_for((long long)L.d_in * 32), 256, 0, s>>>(
            b.XTdt, R, c0, L.path[p].v, L.path[p].g, L.d_in, L.path[p].r, k, G[p].dg, G[p].dv);
    // dX = dt Vg^T: both paths in one product
    if (dx)
        e = gemm_tf32(GemmOperand{b.dt, Ti, R, b.ldr}, GemmOperand{b.Vg, L.d_in, R, b.ldr}, dx,
                      L.d_in, false, b.part, b.part_floats, b.err, s);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace lb
