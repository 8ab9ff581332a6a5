/*
 * lb_oracle.c -- plain fp64 CPU oracle for the LittleBit linear forward.
 *
 * TEST INFRASTRUCTURE ONLY (see lb_oracle.h): never called by the product
 * path.  Written for obviousness, not speed: each function follows one
 * definition of the paper, in the paper's order, with plain loops.  The only
 * parallelism is an OpenMP split over independent output elements; every
 * individual sum is accumulated sequentially, so results are deterministic.
 */
#include "lb_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* Number formats                                                           */
/* ------------------------------------------------------------------------ */

/* IEEE 754 binary16: sign(1) exponent(5, bias 15) fraction(10).
 *   e == 0       : (-1)^s * f * 2^-24            (subnormal, includes zero)
 *   e == 31      : inf (f == 0) or NaN
 *   otherwise    : (-1)^s * (1024 + f) * 2^(e-25) */
double lbo_half_to_double(uint16_t bits)
{
    int s = (bits >> 15) & 1;
    int e = (bits >> 10) & 0x1f;
    int f = bits & 0x3ff;
    double v;
    if (e == 0)
        v = ldexp((double)f, -24);
    else if (e == 31)
        v = f ? NAN : INFINITY;
    else
        v = ldexp((double)(1024 + f), e - 25);
    return s ? -v : v;
}

/* bfloat16: sign(1) exponent(8, bias 127) fraction(7).
 *   e == 0       : (-1)^s * f * 2^-133           (subnormal, includes zero)
 *   e == 255     : inf (f == 0) or NaN
 *   otherwise    : (-1)^s * (128 + f) * 2^(e-134) */
double lbo_bf16_to_double(uint16_t bits)
{
    int s = (bits >> 15) & 1;
    int e = (bits >> 7) & 0xff;
    int f = bits & 0x7f;
    double v;
    if (e == 0)
        v = ldexp((double)f, -133);
    else if (e == 255)
        v = f ? NAN : INFINITY;
    else
        v = ldexp((double)(128 + f), e - 134);
    return s ? -v : v;
}

/* ------------------------------------------------------------------------ */
/* Bit packing (Eq. 2 signs, 32 per uint32, bit = 1 <=> -1, LSB first)       */
/* ------------------------------------------------------------------------ */

static int64_t words_for(int64_t n) { return (n + 31) / 32; }

int lbo_pack_u(const int8_t *signs, int64_t rows, int64_t cols, uint32_t *out)
{
    int64_t nw = words_for(cols);
    for (int64_t o = 0; o < rows; o++) {
        for (int64_t w = 0; w < nw; w++) {
            uint32_t word = 0;
            for (int k = 0; k < 32; k++) {
                int64_t c = 32 * w + k;
                if (c >= cols)
                    break;
                int8_t v = signs[o * cols + c];
                if (v == -1)
                    word |= (uint32_t)1 << k;
                else if (v != 1)
                    return -1;
            }
            out[o * nw + w] = word;
        }
    }
    return 0;
}

int lbo_pack_v(const int8_t *signs, int64_t rows, int64_t cols, uint32_t *out)
{
    int64_t nw = words_for(rows);
    for (int64_t w = 0; w < nw; w++) {
        for (int64_t j = 0; j < cols; j++) {
            uint32_t word = 0;
            for (int k = 0; k < 32; k++) {
                int64_t i = 32 * w + k;
                if (i >= rows)
                    break;
                int8_t v = signs[i * cols + j];
                if (v == -1)
                    word |= (uint32_t)1 << k;
                else if (v != 1)
                    return -1;
            }
            out[w * cols + j] = word;
        }
    }
    return 0;
}

/* Sign of U_sign[o][j] read straight from the U words. */
static int sign_u(const uint32_t *words, int64_t r, int64_t o, int64_t j)
{
    uint32_t word = words[o * words_for(r) + j / 32];
    return ((word >> (j % 32)) & 1u) ? -1 : 1;
}

/* Sign of V_sign[i][j] read straight from the V words. */
static int sign_v(const uint32_t *words, int64_t r, int64_t i, int64_t j)
{
    uint32_t word = words[(i / 32) * r + j];
    return ((word >> (i % 32)) & 1u) ? -1 : 1;
}

void lbo_unpack_u(const uint32_t *words, int64_t rows, int64_t cols, int8_t *signs)
{
    for (int64_t o = 0; o < rows; o++)
        for (int64_t j = 0; j < cols; j++)
            signs[o * cols + j] = (int8_t)sign_u(words, cols, o, j);
}

void lbo_unpack_v(const uint32_t *words, int64_t rows, int64_t cols, int8_t *signs)
{
    for (int64_t i = 0; i < rows; i++)
        for (int64_t j = 0; j < cols; j++)
            signs[i * cols + j] = (int8_t)sign_v(words, cols, i, j);
}

/* ------------------------------------------------------------------------ */
/* Forward                                                                  */
/* ------------------------------------------------------------------------ */

static double *decode_bf16_array(const uint16_t *x, int64_t n)
{
    double *v = (double *)malloc((size_t)(n > 0 ? n : 1) * sizeof(double));
    if (!v)
        return NULL;
    for (int64_t i = 0; i < n; i++)
        v[i] = lbo_bf16_to_double(x[i]);
    return v;
}

/* Dense mode.  W[o][i] = sum_p h_p[o] * sum_j U_p[o][j] l_p[j] V_p[i][j] g_p[i]
 * (Eq. 4, Eq. 5 summed as Eq. 6), then Y[t][o] = sum_i X[t][i] W[o][i]. */
int lbo_forward_dense(const lbo_linear *L, const uint16_t *x, int64_t T, double *y)
{
    int64_t din = L->d_in, dout = L->d_out;
    double *W = (double *)calloc((size_t)(din * dout > 0 ? din * dout : 1), sizeof(double));
    double *X = decode_bf16_array(x, T * din);
    if (!W || !X) {
        free(W);
        free(X);
        return -1;
    }
    for (int p = 0; p < L->n_paths; p++) {
        const lbo_path *P = &L->path[p];
        int64_t r = P->r;
        double *l = (double *)malloc((size_t)(r > 0 ? r : 1) * sizeof(double));
        if (!l) {
            free(W);
            free(X);
            return -1;
        }
        for (int64_t j = 0; j < r; j++)
            l[j] = lbo_half_to_double(P->l[j]);
#pragma omp parallel for schedule(static)
        for (int64_t o = 0; o < dout; o++) {
            double ho = lbo_half_to_double(P->h[o]);
            for (int64_t i = 0; i < din; i++) {
                double gi = lbo_half_to_double(P->g[i]);
                double s = 0.0;
                for (int64_t j = 0; j < r; j++)
                    s += sign_u(P->u_words, r, o, j) * l[j] * sign_v(P->v_words, r, i, j);
                W[o * din + i] += ho * s * gi;
            }
        }
        free(l);
    }
#pragma omp parallel for schedule(static)
    for (int64_t to = 0; to < T * dout; to++) {
        int64_t t = to / dout, o = to % dout;
        double s = 0.0;
        for (int64_t i = 0; i < din; i++)
            s += X[t * din + i] * W[o * din + i];
        y[to] = s;
    }
    free(W);
    free(X);
    return 0;
}

/* Factored mode (Prop. 1), one path at a time, paths summed (Eq. 6):
 *   a = X . g                      (broadcast over rows of X)
 *   t = a V_sign                   [T][r]
 *   z = t . l
 *   y += (z U_sign^T) . h          [T][d_out] */
int lbo_apply_factored(const lbo_linear *L, const double *X, int64_t T, double *y,
                       double *t_out)
{
    int64_t din = L->d_in, dout = L->d_out;
    for (int64_t k = 0; k < T * dout; k++)
        y[k] = 0.0;
    int64_t t_off = 0;
    for (int p = 0; p < L->n_paths; p++) {
        const lbo_path *P = &L->path[p];
        int64_t r = P->r;
        double *a = (double *)malloc((size_t)(T * din > 0 ? T * din : 1) * sizeof(double));
        double *t = (double *)malloc((size_t)(T * r > 0 ? T * r : 1) * sizeof(double));
        if (!a || !t) {
            free(a);
            free(t);
            return -1;
        }
        for (int64_t tt = 0; tt < T; tt++)
            for (int64_t i = 0; i < din; i++)
                a[tt * din + i] = X[tt * din + i] * lbo_half_to_double(P->g[i]);
#pragma omp parallel for schedule(static)
        for (int64_t tj = 0; tj < T * r; tj++) {
            int64_t tt = tj / r, j = tj % r;
            double s = 0.0;
            for (int64_t i = 0; i < din; i++)
                s += a[tt * din + i] * sign_v(P->v_words, r, i, j);
            t[tj] = s;
        }
        if (t_out) {
            memcpy(t_out + t_off, t, (size_t)(T * r) * sizeof(double));
            t_off += T * r;
        }
        for (int64_t tj = 0; tj < T * r; tj++)
            t[tj] *= lbo_half_to_double(P->l[tj % r]);
#pragma omp parallel for schedule(static)
        for (int64_t to = 0; to < T * dout; to++) {
            int64_t tt = to / dout, o = to % dout;
            double s = 0.0;
            for (int64_t j = 0; j < r; j++)
                s += t[tt * r + j] * sign_u(P->u_words, r, o, j);
            y[to] += s * lbo_half_to_double(P->h[o]);
        }
        free(a);
        free(t);
    }
    return 0;
}

int lbo_forward_factored(const lbo_linear *L, const uint16_t *x, int64_t T, double *y)
{
    double *X = decode_bf16_array(x, T * L->d_in);
    if (!X)
        return -1;
    int rc = lbo_apply_factored(L, X, T, y, NULL);
    free(X);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Latent states (Sec. 5 "KV Cache Compression", Fig. 5, Table 4)          */
/* ------------------------------------------------------------------------ */

/* The rank-r latent of each path, the bracketed inner product of Prop. 1
 * after the latent scale: z_p[t][j] = l_p[j] * sum_i V_p,sign[i][j] g_p[i] X[t][i].
 * Stored as [T][r_0 + r_1]: path 0 in columns 0..r_0-1, path 1 after it. */
int lbo_latent(const lbo_linear *L, const uint16_t *x, int64_t T, double *z)
{
    int64_t din = L->d_in, n1 = 0;
    for (int p = 0; p < L->n_paths; p++)
        n1 += L->path[p].r;
    double *X = decode_bf16_array(x, T * din);
    if (!X)
        return -1;
    int64_t off = 0;
    for (int p = 0; p < L->n_paths; p++) {
        const lbo_path *P = &L->path[p];
        int64_t r = P->r;
#pragma omp parallel for schedule(static)
        for (int64_t tj = 0; tj < T * r; tj++) {
            int64_t tt = tj / r, j = tj % r;
            double s = 0.0;
            for (int64_t i = 0; i < din; i++)
                s += X[tt * din + i] * lbo_half_to_double(P->g[i]) * sign_v(P->v_words, r, i, j);
            z[tt * n1 + off + j] = lbo_half_to_double(P->l[j]) * s;
        }
        off += r;
    }
    free(X);
    return 0;
}

/* The output rebuilt from cached latents, Prop. 1's outer part per path,
 * summed over paths (Eq. 6): y[t][o] = sum_p h_p[o] sum_j U_p,sign[o][j] z_p[t][j],
 * z in the layout lbo_latent writes. */
void lbo_expand(const lbo_linear *L, const double *z, int64_t T, double *y)
{
    int64_t dout = L->d_out, n1 = 0;
    for (int p = 0; p < L->n_paths; p++)
        n1 += L->path[p].r;
#pragma omp parallel for schedule(static)
    for (int64_t to = 0; to < T * dout; to++) {
        int64_t tt = to / dout, o = to % dout, off = 0;
        double acc = 0.0;
        for (int p = 0; p < L->n_paths; p++) {
            const lbo_path *P = &L->path[p];
            double s = 0.0;
            for (int64_t j = 0; j < P->r; j++)
                s += z[tt * n1 + off + j] * sign_u(P->u_words, P->r, o, j);
            acc += lbo_half_to_double(P->h[o]) * s;
            off += P->r;
        }
        y[to] = acc;
    }
}

/* ------------------------------------------------------------------------ */
/* Decode chain of the 70B-shaped stack                                     */
/* ------------------------------------------------------------------------ */

/* rho(v) = v / sqrt(mean(v^2)) (RMS normalisation with unit weight, eps 0). */
static void rms_normalize(const double *v, int64_t n, double *dst)
{
    double ss = 0.0;
    for (int64_t i = 0; i < n; i++)
        ss += v[i] * v[i];
    double inv = 1.0 / sqrt(ss / (double)n);
    for (int64_t i = 0; i < n; i++)
        dst[i] = v[i] * inv;
}

/* silu(x) = x * sigmoid(x) = x / (1 + e^-x). */
static double silu(double x) { return x / (1.0 + exp(-x)); }

int lbo_stack_forward(const lbo_linear *lin, int32_t n_layers, int32_t head_dim,
                      const uint16_t *x0, double *out, double *q_out, double *kv_out)
{
    int64_t d = lin[0].d_in;      /* d_model */
    int64_t dkv = lin[1].d_out;   /* n_kv_heads * head_dim */
    int64_t dff = lin[4].d_out;   /* MLP width */
    int64_t group = d / dkv;      /* query heads per kv head */
    double *a = decode_bf16_array(x0, d);
    double *n = (double *)malloc((size_t)d * sizeof(double));
    double *q = (double *)malloc((size_t)d * sizeof(double));
    double *k = (double *)malloc((size_t)dkv * sizeof(double));
    double *v = (double *)malloc((size_t)dkv * sizeof(double));
    double *attn = (double *)malloc((size_t)d * sizeof(double));
    double *o = (double *)malloc((size_t)d * sizeof(double));
    double *gt = (double *)malloc((size_t)dff * sizeof(double));
    double *up = (double *)malloc((size_t)dff * sizeof(double));
    double *dn = (double *)malloc((size_t)d * sizeof(double));
    int rc = -1;
    if (!a || !n || !q || !k || !v || !attn || !o || !gt || !up || !dn)
        goto done;
    for (int32_t layer = 0; layer < n_layers; layer++) {
        const lbo_linear *Lq = &lin[7 * layer + 0], *Lk = &lin[7 * layer + 1],
                         *Lv = &lin[7 * layer + 2], *Lo = &lin[7 * layer + 3],
                         *Lg = &lin[7 * layer + 4], *Lu = &lin[7 * layer + 5],
                         *Ld = &lin[7 * layer + 6];
        /* attention block: n = rho(a); q, k, v projections */
        rms_normalize(a, d, n);
        if (lbo_apply_factored(Lq, n, 1, q, NULL) || lbo_apply_factored(Lk, n, 1, k, NULL) ||
            lbo_apply_factored(Lv, n, 1, v, NULL))
            goto done;
        if (q_out)
            memcpy(q_out + (int64_t)layer * d, q, (size_t)d * sizeof(double));
        if (kv_out) {
            memcpy(kv_out + (2 * (int64_t)layer + 0) * dkv, k, (size_t)dkv * sizeof(double));
            memcpy(kv_out + (2 * (int64_t)layer + 1) * dkv, v, (size_t)dkv * sizeof(double));
        }
        /* attention over a one-position context: the softmax of a single
         * score is 1, so query head hq reads the value of its kv head
         * hq / group unchanged */
        for (int64_t j = 0; j < d; j++) {
            int64_t hq = j / head_dim, c = j % head_dim;
            attn[j] = v[(hq / group) * head_dim + c];
        }
        if (lbo_apply_factored(Lo, attn, 1, o, NULL))
            goto done;
        for (int64_t i = 0; i < d; i++)
            a[i] += o[i];                       /* h = a + o */
        /* MLP block: n = rho(h); m = silu(gate(n)) * up(n); a = h + down(m) */
        rms_normalize(a, d, n);
        if (lbo_apply_factored(Lg, n, 1, gt, NULL) || lbo_apply_factored(Lu, n, 1, up, NULL))
            goto done;
        for (int64_t i = 0; i < dff; i++)
            gt[i] = silu(gt[i]) * up[i];
        if (lbo_apply_factored(Ld, gt, 1, dn, NULL))
            goto done;
        for (int64_t i = 0; i < d; i++)
            a[i] += dn[i];
    }
    memcpy(out, a, (size_t)d * sizeof(double));
    rc = 0;
done:
    free(a);
    free(n);
    free(q);
    free(k);
    free(v);
    free(attn);
    free(o);
    free(gt);
    free(up);
    free(dn);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Accounting (App. E, App. I.1)                                            */
/* ------------------------------------------------------------------------ */

double lbo_bpw(int64_t d_out, int64_t d_in, int64_t r, int32_t n_paths)
{
    double per_path = (double)r * (double)(d_out + d_in)      /* U_sign + V_sign, 1 bit */
                      + 16.0 * (double)(d_out + d_in + r);    /* h, g, l in FP16 */
    return (double)n_paths * per_path / ((double)d_out * (double)d_in);
}

double lbo_rank_for_bpw(double b, int64_t d_out, int64_t d_in, int32_t n_paths)
{
    double s = (double)(d_out + d_in);
    return (b * (double)d_out * (double)d_in - n_paths * 16.0 * s) /
           (n_paths * s + n_paths * 16.0);
}

double lbo_flops(int64_t T, int64_t d_out, int64_t d_in, int64_t r, int32_t n_paths)
{
    return (double)n_paths * 2.0 * (double)T * (double)r * (double)(d_in + d_out);
}

void lbo_set_threads(int32_t n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int32_t lbo_get_threads(void)
{
#ifdef _OPENMP
    return (int32_t)omp_get_max_threads();
#else
    return 1;
#endif
}
