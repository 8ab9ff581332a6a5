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
/* Decode step at position p of a Llama-shaped decoder (App. I.3: only the  */
/* linears are LittleBit; attention and the norms stay dense)              */
/* ------------------------------------------------------------------------ */

/* The bf16 value nearest to v, ties to the even significand: bf16 keeps 8
 * significant bits, so v = m 2^e with 0.5 <= |m| < 1 is rounded to a
 * multiple of 2^(e - 8) (the exponent floor -125 covers the subnormals).
 * This is the rounding applied to the input of each LittleBit linear when the
 * GPU feeds it bf16. */
double lbo_round_bf16(double v)
{
    if (v == 0.0 || !isfinite(v))
        return v;
    int e;
    frexp(v, &e);
    if (e < -125)
        e = -125;
    double q = ldexp(1.0, e - 8);
    double t = v / q, f = floor(t), rem = t - f;
    double n = f;
    if (rem > 0.5 || (rem == 0.5 && fmod(f, 2.0) != 0.0))
        n = f + 1.0;
    return n * q;
}

/* Rotary position embedding of one head of width D at position p (the
 * half-split pairing): for i < D/2, (x_i, x_{i + D/2}) is rotated by
 * theta_i = p * base^(-2i / D). */
void lbo_rope(double *x, int64_t D, int64_t p, double base)
{
    int64_t h = D / 2;
    for (int64_t i = 0; i < h; i++) {
        double th = (double)p * pow(base, -2.0 * (double)i / (double)D);
        double c = cos(th), sn = sin(th), a = x[i], b = x[i + h];
        x[i] = a * c - b * sn;
        x[i + h] = a * sn + b * c;
    }
}

/* One decode step: the token x (bf16 [d]) at position pos, with the keys and
 * values of positions 0 .. pos-1 in the caches ([n_layers][max_pos][d_kv],
 * d_kv = n_kv_heads * head_dim; this step writes row pos of every layer).
 * Per layer, with rho the unit-weight RMS normalisation:
 *   n = rho(a); q, k, v = Q(n), K(n), V(n); q, k rotated (lbo_rope) per head
 *   cache[pos] = (k, v); per query head h of kv head g = h / (n_heads / n_kv_heads)
 *   s_t = q_h . k_t,g / sqrt(head_dim), w = softmax_t(s) over t = 0..pos,
 *   attn_h = sum_t w_t v_t,g;  a += O(attn)
 *   n = rho(a); a += Down(silu(Gate(n)) . Up(n))
 * round_inputs = 1 rounds n, attn and the MLP product to bf16 before their
 * linears (lbo_round_bf16): the chain with bf16 linear inputs; 0 keeps every
 * activation exact (the GPU decode step keeps them in fp32).
 * Optional outputs per layer: attn_out [n_layers][d], qk_out [n_layers][d + d_kv]
 * (the rotated q and k).  0, or -1 (pos out of range or no memory). */
int lbo_decoder_step(const lbo_linear *lin, int32_t n_layers, int32_t n_heads,
                     int32_t n_kv_heads, int32_t head_dim, double rope_base, int64_t pos,
                     int64_t max_pos, int32_t round_inputs, const uint16_t *x, double *kcache,
                     double *vcache, double *out, double *attn_out, double *qk_out)
{
    int64_t d = (int64_t)n_heads * head_dim, dkv = (int64_t)n_kv_heads * head_dim;
    int64_t dff = lin[4].d_out, group = n_heads / n_kv_heads;
    if (pos < 0 || pos >= max_pos || n_kv_heads <= 0 || n_heads % n_kv_heads != 0)
        return -1;
    double *a = decode_bf16_array(x, d);
    double *n = (double *)malloc((size_t)d * sizeof(double));
    double *q = (double *)malloc((size_t)d * sizeof(double));
    double *k = (double *)malloc((size_t)dkv * sizeof(double));
    double *v = (double *)malloc((size_t)dkv * sizeof(double));
    double *attn = (double *)malloc((size_t)d * sizeof(double));
    double *o = (double *)malloc((size_t)d * sizeof(double));
    double *gt = (double *)malloc((size_t)dff * sizeof(double));
    double *up = (double *)malloc((size_t)dff * sizeof(double));
    double *w = (double *)malloc((size_t)(pos + 1) * sizeof(double));
    int rc = -1;
    if (!a || !n || !q || !k || !v || !attn || !o || !gt || !up || !w)
        goto done;
    for (int32_t layer = 0; layer < n_layers; layer++) {
        const lbo_linear *L = &lin[7 * (int64_t)layer];
        double *Kc = kcache + (int64_t)layer * max_pos * dkv;
        double *Vc = vcache + (int64_t)layer * max_pos * dkv;
        rms_normalize(a, d, n);
        if (round_inputs)
            for (int64_t i = 0; i < d; i++)
                n[i] = lbo_round_bf16(n[i]);
        if (lbo_apply_factored(&L[0], n, 1, q, NULL) || lbo_apply_factored(&L[1], n, 1, k, NULL) ||
            lbo_apply_factored(&L[2], n, 1, v, NULL))
            goto done;
        for (int32_t h = 0; h < n_heads; h++)
            lbo_rope(q + (int64_t)h * head_dim, head_dim, pos, rope_base);
        for (int32_t g = 0; g < n_kv_heads; g++)
            lbo_rope(k + (int64_t)g * head_dim, head_dim, pos, rope_base);
        if (qk_out) {
            memcpy(qk_out + (int64_t)layer * (d + dkv), q, (size_t)d * sizeof(double));
            memcpy(qk_out + (int64_t)layer * (d + dkv) + d, k, (size_t)dkv * sizeof(double));
        }
        memcpy(Kc + pos * dkv, k, (size_t)dkv * sizeof(double));
        memcpy(Vc + pos * dkv, v, (size_t)dkv * sizeof(double));
        for (int32_t h = 0; h < n_heads; h++) {
            int64_t g = h / group;
            const double *qh = q + (int64_t)h * head_dim;
            double mx = -INFINITY, sum = 0.0;
            for (int64_t t = 0; t <= pos; t++) {
                double s = 0.0;
                for (int64_t c = 0; c < head_dim; c++)
                    s += qh[c] * Kc[t * dkv + g * head_dim + c];
                w[t] = s / sqrt((double)head_dim);
                if (w[t] > mx)
                    mx = w[t];
            }
            for (int64_t t = 0; t <= pos; t++) {
                w[t] = exp(w[t] - mx);
                sum += w[t];
            }
            for (int64_t c = 0; c < head_dim; c++) {
                double acc = 0.0;
                for (int64_t t = 0; t <= pos; t++)
                    acc += w[t] * Vc[t * dkv + g * head_dim + c];
                attn[(int64_t)h * head_dim + c] = acc / sum;
            }
        }
        if (attn_out)
            memcpy(attn_out + (int64_t)layer * d, attn, (size_t)d * sizeof(double));
        if (round_inputs)
            for (int64_t i = 0; i < d; i++)
                attn[i] = lbo_round_bf16(attn[i]);
        if (lbo_apply_factored(&L[3], attn, 1, o, NULL))
            goto done;
        for (int64_t i = 0; i < d; i++)
            a[i] += o[i];
        rms_normalize(a, d, n);
        if (round_inputs)
            for (int64_t i = 0; i < d; i++)
                n[i] = lbo_round_bf16(n[i]);
        if (lbo_apply_factored(&L[4], n, 1, gt, NULL) || lbo_apply_factored(&L[5], n, 1, up, NULL))
            goto done;
        for (int64_t i = 0; i < dff; i++) {
            gt[i] = up[i] * silu(gt[i]);
            if (round_inputs)
                gt[i] = lbo_round_bf16(gt[i]);
        }
        if (lbo_apply_factored(&L[6], gt, 1, o, NULL))
            goto done;
        for (int64_t i = 0; i < d; i++)
            a[i] += o[i];
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
    free(w);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Dual-SVID initialisation (Sec. 3.2) and Residual Compensation (Sec. 3.3)  */
/* ------------------------------------------------------------------------ */

/* Truncated SVD by one-sided Jacobi (Hestenes).  Plane rotations G act on
 * pairs of columns of A until all columns are mutually orthogonal:
 * A G_1 G_2 ... = B with B's columns b_j = sigma_j u_j, and V = G_1 G_2 ...,
 * so A = sum_j sigma_j u_j v_j^T.  Kept transposed: row j of Bt is column j
 * of A G..., row j of J is column j of V (J starts as I).  For columns x, y
 * with alpha = x.x, beta = y.y, gamma = x.y the rotation x' = c x - s y,
 * y' = s x + c y makes x'.y' = 0 for t = s/c, the smaller root of
 * t^2 + 2 zeta t - 1 = 0, zeta = (beta - alpha) / (2 gamma).
 * Returns the r largest singular values in decreasing order (s[r]) with
 * U[m][r], V[n][r].  Sign convention (u_j, v_j are defined up to a joint
 * sign): the entry of largest magnitude of each v_j, the first one on a tie,
 * is positive.  0, or -1 (r out of range or no memory). */
int lbo_svd_top(const double *A, int64_t m, int64_t n, int64_t r, double *s, double *U, double *V)
{
    if (r < 1 || r > m || r > n)
        return -1;
    double *Bt = (double *)malloc((size_t)(n * m) * sizeof(double));
    double *J = (double *)calloc((size_t)(n * n), sizeof(double));
    double *nrm = (double *)malloc((size_t)n * sizeof(double));
    char *used = (char *)calloc((size_t)n, 1);
    if (!Bt || !J || !nrm || !used) {
        free(Bt);
        free(J);
        free(nrm);
        free(used);
        return -1;
    }
    for (int64_t i = 0; i < m; i++)
        for (int64_t j = 0; j < n; j++)
            Bt[j * m + i] = A[i * n + j];
    for (int64_t j = 0; j < n; j++)
        J[j * n + j] = 1.0;
    for (int sweep = 0; sweep < 60; sweep++) {
        double off = 0.0;
        for (int64_t p = 0; p < n - 1; p++)
            for (int64_t q = p + 1; q < n; q++) {
                double *x = Bt + p * m, *y = Bt + q * m;
                double alpha = 0.0, beta = 0.0, gamma = 0.0;
                for (int64_t i = 0; i < m; i++) {
                    alpha += x[i] * x[i];
                    beta += y[i] * y[i];
                    gamma += x[i] * y[i];
                }
                if (gamma == 0.0)
                    continue;
                double rel = fabs(gamma) / sqrt(alpha * beta);
                if (rel > off)
                    off = rel;
                if (rel < 1e-15)
                    continue;
                double zeta = (beta - alpha) / (2.0 * gamma);
                double t = (zeta >= 0 ? 1.0 : -1.0) / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
                double c = 1.0 / sqrt(1.0 + t * t), sn = c * t;
                for (int64_t i = 0; i < m; i++) {
                    double a = x[i], b = y[i];
                    x[i] = c * a - sn * b;
                    y[i] = sn * a + c * b;
                }
                double *jp = J + p * n, *jq = J + q * n;
                for (int64_t i = 0; i < n; i++) {
                    double a = jp[i], b = jq[i];
                    jp[i] = c * a - sn * b;
                    jq[i] = sn * a + c * b;
                }
            }
        if (off < 1e-14)
            break;
    }
    for (int64_t j = 0; j < n; j++) {
        double ss = 0.0;
        for (int64_t i = 0; i < m; i++)
            ss += Bt[j * m + i] * Bt[j * m + i];
        nrm[j] = sqrt(ss);
    }
    for (int64_t a = 0; a < r; a++) {
        /* the largest remaining column norm (lowest index on a tie) */
        int64_t best = -1;
        for (int64_t b = 0; b < n; b++)
            if (!used[b] && (best < 0 || nrm[b] > nrm[best]))
                best = b;
        used[best] = 1;
        s[a] = nrm[best];
        int64_t imax = 0;
        for (int64_t i = 1; i < n; i++)
            if (fabs(J[best * n + i]) > fabs(J[best * n + imax]))
                imax = i;
        double sg = J[best * n + imax] < 0 ? -1.0 : 1.0;
        for (int64_t i = 0; i < n; i++)
            V[i * r + a] = sg * J[best * n + i];
        for (int64_t i = 0; i < m; i++)
            U[i * r + a] = nrm[best] > 0 ? sg * Bt[best * m + i] / nrm[best] : 0.0;
    }
    free(used);
    free(Bt);
    free(J);
    free(nrm);
    return 0;
}

/* Best rank-1 approximation of a nonnegative matrix M (rows x cols, all
 * entries >= 0) as a b^T with a, b >= 0: its leading singular pair, found
 * by power iteration from b = 1 (for a nonnegative matrix the leading
 * singular vectors can be taken nonnegative, Perron-Frobenius).  The
 * singular value sigma is split evenly: a = sqrt(sigma) u, b = sqrt(sigma) v.
 * A zero matrix gives a = b = 0. */
static void rank1_nonneg(const double *M, int64_t rows, int64_t cols, double *a, double *b)
{
    double *u = (double *)malloc((size_t)rows * sizeof(double));
    double *v = (double *)malloc((size_t)cols * sizeof(double));
    if (!u || !v) {
        free(u);
        free(v);
        return;
    }
    for (int64_t j = 0; j < cols; j++)
        v[j] = 1.0 / sqrt((double)cols);
    double sigma = 0.0;
    for (int it = 0; it < 500; it++) {
        double nu = 0.0, nv = 0.0;
        for (int64_t i = 0; i < rows; i++) {
            double acc = 0.0;
            for (int64_t j = 0; j < cols; j++)
                acc += M[i * cols + j] * v[j];
            u[i] = acc;
            nu += acc * acc;
        }
        nu = sqrt(nu);
        if (nu == 0.0) {
            sigma = 0.0;
            break;
        }
        for (int64_t i = 0; i < rows; i++)
            u[i] /= nu;
        double change = 0.0;
        for (int64_t j = 0; j < cols; j++) {
            double acc = 0.0;
            for (int64_t i = 0; i < rows; i++)
                acc += M[i * cols + j] * u[i];
            change += (acc - nu * v[j]) * (acc - nu * v[j]);
            v[j] = acc;
            nv += acc * acc;
        }
        nv = sqrt(nv);
        for (int64_t j = 0; j < cols; j++)
            v[j] /= nv;
        sigma = nv;
        if (sqrt(change) <= 1e-15 * nv)
            break;
    }
    double sq = sqrt(sigma);
    for (int64_t i = 0; i < rows; i++)
        a[i] = sigma > 0 ? sq * u[i] : 0.0;
    for (int64_t j = 0; j < cols; j++)
        b[j] = sigma > 0 ? sq * v[j] : 0.0;
    free(u);
    free(v);
}

/* Dual-SVID of one path (Sec. 3.2): from R (d_out x d_in, row-major) and
 * rank r,
 *   (1) truncated SVD R ~ U' V'^T with U' = U_r diag(sqrt s), V' = V_r diag(sqrt s)
 *       (the singular values split evenly between the two factors);
 *   (2) U_sign = sign(U'), V_sign = sign(V') (sign(0) = +1);
 *   (3) |U'| ~ h0 l_u^T, |V'| ~ g0 l_v^T (best rank-1, rank1_nonneg), l0 = l_u . l_v.
 * Outputs usign[d_out][r], vsign[d_in][r] (+-1), h[d_out], g[d_in], l[r].
 * 0, or -1. */
int lbo_dual_svid_path(const double *R, int64_t d_out, int64_t d_in, int64_t r, int8_t *usign,
                       int8_t *vsign, double *h, double *g, double *l)
{
    double *s = (double *)malloc((size_t)r * sizeof(double));
    double *U = (double *)malloc((size_t)(d_out * r) * sizeof(double));
    double *V = (double *)malloc((size_t)(d_in * r) * sizeof(double));
    double *lu = (double *)malloc((size_t)r * sizeof(double));
    double *lv = (double *)malloc((size_t)r * sizeof(double));
    int rc = -1;
    if (!s || !U || !V || !lu || !lv || lbo_svd_top(R, d_out, d_in, r, s, U, V) != 0)
        goto out;
    for (int64_t j = 0; j < r; j++) {
        double q = sqrt(s[j]);
        for (int64_t i = 0; i < d_out; i++)
            U[i * r + j] *= q;
        for (int64_t i = 0; i < d_in; i++)
            V[i * r + j] *= q;
    }
    for (int64_t k = 0; k < d_out * r; k++) {
        usign[k] = U[k] < 0 ? -1 : 1;
        U[k] = fabs(U[k]);
    }
    for (int64_t k = 0; k < d_in * r; k++) {
        vsign[k] = V[k] < 0 ? -1 : 1;
        V[k] = fabs(V[k]);
    }
    rank1_nonneg(U, d_out, r, h, lu);
    rank1_nonneg(V, d_in, r, g, lv);
    for (int64_t j = 0; j < r; j++)
        l[j] = lu[j] * lv[j];
    rc = 0;
out:
    free(s);
    free(U);
    free(V);
    free(lu);
    free(lv);
    return rc;
}

/* W_hat of one path from signs and scales, Eq. 4: h_o u_oj l_j v_ij g_i. */
void lbo_path_weight(const int8_t *usign, const int8_t *vsign, const double *h, const double *g,
                     const double *l, int64_t d_out, int64_t d_in, int64_t r, double *What)
{
#pragma omp parallel for schedule(static)
    for (int64_t o = 0; o < d_out; o++)
        for (int64_t i = 0; i < d_in; i++) {
            double acc = 0.0;
            for (int64_t j = 0; j < r; j++)
                acc += usign[o * r + j] * l[j] * vsign[i * r + j];
            What[o * d_in + i] = h[o] * acc * g[i];
        }
}

/* ------------------------------------------------------------------------ */
/* QAT forward / backward with SmoothSign (Sec. 4 settings, App. "SmoothSign") */
/* ------------------------------------------------------------------------ */

/* Sign of a latent entry as the forward uses it: +1 for x >= 0, else -1;
 * with relaxed != 0 the latent value itself (the continuous relaxation used
 * to check the gradients with respect to the sign matrices). */
static double qat_sign(double x, int relaxed) { return relaxed ? x : (x < 0 ? -1.0 : 1.0); }

/* Y = sum_p ((((X . g) S(V)) . l) S(U)^T) . h with S the sign (Prop. 1 on the
 * latent factors).  X [T][d_in], Y [T][d_out]. */
int lbo_train_forward(const lbo_train_linear *L, const double *X, int64_t T, double *Y, int relaxed)
{
    int64_t din = L->d_in, dout = L->d_out;
    for (int64_t k = 0; k < T * dout; k++)
        Y[k] = 0.0;
    for (int p = 0; p < L->n_paths; p++) {
        const lbo_train_path *P = &L->path[p];
        int64_t r = P->r;
        double *z = (double *)malloc((size_t)(T * r > 0 ? T * r : 1) * sizeof(double));
        if (!z)
            return -1;
#pragma omp parallel for schedule(static)
        for (int64_t tj = 0; tj < T * r; tj++) {
            int64_t t = tj / r, j = tj % r;
            double s = 0.0;
            for (int64_t i = 0; i < din; i++)
                s += X[t * din + i] * P->g[i] * qat_sign(P->v[i * r + j], relaxed);
            z[tj] = s * P->l[j];
        }
#pragma omp parallel for schedule(static)
        for (int64_t to = 0; to < T * dout; to++) {
            int64_t t = to / dout, o = to % dout;
            double s = 0.0;
            for (int64_t j = 0; j < r; j++)
                s += z[t * r + j] * qat_sign(P->u[o * r + j], relaxed);
            Y[to] += s * P->h[o];
        }
        free(z);
    }
    return 0;
}

/* Gradients of the loss sum(Y . dY) through the forward above, by the chain
 * rule along Prop. 1's steps, per path (a = X . g, t = a S(V), z = t . l,
 * q = z S(U)^T, y = q . h):
 *   dh_o = sum_t dY_to q_to          dq = dY . h
 *   dS(U) = dq^T z                   dz = dq S(U)
 *   dl_j = sum_t dz_tj t_tj          dt = dz . l
 *   dS(V) = a^T dt                   da = dt S(V)^T
 *   dg_i = sum_t da_ti X_ti          dX += da . g
 * and through the sign by SmoothSign, d sign(x)/dx := k (1 - tanh(k x)^2)
 * (the derivative of tanh(k x)): dU = dS(U) . k (1 - tanh^2(k U)), likewise
 * dV.  With relaxed != 0 the sign is the identity and dU = dS(U).
 * Outputs per path (arrays of the path's shapes, overwritten) and dX [T][d_in]
 * (may be NULL). */
int lbo_train_backward(const lbo_train_linear *L, const double *X, const double *dY, int64_t T,
                       double k, int relaxed, lbo_train_grad *G, double *dX)
{
    int64_t din = L->d_in, dout = L->d_out;
    if (dX)
        for (int64_t q = 0; q < T * din; q++)
            dX[q] = 0.0;
    for (int p = 0; p < L->n_paths; p++) {
        const lbo_train_path *P = &L->path[p];
        lbo_train_grad *D = &G[p];
        int64_t r = P->r;
        double *t = (double *)malloc((size_t)(T * r + 1) * sizeof(double));
        double *z = (double *)malloc((size_t)(T * r + 1) * sizeof(double));
        double *dz = (double *)malloc((size_t)(T * r + 1) * sizeof(double));
        double *q = (double *)malloc((size_t)(T * dout + 1) * sizeof(double));
        double *da = (double *)malloc((size_t)(T * din + 1) * sizeof(double));
        if (!t || !z || !dz || !q || !da) {
            free(t);
            free(z);
            free(dz);
            free(q);
            free(da);
            return -1;
        }
        /* forward intermediates */
#pragma omp parallel for schedule(static)
        for (int64_t tj = 0; tj < T * r; tj++) {
            int64_t tt = tj / r, j = tj % r;
            double s = 0.0;
            for (int64_t i = 0; i < din; i++)
                s += X[tt * din + i] * P->g[i] * qat_sign(P->v[i * r + j], relaxed);
            t[tj] = s;
            z[tj] = s * P->l[j];
        }
#pragma omp parallel for schedule(static)
        for (int64_t to = 0; to < T * dout; to++) {
            int64_t tt = to / dout, o = to % dout;
            double s = 0.0;
            for (int64_t j = 0; j < r; j++)
                s += z[tt * r + j] * qat_sign(P->u[o * r + j], relaxed);
            q[to] = s;
        }
        /* dh, dS(U) -> dU */
        for (int64_t o = 0; o < dout; o++) {
            double s = 0.0;
            for (int64_t tt = 0; tt < T; tt++)
                s += dY[tt * dout + o] * q[tt * dout + o];
            D->dh[o] = s;
        }
#pragma omp parallel for schedule(static)
        for (int64_t oj = 0; oj < dout * r; oj++) {
            int64_t o = oj / r, j = oj % r;
            double s = 0.0;
            for (int64_t tt = 0; tt < T; tt++)
                s += dY[tt * dout + o] * P->h[o] * z[tt * r + j];
            double th = tanh(k * P->u[oj]);
            D->du[oj] = relaxed ? s : s * k * (1.0 - th * th);
        }
        /* dz, dl, dt */
#pragma omp parallel for schedule(static)
        for (int64_t tj = 0; tj < T * r; tj++) {
            int64_t tt = tj / r, j = tj % r;
            double s = 0.0;
            for (int64_t o = 0; o < dout; o++)
                s += dY[tt * dout + o] * P->h[o] * qat_sign(P->u[o * r + j], relaxed);
            dz[tj] = s;
        }
        for (int64_t j = 0; j < r; j++) {
            double s = 0.0;
            for (int64_t tt = 0; tt < T; tt++)
                s += dz[tt * r + j] * t[tt * r + j];
            D->dl[j] = s;
        }
        for (int64_t tj = 0; tj < T * r; tj++)
            dz[tj] *= P->l[tj % r]; /* dz now holds dt */
        /* dS(V) -> dV, da, dg, dX */
#pragma omp parallel for schedule(static)
        for (int64_t ij = 0; ij < din * r; ij++) {
            int64_t i = ij / r, j = ij % r;
            double s = 0.0;
            for (int64_t tt = 0; tt < T; tt++)
                s += X[tt * din + i] * P->g[i] * dz[tt * r + j];
            double th = tanh(k * P->v[ij]);
            D->dv[ij] = relaxed ? s : s * k * (1.0 - th * th);
        }
#pragma omp parallel for schedule(static)
        for (int64_t ti = 0; ti < T * din; ti++) {
            int64_t tt = ti / din, i = ti % din;
            double s = 0.0;
            for (int64_t j = 0; j < r; j++)
                s += dz[tt * r + j] * qat_sign(P->v[i * r + j], relaxed);
            da[ti] = s;
        }
        for (int64_t i = 0; i < din; i++) {
            double s = 0.0;
            for (int64_t tt = 0; tt < T; tt++)
                s += da[tt * din + i] * X[tt * din + i];
            D->dg[i] = s;
        }
        if (dX)
            for (int64_t ti = 0; ti < T * din; ti++)
                dX[ti] += da[ti] * P->g[ti % din];
        free(t);
        free(z);
        free(dz);
        free(q);
        free(da);
    }
    return 0;
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
