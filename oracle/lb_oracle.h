/*
 * lb_oracle.h -- CPU oracle for the LittleBit linear forward.
 *
 * TEST INFRASTRUCTURE ONLY.  This oracle exists to check the CUDA path; it is
 * never on the product path.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load it.  It shares no code,
 * header, table or helper with the CUDA library: it defines its own parameter
 * struct, its own fp16/bf16 decoders and its own bit packer.
 *
 * Everything is computed in IEEE fp64 ("double") from the definitions in the
 * paper (LittleBit, arXiv 2506.13771):
 *   Eq. 2   U_sign = sign(U), V_sign = sign(V) in {-1,+1}
 *   Eq. 3   h in R^{d_out}, g in R^{d_in}, l in R^{r}, stored as FP16
 *   Eq. 4   W_pri = diag(h) U_sign diag(l) V_sign^T diag(g)
 *   Eq. 5   W_res has the same structure with its own parameters
 *   Eq. 6   W = W_pri + W_res
 *   Prop. 1 Y = ((((X . g) V_sign) . l) U_sign^T) . h   (per path)
 *   App. E  bits-per-weight accounting and the rank solve
 *
 * Readings where the paper is silent (documented with the data layout):
 *   - sign(0) = +1; a packed bit set to 1 means -1, 0 means +1.
 *   - bits are packed LSB-first, 32 per uint32 along the reduction dim:
 *       U words: [d_out][ceil(r/32)],    bit k of word (o,w) = element (o, 32w+k)
 *       V words: [ceil(d_in/32)][r],     bit k of word (w,j) = element (32w+k, j)
 *     padding bits beyond the matrix are written 0 and never read.
 *
 * Parity status of every function is pinned by tests (see tests/test_oracle_*.py).
 */
#ifndef LB_ORACLE_H
#define LB_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* One LittleBit path (Eq. 4 / Eq. 5).  All pointers are host memory. */
typedef struct {
    int32_t r;                 /* latent rank */
    const uint32_t *v_words;   /* V_sign bits, [ceil(d_in/32)][r] */
    const uint32_t *u_words;   /* U_sign bits, [d_out][ceil(r/32)] */
    const uint16_t *g;         /* fp16 bit patterns, [d_in]  (column scale) */
    const uint16_t *l;         /* fp16 bit patterns, [r]     (latent scale) */
    const uint16_t *h;         /* fp16 bit patterns, [d_out] (row scale) */
} lbo_path;

/* One LittleBit linear: n_paths = 1 (primary only) or 2 (primary + residual). */
typedef struct {
    int32_t d_in, d_out, n_paths;
    lbo_path path[2];
} lbo_linear;

/* Number decoding from the format definitions. */
double lbo_half_to_double(uint16_t bits);   /* IEEE 754 binary16 */
double lbo_bf16_to_double(uint16_t bits);   /* bfloat16 = top half of binary32 */

/* Packing of a row-major [rows][cols] matrix of +-1 (int8).  Returns 0, or -1
 * if an element is neither +1 nor -1 (out is then undefined).
 * lbo_pack_u packs along cols  (U layout), out has rows*ceil(cols/32) words.
 * lbo_pack_v packs along rows  (V layout), out has ceil(rows/32)*cols words. */
int lbo_pack_u(const int8_t *signs, int64_t rows, int64_t cols, uint32_t *out);
int lbo_pack_v(const int8_t *signs, int64_t rows, int64_t cols, uint32_t *out);
/* Inverse of the above; padding bits are ignored. */
void lbo_unpack_u(const uint32_t *words, int64_t rows, int64_t cols, int8_t *signs);
void lbo_unpack_v(const uint32_t *words, int64_t rows, int64_t cols, int8_t *signs);

/* Dense mode: rebuild W (Eq. 4-6) in fp64, then Y = X W^T.
 * x: bf16 bit patterns [T][d_in]; y: [T][d_out].  Returns 0 or -1 (no memory). */
int lbo_forward_dense(const lbo_linear *L, const uint16_t *x, int64_t T, double *y);

/* Factored mode (Prop. 1), summed over paths (Eq. 6).  x: bf16 [T][d_in]. */
int lbo_forward_factored(const lbo_linear *L, const uint16_t *x, int64_t T, double *y);

/* Factored mode on an fp64 input [T][d_in]; optionally returns the stage-1
 * latent vectors t_p = (X . g_p) V_p,sign, as [n_paths][T][r_p] (may be NULL). */
int lbo_apply_factored(const lbo_linear *L, const double *x, int64_t T, double *y,
                       double *t_out);

/* Latent states (Sec. 5, KV cache compression; Prop. 1's inner product after
 * the latent scale): z[t][off_p + j] = l_p[j] * ((X[t] . g_p) V_p,sign)[j],
 * off_0 = 0, off_1 = r_0; z is [T][r_0 + r_1].  x: bf16 [T][d_in].  0 / -1. */
int lbo_latent(const lbo_linear *L, const uint16_t *x, int64_t T, double *z);
/* The output from latents: y[t][o] = sum_p h_p[o] (U_p,sign z_p[t])[o], z in
 * lbo_latent's layout, y: [T][d_out]. */
void lbo_expand(const lbo_linear *L, const double *z, int64_t T, double *y);

/* One decode step of a Llama-shaped decoder stack at sequence position 0,
 * n_layers x (q, k, v, o, gate, up, down), seven linears per layer in that
 * order, only the linears being LittleBit (the paper's end-to-end setting
 * keeps attention and norms in FP16, App. I.3).  With rho(v) = v /
 * sqrt(mean(v^2)) and a = x0:
 *   n = rho(a); q = Q(n); k = K(n); v = V(n)
 *   attn = v broadcast over the query heads of each kv head (attention over a
 *          one-position context: the softmax of one score is 1)
 *   h = a + O(attn)
 *   n = rho(h); m = silu(Gate(n)) * Up(n); a = h + Down(m)
 * head_dim: width of one attention head (d_model and d_kv are multiples).
 * x0: bf16 [d_model]; out: the final a, [d_model]; q_out: [n_layers][d_model]
 * and kv_out: [n_layers][2][d_kv] (k then v), each may be NULL.  Returns 0/-1. */
int lbo_stack_forward(const lbo_linear *lin, int32_t n_layers, int32_t head_dim,
                      const uint16_t *x0, double *out, double *q_out, double *kv_out);

/* Dual-SVID initialisation (Sec. 3.2).
 * lbo_svd_top: the r largest singular triples of A (m x n, row-major) by
 * one-sided Jacobi; s[r] decreasing, U[m][r], V[n][r]; each v_j has its
 * largest-magnitude entry (first on a tie) positive.  0 / -1.
 * lbo_dual_svid_path: truncated SVD R ~ U' V'^T (U' = U diag(sqrt s), V' =
 * V diag(sqrt s)), U_sign = sign(U'), V_sign = sign(V') (sign(0) = +1), best
 * rank-1 |U'| ~ h l_u^T and |V'| ~ g l_v^T (singular value split evenly),
 * l = l_u . l_v.  usign[d_out][r], vsign[d_in][r] (+-1).  0 / -1.
 * lbo_path_weight: W_hat = diag(h) U_sign diag(l) V_sign^T diag(g) (Eq. 4). */
int lbo_svd_top(const double *A, int64_t m, int64_t n, int64_t r, double *s, double *U, double *V);
int lbo_dual_svid_path(const double *R, int64_t d_out, int64_t d_in, int64_t r, int8_t *usign,
                       int8_t *vsign, double *h, double *g, double *l);
void lbo_path_weight(const int8_t *usign, const int8_t *vsign, const double *h, const double *g,
                     const double *l, int64_t d_out, int64_t d_in, int64_t r, double *What);

/* QAT (training) form of a linear: latent fp64 factors U [d_out][r],
 * V [d_in][r] and scales, the forward using their signs (Eq. 2). */
typedef struct {
    int32_t r;
    const double *u, *v, *g, *l, *h;
} lbo_train_path;
typedef struct {
    int32_t d_in, d_out, n_paths;
    lbo_train_path path[2];
} lbo_train_linear;
/* Gradients of one path (shapes of u, v, g, l, h). */
typedef struct {
    double *du, *dv, *dg, *dl, *dh;
} lbo_train_grad;
/* Y = sum_p Prop. 1 with S(U), S(V); S = sign (x >= 0 -> +1), or the identity
 * when relaxed != 0.  X [T][d_in], Y [T][d_out].  0 / -1. */
int lbo_train_forward(const lbo_train_linear *L, const double *X, int64_t T, double *Y, int relaxed);
/* Gradients of sum(Y . dY): chain rule along Prop. 1, SmoothSign
 * k (1 - tanh^2(k x)) through the sign (identity when relaxed).  dX may be
 * NULL.  0 / -1. */
int lbo_train_backward(const lbo_train_linear *L, const double *X, const double *dY, int64_t T,
                       double k, int relaxed, lbo_train_grad *G, double *dX);

/* App. E bits per weight: total parameter bits / (d_out * d_in), where each
 * path stores r*(d_out+d_in) sign bits and 16*(d_out+d_in+r) scale bits. */
double lbo_bpw(int64_t d_out, int64_t d_in, int64_t r, int32_t n_paths);
/* App. E rank solve (the real-valued r that gives exactly b). */
double lbo_rank_for_bpw(double b, int64_t d_out, int64_t d_in, int32_t n_paths);
/* App. I.1 operation count of one factored forward: 2*T*r*(d_in+d_out) per path. */
double lbo_flops(int64_t T, int64_t d_out, int64_t d_in, int64_t r, int32_t n_paths);

/* Threads used by the OpenMP loops (0 = the OpenMP default). */
/* Decode step at position pos of a Llama-shaped decoder (App. I.3): RMS
 * norms, rotary embedding, softmax attention over the KV cache, SiLU MLP,
 * residual stream; the linears are LittleBit (lin[7 * layer + 0..6] = q, k,
 * v, o, gate, up, down).  See lb_oracle.c for the exact definition. */
double lbo_round_bf16(double v);
void lbo_rope(double *x, int64_t D, int64_t p, double base);
int lbo_decoder_step(const lbo_linear *lin, int32_t n_layers, int32_t n_heads,
                     int32_t n_kv_heads, int32_t head_dim, double rope_base, int64_t pos,
                     int64_t max_pos, int32_t round_inputs, const uint16_t *x, double *kcache,
                     double *vcache, double *out, double *attn_out, double *qk_out);

void lbo_set_threads(int32_t n);
int32_t lbo_get_threads(void);

#ifdef __cplusplus
}
#endif
#endif
