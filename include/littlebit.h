/*
 * littlebit.h -- C ABI of the GB300 (sm_103a) LittleBit linear forward.
 *
 * LittleBit (arXiv 2506.13771) stores a d_out x d_in weight as one or two
 * factored, binarised paths (Sec. 3.1, Eq. 1-4; Residual Compensation,
 * Sec. 3.3, Eq. 5-6):
 *
 *     W_p  = diag(h_p) U_p,sign diag(l_p) V_p,sign^T diag(g_p)      (Eq. 4, 5)
 *     W    = W_pri + W_res                                          (Eq. 6)
 *
 * with U_sign in {-1,+1}^{d_out x r}, V_sign in {-1,+1}^{d_in x r} (Eq. 2) and
 * FP16 scales h in R^{d_out}, g in R^{d_in}, l in R^r (Eq. 3).  The forward
 * Y = X W^T is computed as Prop. 1 prescribes, per path,
 *
 *     Y += ((((X . g) V_sign) . l) U_sign^T) . h
 *
 * i.e. a +-1 reduction over d_in (stage 1, rank-r output t), a latent scale,
 * a +-1 reduction over r (stage 2) and a row scale.
 *
 * Conventions shared by every entry point
 *   - Sign bits: bit = 1 means -1, bit = 0 means +1 (sign(0) = +1).  Bits are
 *     packed LSB first, 32 per uint32, along the reduction dimension:
 *       U words  [d_out][ceil(r/32)]    bit k of word (o, w) = U_sign[o][32w+k]
 *       V words  [ceil(d_in/32)][r]     bit k of word (w, j) = V_sign[32w+k][j]
 *     Padding bits (beyond r, beyond d_in) are ignored on input.
 *   - Scales h, g, l are IEEE binary16 bit patterns; activations X are
 *     bfloat16 bit patterns, row-major [T][d_in]; Y is row-major [T][d_out].
 *   - All pointers passed to forward calls are DEVICE pointers on the current
 *     CUDA device and must be 16-byte aligned; the library checks alignment
 *     and nullness, not that the memory is on the device.
 *   - The caller owns every buffer.  The library allocates no device memory;
 *     scratch space is the caller's workspace ("ws"), sized by the
 *     *_workspace_size functions, 256-byte aligned, and zero-filled once
 *     before its first use (its first word is the sticky error word below;
 *     the calls themselves re-initialise everything else they use).
 *   - Everything is enqueued on the given stream (NULL = legacy default
 *     stream); no call synchronises except littlebit_poll_error.  Calls are
 *     safe from several host threads if they use distinct workspaces.
 *   - Arithmetic: products and sums in fp32 (the paper's kernel uses FP16,
 *     App. I.2; fp32 accumulation is this library's choice); outputs are
 *     bf16 (round to nearest even) or fp32.
 *   - Errors are returned as lb_status; launch failures map to LB_ERR_CUDA.
 *     Asynchronous device faults surface on a later CUDA call.  A grid-wide
 *     wait that exceeds its time limit (about one second) makes the kernel
 *     record LB_ERR_TIMEOUT in the workspace's sticky error word and return;
 *     while that word is set, kernels using the workspace return at once
 *     without writing outputs; littlebit_poll_error reads and clears it.
 *     A launch that timed out may leave exchange words behind: zero-fill the
 *     workspace again (or prepare a stack workspace again) before reusing it.
 */
#ifndef LITTLEBIT_H
#define LITTLEBIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream (cudaStream_t).  NULL selects the legacy default stream. */
typedef struct CUstream_st *lb_stream_t;

typedef enum {
    LB_OK = 0,
    LB_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad size or layout */
    LB_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels handle */
    LB_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed */
    LB_ERR_TIMEOUT = 4,      /* a device-side grid wait ran out (see poll) */
    LB_ERR_WORKSPACE = 5,    /* ws is NULL, misaligned or too small */
    LB_ERR_PLAN = 6,         /* stack workspace not prepared for these linears */
    LB_ERR_RANGE = 7         /* a stack intermediate left the exchange's range, or a
                                decode position lies outside the KV cache */
} lb_status;

typedef enum { LB_OUT_BF16 = 0, LB_OUT_FP32 = 1 } lb_out_dtype;

typedef enum {
    LB_PACK_U = 0,  /* pack a [rows][cols] matrix along cols -> [rows][ceil(cols/32)] */
    LB_PACK_V = 1   /* pack a [rows][cols] matrix along rows -> [ceil(rows/32)][cols] */
} lb_pack_layout;

/* One path of Eq. 4 / Eq. 5.  All pointers are device memory. */
typedef struct {
    int32_t r;                /* latent rank, 1 <= r <= 1024 */
    const uint32_t *v_bits;   /* V_sign, [ceil(d_in/32)][r] words */
    const uint32_t *u_bits;   /* U_sign, [d_out][ceil(r/32)] words */
    const uint16_t *g;        /* column scale, fp16 [d_in] */
    const uint16_t *l;        /* latent scale, fp16 [r] */
    const uint16_t *h;        /* row scale,    fp16 [d_out] */
} lb_path;

/* One LittleBit linear: n_paths = 2 (primary + residual, Eq. 6) or 1 (the
 * paper's variant without Residual Compensation, App. E note). */
typedef struct {
    int32_t d_in, d_out, n_paths;
    lb_path path[2];
} lb_linear;

/* Human-readable name of a status code (static string, never NULL). */
const char *littlebit_status_string(lb_status s);

/* Eq. 2 binarisation of already-signed factors: packs a row-major int8
 * [rows][cols] matrix of +1/-1 (DEVICE memory) into sign words (DEVICE) in
 * the given layout; out_words must be at least the layout's word count.
 * Padding bits are written 0.  An element other than +1/-1 makes the kernel
 * set *bad (a DEVICE int32, may be NULL) to 1; the words are then undefined.
 * *bad is not cleared by the call.  rows, cols >= 1. */
lb_status littlebit_pack(const int8_t *signs, int64_t rows, int64_t cols, int32_t layout,
                         uint32_t *out, int64_t out_words, int32_t *bad, lb_stream_t stream);

/* Workspace bytes littlebit_linear_forward needs for this layer and T tokens
 * (0 if the arguments are invalid). */
size_t littlebit_workspace_size(const lb_linear *L, int64_t T);

/* Y = X W^T for one LittleBit linear (Prop. 1 per path, paths summed by
 * Eq. 6).  L is a HOST struct holding device pointers.  x: bf16 [T][d_in];
 * y: [T][d_out] in y_dtype.  T = 0 is a no-op.  Requires d_in % 32 == 0 and
 * 1 <= r <= 1024 for every path (else LB_ERR_UNSUPPORTED).
 * Paths taken: T = 1 with every r % 8 == 0 and d_out % 8 == 0 -> one launch
 * of the single-token kernel (it keeps its exchange words in ws between
 * calls, so a workspace must not be shared by concurrent calls); T >= 16
 * and T * (r_0 + r_1) > 8192, with d_in and every r multiples of 64,
 * r <= 512 and d_out % 8 == 0 -> the tensor-core path (fp16 operands, see
 * its tolerance in the design notes); otherwise the two-launch CUDA-core
 * path.  On the tensor-core path with T >= 385, r_0 + r_1 a multiple of 512
 * and at least 96 stage-1 tiles of 128 x 512 (T >= 6144 at r_0 + r_1 =
 * 1024), the forward runs on SM pairs (tcgen05 cta_group::2) as three
 * launches in stream order; the environment variable LB_PREFILL_2SM=0, read
 * at each call, selects the one-launch form on single SMs instead.  Results
 * of the two forms agree to the path's tolerance, not bit for bit. */
lb_status littlebit_linear_forward(const lb_linear *L, const uint16_t *x, int64_t T, void *y,
                                   int32_t y_dtype, void *ws, size_t ws_bytes,
                                   lb_stream_t stream);

/* Element type of a latent-state buffer (littlebit_linear_latent / _expand). */
typedef enum { LB_LATENT_FP32 = 0, LB_LATENT_FP16 = 1 } lb_latent_dtype;

/* Latent states of a LittleBit linear (Sec. 5, KV cache compression; Fig. 5,
 * Table 4): Prop. 1 split after its latent scale.  Per path,
 *     z_p[t][j] = l_p[j] * sum_i V_p,sign[i][j] g_p[i] X[t][i]
 * written row-major as z [T][r_0 + r_1] (path 0's r_0 columns, then path
 * 1's).  Caching z of the key and value projections in place of their
 * outputs divides the KV cache by d_kv / (r_0 + r_1) (Table 4 lists
 * d_model / r for one path); littlebit_linear_expand turns z back into the
 * projection's output.
 * x: bf16 [T][d_in]; z: device, 16-byte aligned, in z_dtype: LB_LATENT_FP32,
 * or LB_LATENT_FP16 (round to nearest even; a magnitude above 65504 becomes
 * inf).  ws: littlebit_workspace_size(L, T) bytes, rules as for the forward.
 * T = 0 is a no-op.  Shape rules and the choice of path (tensor-core stage 1
 * with fp16 operands, or the CUDA-core stage 1 with an fp32 reduction) are
 * those of littlebit_linear_forward for the same L and T, except that one
 * token also takes the CUDA-core stage. */
lb_status littlebit_linear_latent(const lb_linear *L, const uint16_t *x, int64_t T, void *z,
                                  int32_t z_dtype, void *ws, size_t ws_bytes,
                                  lb_stream_t stream);

/* The projection's output from latent states in littlebit_linear_latent's
 * layout: Y[t][o] = sum_p h_p[o] sum_j U_p,sign[o][j] z_p[t][j] (Prop. 1's
 * outer part, paths summed by Eq. 6), so that expanding the latent of X
 * gives the forward of X up to rounding.  z: device [T][r_0 + r_1] in
 * z_dtype, 16-byte aligned; y: [T][d_out] in y_dtype.  ws:
 * littlebit_workspace_size(L, T) bytes.  T = 0 is a no-op.  Path: the
 * tensor-core stage 2 where the forward would take it (an fp32 z is first
 * rounded to fp16 in ws), else the CUDA-core stage 2 (fp32 arithmetic). */
lb_status littlebit_linear_expand(const lb_linear *L, const void *z, int32_t z_dtype, int64_t T,
                                  void *y, int32_t y_dtype, void *ws, size_t ws_bytes,
                                  lb_stream_t stream);

/* Output buffers of one path for littlebit_dual_svid: device memory in the
 * layouts of lb_path (the caller allocates them). */
typedef struct {
    int32_t r;           /* rank of this path, 1 <= r <= min(d_out, d_in), r <= 1024 */
    uint32_t *v_bits;    /* V_sign, [ceil(d_in/32)][r] words */
    uint32_t *u_bits;    /* U_sign, [d_out][ceil(r/32)] words */
    uint16_t *g;         /* fp16 [d_in] */
    uint16_t *l;         /* fp16 [r] */
    uint16_t *h;         /* fp16 [d_out] */
} lb_path_init;

/* Workspace bytes littlebit_dual_svid needs (0 if the arguments are invalid). */
size_t littlebit_dual_svid_workspace_size(int32_t d_out, int32_t d_in, int32_t n_paths,
                                          const lb_path_init *paths);

/* Dual-SVID initialisation (Sec. 3.2) of a LittleBit linear from a dense
 * weight, with Residual Compensation (Sec. 3.3): path 0 from W, path 1 (if
 * n_paths = 2) from the residual W - W_hat_0, where W_hat_0 uses path 0's
 * scales as stored (fp16).  Per path, with the path's rank r:
 *   (1) truncated SVD R ~ U' V'^T, the singular values split evenly
 *       (U' = U_r diag(sqrt s), V' = V_r diag(sqrt s)); the joint sign of each
 *       singular pair makes the largest-magnitude entry of v_j positive;
 *   (2) U_sign = sign(U'), V_sign = sign(V'), sign(0) = +1;
 *   (3) |U'| ~ h l_u^T and |V'| ~ g l_v^T, each the leading singular pair of
 *       the nonnegative matrix with its singular value split evenly, and
 *       l = l_u . l_v; h, g, l rounded to fp16 (nearest even).
 * The SVD is computed by subspace iteration (iters >= 1 passes of
 * Y = R Q, Q = R^T Y with Cholesky-QR re-orthonormalisation, 8 columns of
 * oversampling, then a Rayleigh-Ritz step); it converges to the exact
 * truncated SVD when the r-th and (r + 9)-th singular values are apart.
 * W: DEVICE fp32 row-major [d_out][d_in]; paths: HOST array of n_paths
 * (1 or 2) output descriptors.  ws: littlebit_dual_svid_workspace_size
 * bytes, 256-byte aligned (no zero fill needed).  Its GEMMs are the
 * library's own fp32 / fp64 CUDA-core GEMM (full-precision products) on the
 * given stream; the library keeps no handle.  Errors: LB_ERR_INVALID_ARG (shapes, ranks,
 * pointers), LB_ERR_WORKSPACE, LB_ERR_CUDA. */
lb_status littlebit_dual_svid(const float *W, int32_t d_out, int32_t d_in, int32_t n_paths,
                              const lb_path_init *paths, int32_t iters, void *ws, size_t ws_bytes,
                              lb_stream_t stream);

/* QAT (quantization-aware training) form of one path: the latent full-
 * precision factors the forward binarises (Eq. 2) and fp32 scales.  All
 * pointers are device memory, fp32, row-major. */
typedef struct {
    int32_t r;           /* rank, 1 <= r <= 1024 */
    const float *u;      /* latent U, [d_out][r] */
    const float *v;      /* latent V, [d_in][r] */
    const float *g;      /* [d_in] */
    const float *l;      /* [r] */
    const float *h;      /* [d_out] */
} lb_train_path;

typedef struct {
    int32_t d_in, d_out, n_paths;   /* n_paths 1 or 2 */
    lb_train_path path[2];
} lb_train_linear;

/* Gradient buffers of one path (device, fp32, the shapes of u, v, g, l, h);
 * overwritten. */
typedef struct {
    float *du, *dv, *dg, *dl, *dh;
} lb_train_grad;

/* Workspace bytes littlebit_train_forward / littlebit_train_backward need for
 * T tokens (0 if the arguments are invalid). */
size_t littlebit_train_workspace_size(const lb_train_linear *L, int64_t T);

/* QAT forward: Y = sum_p Prop. 1 with U_sign = sign(U), V_sign = sign(V)
 * (sign(0) = +1) of the latent factors.  x: fp32 [T][d_in]; y: fp32
 * [T][d_out].  The two products per path run on the tensor cores with TF32
 * inputs (the +-1 factors are exact; x and the latent z = l . (X . g) V_sign
 * round to 10 mantissa bits) and fp32 accumulation.  T = 0 is a no-op. */
lb_status littlebit_train_forward(const lb_train_linear *L, const float *x, int64_t T, float *y,
                                  void *ws, size_t ws_bytes, lb_stream_t stream);

/* QAT backward (the paper's training, SmoothSign): given dy = dLoss/dY
 * (fp32 [T][d_out]) and the forward's input x, writes per path dLoss/dU,
 * dLoss/dV, dLoss/dg, dLoss/dl, dLoss/dh into grads[p] (HOST array of
 * n_paths descriptors) and dLoss/dX into dx (fp32 [T][d_in], may be NULL).
 * Through the sign the derivative is SmoothSign's proxy
 * d tanh(k x)/dx = k (1 - tanh^2(k x)) with k = k_smooth (the paper: 100).
 * Five GEMM-shaped products per path on the tensor cores (TF32 inputs, fp32
 * accumulation); the scale gradients and the SmoothSign factor are fused into
 * the reductions that follow them. */
lb_status littlebit_train_backward(const lb_train_linear *L, const float *x, const float *dy,
                                   int64_t T, float k_smooth, const lb_train_grad *grads,
                                   float *dx, void *ws, size_t ws_bytes, lb_stream_t stream);

/* The same backward reusing its forward, as a training framework keeps a
 * forward's activations for the backward: littlebit_train_forward leaves in
 * its workspace the signs of U and V folded with h and g, l, the latent t
 * and z = l . t, and a fingerprint of (L's shapes and pointers, x, T); this
 * call uses them instead of recomputing them (the sign folds and the t
 * product are the part of a backward the forward already did).  Its
 * arguments and results are those of littlebit_train_backward.  Contract:
 * the workspace's most recent forward was littlebit_train_forward with the
 * same L, x and T, and neither the factors, the scales nor x have changed
 * since (a backward may come in between).  A fingerprint that differs is
 * refused on the device: LB_ERR_PLAN is recorded in the workspace's error
 * word (read it with littlebit_poll_error) and the gradients are
 * meaningless. */
lb_status littlebit_train_backward_saved(const lb_train_linear *L, const float *x,
                                         const float *dy, int64_t T, float k_smooth,
                                         const lb_train_grad *grads, float *dx, void *ws,
                                         size_t ws_bytes, lb_stream_t stream);

/* Workspace bytes littlebit_stack_prepare / littlebit_stack_forward need
 * (0 if the arguments are invalid). */
size_t littlebit_stack_workspace_size(const lb_linear *lin, int32_t n_layers, int32_t head_dim);

/* Prepares a stack workspace for the linears lin[0 .. 7*n_layers): validates
 * them (same rules as littlebit_stack_forward), writes their device
 * descriptor table into ws, zeroes its counters and accumulators and records
 * a fingerprint of (lin, n_layers, head_dim).  Enqueued on the stream.  Call
 * it once per workspace, again whenever the linears change, and after any
 * error a stack launch recorded in the workspace. */
lb_status littlebit_stack_prepare(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                                  void *ws, size_t ws_bytes, lb_stream_t stream);

/* One decode step, at sequence position 0, of n_layers Llama-shaped decoder
 * blocks whose seven linears are LittleBit linears, lin[7*l + {0..6}] =
 * q, k, v, o, gate, up, down of layer l.  The paper's end-to-end setting
 * (App. I.3) replaces only nn.Linear; the rest of the block is computed here
 * in fp32 with unit RMSNorm weights.  With rho(v) = v / sqrt(mean(v^2)) and
 * a = x0, each layer computes
 *     n = rho(a);  q = Q(n);  k = K(n);  v = V(n)
 *     attn = v broadcast over the query heads of each kv head (attention over
 *            a one-position context: the softmax of a single score is 1)
 *     h = a + O(attn)
 *     n = rho(h);  m = silu(Gate(n)) * Up(n);  a = h + Down(m)
 * Shapes: q, o d->d; k, v d->d_kv; gate, up d->d_ff; down d_ff->d, with
 * d = n_heads * head_dim, d_kv = n_kv_heads * head_dim and n_heads a multiple
 * of n_kv_heads (else LB_ERR_INVALID_ARG); every layer has the same shapes
 * and ranks, d and d_ff are multiples of 32 (else LB_ERR_UNSUPPORTED).
 * lin is a HOST array of 7*n_layers structs holding device pointers.
 * x0: bf16 [d]; out: fp32 [d], the last a; q_out: fp32 [n_layers][d] or NULL;
 * kv_out: fp32 [n_layers][2][d_kv] (k then v) or NULL.  ws must have been
 * prepared for the same lin array by littlebit_stack_prepare: the launch
 * compares fingerprints on the device and, on a mismatch, records
 * LB_ERR_PLAN in the sticky error word and writes nothing.  Runs as ONE
 * persistent kernel with one CTA per SM (LB_ERR_UNSUPPORTED if the GPU
 * cannot hold that grid) and leaves the workspace ready for the next call;
 * its 4 grid-wide exchanges per layer use the bounded wait described above.
 * Calls that share a workspace must not overlap in time. */
lb_status littlebit_stack_forward(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                                  const uint16_t *x0, float *out, float *q_out, float *kv_out,
                                  void *ws, size_t ws_bytes, lb_stream_t stream);

/* ---------------------------------------------------------------- decode at position p
 * The paper's end-to-end decoding setting (App. I.3, Table 12: Llama2
 * decoding with only nn.Linear replaced by LittleBit, attention and the norms
 * left dense) as one decode step at any position p of a KV cache.
 * n_heads query heads and n_kv_heads key/value heads of head_dim dimensions:
 * d = n_heads * head_dim, d_kv = n_kv_heads * head_dim.  The linears are
 * lin[7*l + {0..6}] = q, k, v, o, gate, up, down of layer l (HOST array of
 * structs holding device pointers), shapes as for littlebit_stack_forward
 * and the same in every layer (else LB_ERR_UNSUPPORTED). */
typedef struct {
    int32_t n_layers, n_heads, n_kv_heads;
    int32_t head_dim;   /* 64, 128 or 256 */
    int32_t max_pos;    /* KV cache rows per layer, 1 .. 8192 */
    float rope_base;    /* rotary base, > 1 (10000 for Llama 2) */
} lb_decoder_shape;

/* Workspace bytes littlebit_decoder_step needs (0 if the arguments are invalid). */
size_t littlebit_decoder_workspace_size(const lb_linear *lin, const lb_decoder_shape *S);

/* One decode step of the token x (bf16 [d]) at position p = *pos (a DEVICE
 * int32, read by the step's kernels and incremented by its last one, so the
 * same sequence of launches serves every token and can be captured once as a
 * CUDA graph).  With rho(v) = v / sqrt(mean(v^2)) and a = x, each layer:
 *     n = rho(a);  q, k, v = Q(n), K(n), V(n)
 *     rotary embedding of q and k at p, per head: the pair (i, i + head_dim/2)
 *       rotated by theta_i = p * rope_base^(-2i/head_dim)
 *     kcache[l][p] = k;  vcache[l][p] = v
 *     attn_h = sum_{t<=p} softmax_t(q_h . k_{t,g} / sqrt(head_dim)) v_{t,g},
 *       g = h / (n_heads / n_kv_heads)
 *     a += O(attn);  n = rho(a);  a += Down(silu(Gate(n)) * Up(n))
 * All activations are fp32 (the linears take them as fp32 inputs).  kcache,
 * vcache: fp32 [n_layers][max_pos][d_kv]; rows < p must hold the earlier
 * steps' keys and values, rows > p are not read.  out: fp32 [d], the last a.
 * A position outside [0, max_pos) records LB_ERR_RANGE in the decoder
 * workspace's error word and the step writes nothing (read it with
 * littlebit_decoder_poll_error).  Every linear's d_out and ranks must be
 * multiples of 8 (else LB_ERR_UNSUPPORTED).  ws: zero-filled before first
 * use, not shared with concurrent calls.  Enqueues 2 + 5 * n_layers launches
 * on the stream when q / k / v share a shape (up to 1 + 10 * n_layers
 * otherwise): per layer the single-token LittleBit linears, with q / k / v
 * (or k / v) and gate / up each grouped into one launch when they share a
 * shape (as littlebit_linear_forward_multi) -- a grouped launch also does the
 * residual add and RMS norm ahead of it -- down reading silu(gate) * up
 * itself, the attention kernel, and the norm kernels the grouping leaves. */
lb_status littlebit_decoder_step(const lb_linear *lin, const lb_decoder_shape *S,
                                 const uint16_t *x, float *kcache, float *vcache, int32_t *pos,
                                 float *out, void *ws, size_t ws_bytes, lb_stream_t stream);

/* littlebit_poll_error over a decoder workspace: the step's own error word
 * and each linear's, all cleared; returns the first error found, or LB_OK. */
lb_status littlebit_decoder_poll_error(const lb_linear *lin, const lb_decoder_shape *S, void *ws,
                                       lb_stream_t stream);

/* One token (T = 1) through M LittleBit linears of one shape that read the
 * same input, in one launch: a decoder layer's q / k / v or gate / up
 * projections, or M independent weight sets (Prop. 1 and Eq. 6 per linear,
 * as littlebit_linear_forward).  L: HOST array of M structs (device
 * pointers), 1 <= M <= 24, all with the same d_in, d_out, n_paths and ranks,
 * d_out and the ranks multiples of 8 (else LB_ERR_UNSUPPORTED; other shape
 * errors LB_ERR_INVALID_ARG).  x: bf16 [d_in]; y: [M][d_out] in y_dtype,
 * row m the output of L[m].  One persistent launch of one CTA per SM that
 * streams the linears' factors through shared memory and overlaps each
 * linear's exchange with the next linears' work; the results equal M calls
 * of littlebit_linear_forward at T = 1.  ws: littlebit_multi_workspace_size
 * bytes, zero-filled before first use; a workspace serves one (shape, M) and
 * calls on it must not overlap in time. */
size_t littlebit_multi_workspace_size(const lb_linear *L, int32_t M);
lb_status littlebit_linear_forward_multi(const lb_linear *L, int32_t M, const uint16_t *x,
                                         void *y, int32_t y_dtype, void *ws, size_t ws_bytes,
                                         lb_stream_t stream);

/* The forward of littlebit_linear_forward for callers that cannot allocate
 * device memory.  The paper has no counterpart: this exists for hosts such as
 * serving loops and plugins whose device memory is owned by someone else or
 * whose hot path may not call cudaMalloc (it can synchronise the whole device
 * and take unbounded time), so they cannot provide a workspace.
 *
 * Same arguments and results as littlebit_linear_forward minus the
 * workspace; it runs the two-launch CUDA-core path (any T).  Its scratch is
 * a 256 KiB array compiled into the library, held by every GPU that loads
 * the library until the process exits, and shared by all calls: it allocates
 * nothing and calls no allocating routine.
 *   - Limit: T * (sum of the paths' ranks) <= 65536 fp32 values; a larger
 *     request returns LB_ERR_WORKSPACE without launching anything.
 *   - The first call in each CUDA context looks up the array's device
 *     address (cudaGetSymbolAddress, with that context's device current);
 *     make that first call before any stream capture.  Later calls in the
 *     same context reuse the address; a new context on the device (after
 *     cudaDeviceReset, or another context made current) gets a fresh
 *     look-up on its first call, which again belongs before any capture.
 *   - Each call clears the part of the array it uses before adding into it,
 *     but the array keeps the last call's contents afterwards.  Calls whose
 *     kernels overlap on the GPU (different streams, or different host
 *     threads, without ordering between them) race on the shared array:
 *     order them, e.g. issue them on one stream. */
lb_status littlebit_linear_forward_noalloc(const lb_linear *L, const uint16_t *x, int64_t T,
                                           void *y, int32_t y_dtype, lb_stream_t stream);

/* Synchronises the stream, reads the workspace's sticky error word, clears
 * it, and returns LB_OK or the recorded error (LB_ERR_TIMEOUT, LB_ERR_PLAN). */
lb_status littlebit_poll_error(void *ws, lb_stream_t stream);

/* Diagnostic for the bounded grid-wide wait used by the persistent kernels:
 * launches one CTA that waits on an arrival which never comes.  The wait
 * gives up after its limit (about one second), records LB_ERR_TIMEOUT in the
 * workspace's sticky error word and the kernel returns; read it with
 * littlebit_poll_error.  ws: a zero-filled workspace of at least 256 bytes. */
lb_status littlebit_selftest_wait_timeout(void *ws, lb_stream_t stream);

/* Diagnostic: the latency floor of the exchange that the single-token
 * kernels run between stage 1 and stage 2 of every linear (Prop. 1: the
 * rank-r partial sums t = V_sign^T (g . x) of every CTA's input slice,
 * all-reduced across the GPU before stage 2).  One persistent launch, one CTA
 * per SM, runs n_rounds dependent exchanges of sizes[k % n_sizes] elements
 * (1 <= n_sizes <= 8, 1 <= sizes[i] <= 2048) with the polling of
 * littlebit_stack_forward, optionally (cluster = 2) its two-CTA
 * distributed-shared-memory pre-reduction, and the encoding of the stack
 * (words = 1: one 64-bit word per element at a bounded scale) or of the
 * single-linear kernels (words = 2: the exact hi / lo pair), and nothing
 * else: elapsed time / n_rounds is the exchange's cost on the critical path.  ws: 256-byte aligned,
 * littlebit_selftest_exchange_workspace_size bytes, header zero-filled before
 * the first use (the call clears the rest); an error (a wait that ran out)
 * is recorded in the header like the other kernels', read with
 * littlebit_poll_error.  The paper has no counterpart: it is a measurement. */
size_t littlebit_selftest_exchange_workspace_size(int32_t n_rounds, const int32_t *sizes,
                                                   int32_t n_sizes);
lb_status littlebit_selftest_exchange(int32_t n_rounds, const int32_t *sizes, int32_t n_sizes,
                                      int32_t cluster, int32_t words, void *ws, size_t ws_bytes,
                                      lb_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* LITTLEBIT_H */
