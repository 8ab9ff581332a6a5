// lb_kernels.h -- host-side launchers of the LittleBit kernels (internal).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "littlebit.h"

namespace lb {

struct LinDesc;

// Shape and pointer checks of one linear, as littlebit_linear_forward does them.
lb_status validate_linear(const lb_linear *L);

// Two-launch CUDA-core path for any T (lb_generic.cu).  Stage 1 writes the
// latent z = l . ((X . g) V_sign) as fp32 [T][r_0 + r_1] (z32 is zeroed by the
// launcher), stage 2 reads z (fp32, or fp16 when z_half) and writes Y.
// launch_generic runs both with z in z_ws: generic_ws_floats() floats.
size_t generic_ws_floats(const lb_linear &L, int64_t T);
cudaError_t launch_generic(const lb_linear &L, const uint16_t *x, int64_t T, void *y, int y_fp32,
                           float *z_ws, int num_sms, cudaStream_t s);
cudaError_t launch_latent_generic(const lb_linear &L, const uint16_t *x, int64_t T, float *z32,
                                  int num_sms, cudaStream_t s);
cudaError_t launch_expand_generic(const lb_linear &L, const void *z, int z_half, int64_t T,
                                  void *y, int y_fp32, cudaStream_t s);
// z16[i] = fp16(z32[i]) (round to nearest even), n elements.
cudaError_t launch_to_half(const float *z32, uint16_t *z16, long long n, cudaStream_t s);

// Single-launch decode of one linear, T = 1 (lb_decode.cu): ranks multiples
// of 8, d_out a multiple of 8.  xw: decode_ws_bytes of exchange words (two
// buffers), zero before the first launch; completed launches keep them so.
// Returns cudaErrorCooperativeLaunchTooLarge when the grid cannot be co-resident.
bool decode_supported(const lb_linear &L, int num_sms);
size_t decode_ws_bytes(const lb_linear &L);
cudaError_t launch_decode(const lb_linear &L, const void *x, int x_fp32, void *y, int y_fp32,
                          unsigned *ws_words, void *xw, int num_sms, cudaStream_t s);

// T = 1 through M linears of one shape that read the same x (lb_multi.cu).
// x_fp32: 0 bf16 x, 1 fp32 x, 3 residual input: x = res_a + res_y (fp32,
// written back to res_a) and every output scaled by 1 / rms(x).
constexpr int kMaxMultiLinears = 24;
bool multi_supported(const lb_linear *L, int M, int num_sms);
size_t multi_ws_bytes(const lb_linear &L, int M);
cudaError_t launch_decode_multi(const lb_linear *L, int M, const void *x, int x_fp32, void *y,
                                int y_fp32, unsigned *ws_words, void *xw, int num_sms,
                                cudaStream_t s, float *res_a = nullptr,
                                const float *res_y = nullptr);

// Persistent decode of the seven-linear-per-layer stack (lb_stack.cu).
struct StackShape {
    int n_layers, d, dkv, dff, head_dim;
};
size_t stack_ws_bytes_after_header(const lb_linear *lin, int n_layers);
// `cluster`: CTAs per thread-block cluster, 1 or 2 (with 2 the stage-1
// partials of a pair meet in distributed shared memory before the exchange).
// Writes the device descriptor table and the per-CTA programs for num_sms
// CTAs, zeroes counters and accumulators, and stores the plan fingerprint.
// cudaErrorNotSupported when the shapes or the programs do not fit.
cudaError_t launch_stack_prepare(const lb_linear *lin, int n_layers, const StackShape &shape,
                                 int num_sms, int cluster, unsigned long long plan,
                                 unsigned *ws_words, char *ws_after_header, cudaStream_t s);
// Whether the one-launch stack kernel handles these shapes on this GPU
// (ranks multiples of 8, head_dim multiple of 32, d_kv multiple of 8, the
// shared-memory plan fits, num_sms a multiple of the cluster size).
bool stack_supported(const lb_linear *lin, const StackShape &shape, int num_sms, int cluster);
// The grid of the one-launch stack kernel on this GPU: a whole number of
// co-resident thread-block clusters, at most num_sms CTAs (0: cannot launch).
// Programs, fingerprints and launches all use this count.
int stack_grid_ctas(const lb_linear *lin, const StackShape &shape, int num_sms, int cluster);
// One persistent launch; leaves counters and accumulators zeroed.
cudaError_t launch_stack(const lb_linear *lin, int n_layers, const StackShape &shape,
                         unsigned long long plan, const uint16_t *x0, float *out, float *q_out,
                         float *kv_out, unsigned *ws_words, char *ws_after_header, int num_sms,
                         int cluster, cudaStream_t s);

// Many-token path on the tensor cores (lb_prefill.cu).  The latent half
// writes z = l . ((X . g) V_sign) as fp16 into z16, or as fp32 into z32 when
// that is not null; the expansion half reads an fp16 z ([T][r_0 + r_1],
// 16-byte aligned).  ws: prefill_ws_bytes; launch_prefill keeps z at its start.
bool prefill_supported(const lb_linear &L, int64_t T);
size_t prefill_ws_bytes(const lb_linear &L, int64_t T);
cudaError_t launch_prefill(const lb_linear &L, const uint16_t *x, int64_t T, void *y, int y_fp32,
                           unsigned *ws_words, void *ws, cudaStream_t s);
cudaError_t launch_prefill_latent(const lb_linear &L, const uint16_t *x, int64_t T, uint16_t *z16,
                                  float *z32, unsigned *ws_words, void *ws, cudaStream_t s);
cudaError_t launch_prefill_expand(const lb_linear &L, const uint16_t *z16, int64_t T, void *y,
                                  int y_fp32, unsigned *ws_words, void *ws, cudaStream_t s);

// Column-major C = alpha op(A) op(B) + beta C on the CUDA cores, fp32 or fp64
// (lb_simt_gemm.cu): op(A) M x K is A[m + k lda] or, with ta, A[k + m lda];
// op(B) K x N likewise; beta = 0 does not read C.
cudaError_t gemm_simt(bool ta, bool tb, int M, int N, int K, float alpha, const float *A,
                      long long lda, const float *B, long long ldb, float beta, float *C,
                      long long ldc, cudaStream_t s);
cudaError_t gemm_simt(bool ta, bool tb, int M, int N, int K, double alpha, const double *A,
                      long long lda, const double *B, long long ldb, double beta, double *C,
                      long long ldc, cudaStream_t s);

// Dual-SVID initialisation (lb_svid.cu): W fp32 row-major [d_out][d_in],
// per path the output sign words and fp16 scales; ws: svid_ws_bytes.
int svid_k(int r, int d_out, int d_in);
size_t svid_ws_bytes(int d_out, int d_in, const int *ranks, int n_paths);
cudaError_t launch_dual_svid(const float *W, int d_out, int d_in, int n_paths, const int *ranks,
                             uint32_t *const *v_bits, uint32_t *const *u_bits, uint16_t *const *g,
                             uint16_t *const *l, uint16_t *const *h, int iters, void *ws,
                             cudaStream_t s);

// C[M][N] (+)= A[M][K] B[N][K]^T on the tensor cores, TF32 operands and fp32
// accumulation (lb_gemm.cu).  An operand is fp32, row-major [rows][ld] with
// its K = k columns first (ld >= k, ld a multiple of 4, 16-byte aligned base);
// C is row-major at ldc.  A long K over few tiles is split into slices whose
// partials go to part (gemm_part_floats floats; with less the split is
// dropped) and are added in slice order.  A bounded wait that runs out
// records LB_ERR_TIMEOUT in *err; launches return early while it is set.
struct GemmOperand {
    const float *p;
    int rows, k;
    long long ld;
};
bool gemm_operand_ok(const GemmOperand &A);
size_t gemm_part_floats(int M, int N, int K);
// C2 (optional, not with accumulate): C2[m][n] = C[m][n] * scale2[n] at ldc2,
// written beside C (a column scaling that follows the product).
cudaError_t gemm_tf32(const GemmOperand &A, const GemmOperand &B, float *C, long long ldc,
                      bool accumulate, float *part, size_t part_floats, unsigned *err,
                      cudaStream_t s, float *C2 = nullptr, const float *scale2 = nullptr,
                      long long ldc2 = 0);

// QAT forward / backward on latent factors (lb_qat.cu); ws: qat_ws_bytes for
// the sum of the paths' ranks (a 256-byte header whose first word is the
// error word, then the buffers).
size_t qat_ws_bytes(int d_in, int d_out, int rsum, long long T);
// tag: a fingerprint of (L, x, T); the forward records it in the workspace,
// a backward with saved = true reuses the forward's folded factors, l, t and
// z instead of recomputing them and records LB_ERR_PLAN if the tags differ.
cudaError_t launch_train_forward(const lb_train_linear &L, const float *x, long long T, float *y,
                                 void *ws, unsigned long long tag, cudaStream_t s);
cudaError_t launch_train_backward(const lb_train_linear &L, const float *x, const float *dy,
                                  long long T, float k, const lb_train_grad *G, float *dx, void *ws,
                                  bool saved, unsigned long long tag, cudaStream_t s);

// Bounded-wait diagnostic (lb_persistent.cu).
cudaError_t launch_wait_timeout(unsigned *ws_words, cudaStream_t s);

// Exchange-chain diagnostic (lb_xchain.cu): n_rounds dependent all-reduces
// of sizes[k % n_sizes] elements over the grid (cluster 1 or 2); buf holds
// n_rounds buffers and is cleared by the launcher.
size_t xchain_ws_bytes(int n_rounds, const int *sizes, int n_sizes);
cudaError_t launch_xchain(int n_rounds, const int *sizes, int n_sizes, int cluster, int words,
                          unsigned *ws_words, void *buf, int num_sms, cudaStream_t s);

// Sign packing (lb_pack.cu).
cudaError_t launch_pack(const int8_t *signs, int64_t rows, int64_t cols, int layout,
                        uint32_t *out, int32_t *bad, cudaStream_t s);

}  // namespace lb
