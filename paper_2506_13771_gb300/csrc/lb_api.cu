// lb_api.cu -- the extern "C" entry points of liblittlebit.so: argument
// validation, workspace layout and dispatch to the kernels.  See
// include/littlebit.h for the contract of every function.
#include <cstdint>
#include <cstdlib>
#include <cstring>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace {

using lb::kWsHeader;

constexpr int kMaxDevices = 64;
int g_num_sms[kMaxDevices];  // per-device SM count cache (0 = unknown)

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

lb_status from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return LB_OK;
    if (e == cudaErrorCooperativeLaunchTooLarge) {
        cudaGetLastError();
        return LB_ERR_UNSUPPORTED;
    }
    return LB_ERR_CUDA;
}

lb_status num_sms(int *out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LB_ERR_CUDA;
    if (dev >= 0 && dev < kMaxDevices && g_num_sms[dev] > 0) {
        *out = g_num_sms[dev];
        return LB_OK;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
        return LB_ERR_CUDA;
    if (dev >= 0 && dev < kMaxDevices) g_num_sms[dev] = n;
    *out = n;
    return LB_OK;
}

// Shape and pointer checks of one linear.  Returns LB_OK, LB_ERR_INVALID_ARG
// or LB_ERR_UNSUPPORTED.
lb_status check_linear(const lb_linear *L) {
    if (!L) return LB_ERR_INVALID_ARG;
    if (L->d_in <= 0 || L->d_out <= 0) return LB_ERR_INVALID_ARG;
    if (L->n_paths != 1 && L->n_paths != 2) return LB_ERR_INVALID_ARG;
    for (int p = 0; p < L->n_paths; ++p) {
        const lb_path &P = L->path[p];
        if (P.r <= 0) return LB_ERR_INVALID_ARG;
        if (!P.v_bits || !P.u_bits || !P.g || !P.l || !P.h) return LB_ERR_INVALID_ARG;
        if (!aligned16(P.v_bits) || !aligned16(P.u_bits) || !aligned16(P.g) || !aligned16(P.l) ||
            !aligned16(P.h))
            return LB_ERR_INVALID_ARG;
        if (P.r > lb::kMaxRank) return LB_ERR_UNSUPPORTED;
    }
    if (L->d_in % 32 != 0) return LB_ERR_UNSUPPORTED;
    return LB_OK;
}

bool same_shape(const lb_linear &a, const lb_linear &b) {
    if (a.d_in != b.d_in || a.d_out != b.d_out || a.n_paths != b.n_paths) return false;
    for (int p = 0; p < a.n_paths; ++p)
        if (a.path[p].r != b.path[p].r) return false;
    return true;
}

// Shape checks of the seven-linear-per-layer chain.
lb_status check_stack(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                      lb::StackShape *shape) {
    if (!lin || n_layers <= 0 || head_dim <= 0) return LB_ERR_INVALID_ARG;
    for (int i = 0; i < 7 * n_layers; ++i) {
        lb_status st = check_linear(&lin[i]);
        if (st != LB_OK) return st;
    }
    const int d = lin[0].d_in, dkv = lin[1].d_out, dff = lin[4].d_out;
    // q: d->d, k, v: d->dkv, o: d->d, gate, up: d->dff, down: dff->d
    const bool chain = lin[0].d_out == d && lin[1].d_in == d && lin[2].d_in == d &&
                       lin[2].d_out == dkv && lin[3].d_in == d && lin[3].d_out == d &&
                       lin[4].d_in == d && lin[5].d_in == d && lin[5].d_out == dff &&
                       lin[6].d_in == dff && lin[6].d_out == d;
    if (!chain) return LB_ERR_INVALID_ARG;
    for (int i = 7; i < 7 * n_layers; ++i)
        if (!same_shape(lin[i], lin[i - 7])) return LB_ERR_UNSUPPORTED;
    // attention heads: d = n_heads * head_dim, dkv = n_kv_heads * head_dim,
    // n_heads a multiple of n_kv_heads (grouped-query attention)
    if (d % head_dim != 0 || dkv % head_dim != 0 || (d / head_dim) % (dkv / head_dim) != 0)
        return LB_ERR_INVALID_ARG;
    if (d % 32 != 0 || dff % 32 != 0) return LB_ERR_UNSUPPORTED;
    shape->head_dim = head_dim;
    shape->n_layers = n_layers;
    shape->d = d;
    shape->dkv = dkv;
    shape->dff = dff;
    return LB_OK;
}

// CTAs per thread-block cluster of the stack kernel: 2 when the environment
// variable LB_STACK_CLUSTER is "2", else 1 (read at every prepare and
// forward; the fingerprint holds it, so a workspace prepared with the other
// value is refused with LB_ERR_PLAN).
int stack_cluster() {
    const char *v = std::getenv("LB_STACK_CLUSTER");
    return v && v[0] == '2' && v[1] == '\0' ? 2 : 1;
}

// FNV-1a over the host description of a stack (shapes, ranks and pointers),
// the SM count the per-CTA programs were built for and the cluster size.
unsigned long long stack_fingerprint(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                                     int sms, int cluster) {
    unsigned long long h = 1469598103934665603ull;
    auto mix = [&h](unsigned long long v) {
        for (int b = 0; b < 8; ++b) {
            h ^= (v >> (8 * b)) & 0xffu;
            h *= 1099511628211ull;
        }
    };
    mix((unsigned long long)n_layers);
    mix((unsigned long long)head_dim);
    mix((unsigned long long)sms);
    mix((unsigned long long)cluster);
    for (int i = 0; i < 7 * n_layers; ++i) {
        const lb_linear &L = lin[i];
        mix((unsigned long long)L.d_in);
        mix((unsigned long long)L.d_out);
        mix((unsigned long long)L.n_paths);
        for (int p = 0; p < L.n_paths; ++p) {
            mix((unsigned long long)L.path[p].r);
            mix(reinterpret_cast<uintptr_t>(L.path[p].v_bits));
            mix(reinterpret_cast<uintptr_t>(L.path[p].u_bits));
            mix(reinterpret_cast<uintptr_t>(L.path[p].g));
            mix(reinterpret_cast<uintptr_t>(L.path[p].l));
            mix(reinterpret_cast<uintptr_t>(L.path[p].h));
        }
    }
    return h | 1ull;  // never 0, the value of a zero-filled workspace
}

// One token goes through the single-launch persistent kernel.
bool use_decode(const lb_linear &, int64_t T) { return T == 1; }

// From this many tokens on, and once the stage-1 output (T x sum of ranks)
// fills a few tensor-core tiles, the layer is a dense contraction worth the
// tensor cores (tcgen05, 128-token tiles).  Below that the two-launch
// CUDA-core path finishes first (measured on GB300 for the 4096 <-> 11008
// shapes: at rank sums 256 and T = 16 it takes 25 us against 30-37 us, at
// T = 32 they tie, from T = 64 or rank sum 1024 on the tensor cores win).
constexpr int64_t kPrefillMinTokens = 16;
constexpr int64_t kPrefillMinLatent = 8192;
bool use_prefill(const lb_linear &L, int64_t T) {
    int64_t n1 = 0;
    for (int p = 0; p < L.n_paths; ++p) n1 += L.path[p].r;
    return T >= kPrefillMinTokens && T * n1 > kPrefillMinLatent && lb::prefill_supported(L, T);
}

// Workspace of a linear: header | the single-token kernel's exchange words
// (a region no other path writes, so it stays clean between its launches) |
// the data of the path a call takes.
size_t linear_data_offset(const lb_linear &L) { return kWsHeader + lb::decode_ws_bytes(L); }

}  // namespace

lb_status lb::validate_linear(const lb_linear *L) { return check_linear(L); }

extern "C" {

const char *littlebit_status_string(lb_status s) {
    switch (s) {
        case LB_OK: return "LB_OK";
        case LB_ERR_INVALID_ARG: return "LB_ERR_INVALID_ARG";
        case LB_ERR_UNSUPPORTED: return "LB_ERR_UNSUPPORTED";
        case LB_ERR_CUDA: return "LB_ERR_CUDA";
        case LB_ERR_TIMEOUT: return "LB_ERR_TIMEOUT";
        case LB_ERR_WORKSPACE: return "LB_ERR_WORKSPACE";
        case LB_ERR_PLAN: return "LB_ERR_PLAN";
        case LB_ERR_RANGE: return "LB_ERR_RANGE";
    }
    return "LB_ERR_UNKNOWN";
}

lb_status littlebit_pack(const int8_t *signs, int64_t rows, int64_t cols, int32_t layout,
                         uint32_t *out, int64_t out_words, int32_t *bad, lb_stream_t stream) {
    if (!signs || !out || rows <= 0 || cols <= 0) return LB_ERR_INVALID_ARG;
    if (layout != LB_PACK_U && layout != LB_PACK_V) return LB_ERR_INVALID_ARG;
    const int64_t need = layout == LB_PACK_U ? rows * ((cols + 31) / 32) : ((rows + 31) / 32) * cols;
    if (out_words < need) return LB_ERR_INVALID_ARG;
    if (!aligned16(signs) || !aligned16(out)) return LB_ERR_INVALID_ARG;
    return from_cuda(lb::launch_pack(signs, rows, cols, layout, out, bad, (cudaStream_t)stream));
}

size_t littlebit_workspace_size(const lb_linear *L, int64_t T) {
    if (check_linear(L) != LB_OK || T < 0) return 0;
    const size_t floats = lb::generic_ws_floats(*L, T);
    size_t bytes = (floats * sizeof(float) + 255) & ~(size_t)255;
    if (use_prefill(*L, T) && lb::prefill_ws_bytes(*L, T) > bytes) bytes = lb::prefill_ws_bytes(*L, T);
    return linear_data_offset(*L) + bytes;
}


lb_status littlebit_linear_forward(const lb_linear *L, const uint16_t *x, int64_t T, void *y,
                                   int32_t y_dtype, void *ws, size_t ws_bytes,
                                   lb_stream_t stream) {
    lb_status st = check_linear(L);
    if (st != LB_OK) return st;
    if (T < 0 || (y_dtype != LB_OUT_BF16 && y_dtype != LB_OUT_FP32)) return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (T > INT32_MAX / 8) return LB_ERR_UNSUPPORTED;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_workspace_size(L, T))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    if ((st = num_sms(&sms)) != LB_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    unsigned *words = static_cast<unsigned *>(ws);
    float *data = reinterpret_cast<float *>(static_cast<char *>(ws) + linear_data_offset(*L));
    const int fp32 = y_dtype == LB_OUT_FP32;
    if (use_decode(*L, T) && lb::decode_supported(*L, sms)) {
        cudaError_t e = lb::launch_decode(*L, x, 0, y, fp32, words,
                                          static_cast<char *>(ws) + kWsHeader, sms, s);
        if (e != cudaErrorCooperativeLaunchTooLarge) return from_cuda(e);
        cudaGetLastError();  // too large for one co-resident grid: take the two-launch path
    }
    if (use_prefill(*L, T)) return from_cuda(lb::launch_prefill(*L, x, T, y, fp32, words, data, s));
    return from_cuda(lb::launch_generic(*L, x, T, y, fp32, data, sms, s));
}

size_t littlebit_multi_workspace_size(const lb_linear *L, int32_t M) {
    if (!L || M < 1 || M > lb::kMaxMultiLinears) return 0;
    for (int m = 0; m < M; ++m)
        if (check_linear(&L[m]) != LB_OK) return 0;
    return kWsHeader + lb::multi_ws_bytes(L[0], M);
}

lb_status littlebit_linear_forward_multi(const lb_linear *L, int32_t M, const uint16_t *x,
                                         void *y, int32_t y_dtype, void *ws, size_t ws_bytes,
                                         lb_stream_t stream) {
    if (!L || M < 1 || M > lb::kMaxMultiLinears) return LB_ERR_INVALID_ARG;
    for (int m = 0; m < M; ++m) {
        const lb_status st = check_linear(&L[m]);
        if (st != LB_OK) return st;
    }
    if (y_dtype != LB_OUT_BF16 && y_dtype != LB_OUT_FP32) return LB_ERR_INVALID_ARG;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_multi_workspace_size(L, M))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    lb_status st = num_sms(&sms);
    if (st != LB_OK) return st;
    if (!lb::multi_supported(L, M, sms)) return LB_ERR_UNSUPPORTED;
    const cudaError_t e = lb::launch_decode_multi(
        L, M, x, 0, y, y_dtype == LB_OUT_FP32, static_cast<unsigned *>(ws),
        static_cast<char *>(ws) + kWsHeader, sms, (cudaStream_t)stream);
    return e == cudaErrorCooperativeLaunchTooLarge ? LB_ERR_UNSUPPORTED : from_cuda(e);
}

lb_status littlebit_linear_latent(const lb_linear *L, const uint16_t *x, int64_t T, void *z,
                                  int32_t z_dtype, void *ws, size_t ws_bytes,
                                  lb_stream_t stream) {
    lb_status st = check_linear(L);
    if (st != LB_OK) return st;
    if (T < 0 || (z_dtype != LB_LATENT_FP32 && z_dtype != LB_LATENT_FP16)) return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (T > INT32_MAX / 8) return LB_ERR_UNSUPPORTED;
    if (!x || !z || !aligned16(x) || !aligned16(z)) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_workspace_size(L, T))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    if ((st = num_sms(&sms)) != LB_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    unsigned *words = static_cast<unsigned *>(ws);
    char *data = static_cast<char *>(ws) + linear_data_offset(*L);
    const bool half = z_dtype == LB_LATENT_FP16;
    if (use_prefill(*L, T))
        return from_cuda(lb::launch_prefill_latent(
            *L, x, T, half ? static_cast<uint16_t *>(z) : nullptr,
            half ? nullptr : static_cast<float *>(z), words, data, s));
    if (!half) return from_cuda(lb::launch_latent_generic(*L, x, T, static_cast<float *>(z), sms, s));
    float *z32 = reinterpret_cast<float *>(data);
    cudaError_t e = lb::launch_latent_generic(*L, x, T, z32, sms, s);
    if (e == cudaSuccess)
        e = lb::launch_to_half(z32, static_cast<uint16_t *>(z),
                               (long long)lb::generic_ws_floats(*L, T), s);
    return from_cuda(e);
}

lb_status littlebit_linear_expand(const lb_linear *L, const void *z, int32_t z_dtype, int64_t T,
                                  void *y, int32_t y_dtype, void *ws, size_t ws_bytes,
                                  lb_stream_t stream) {
    lb_status st = check_linear(L);
    if (st != LB_OK) return st;
    if (T < 0 || (z_dtype != LB_LATENT_FP32 && z_dtype != LB_LATENT_FP16) ||
        (y_dtype != LB_OUT_BF16 && y_dtype != LB_OUT_FP32))
        return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (T > INT32_MAX / 8) return LB_ERR_UNSUPPORTED;
    if (!z || !y || !aligned16(z) || !aligned16(y)) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_workspace_size(L, T))
        return LB_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    unsigned *words = static_cast<unsigned *>(ws);
    char *data = static_cast<char *>(ws) + linear_data_offset(*L);
    const int fp32 = y_dtype == LB_OUT_FP32;
    const bool half = z_dtype == LB_LATENT_FP16;
    if (use_prefill(*L, T)) {
        const uint16_t *z16 = static_cast<const uint16_t *>(z);
        if (!half) {
            // the tensor-core stage takes fp16 operands: round z at the start of ws
            uint16_t *zc = reinterpret_cast<uint16_t *>(data);
            const cudaError_t e = lb::launch_to_half(static_cast<const float *>(z), zc,
                                                     (long long)lb::generic_ws_floats(*L, T), s);
            if (e != cudaSuccess) return from_cuda(e);
            z16 = zc;
        }
        return from_cuda(lb::launch_prefill_expand(*L, z16, T, y, fp32, words, data, s));
    }
    return from_cuda(lb::launch_expand_generic(*L, z, half ? 1 : 0, T, y, fp32, s));
}

namespace {
bool check_svid(int32_t d_out, int32_t d_in, int32_t n_paths, const lb_path_init *paths) {
    if (d_out <= 0 || d_in <= 0 || (n_paths != 1 && n_paths != 2) || !paths) return false;
    for (int p = 0; p < n_paths; ++p) {
        const lb_path_init &P = paths[p];
        if (P.r < 1 || P.r > lb::kMaxRank || P.r > d_out || P.r > d_in) return false;
    }
    return true;
}
}  // namespace

size_t littlebit_dual_svid_workspace_size(int32_t d_out, int32_t d_in, int32_t n_paths,
                                          const lb_path_init *paths) {
    if (!check_svid(d_out, d_in, n_paths, paths)) return 0;
    int ranks[2] = {paths[0].r, n_paths > 1 ? paths[1].r : 0};
    return lb::svid_ws_bytes(d_out, d_in, ranks, n_paths);
}

lb_status littlebit_dual_svid(const float *W, int32_t d_out, int32_t d_in, int32_t n_paths,
                              const lb_path_init *paths, int32_t iters, void *ws, size_t ws_bytes,
                              lb_stream_t stream) {
    if (!check_svid(d_out, d_in, n_paths, paths) || !W || !aligned16(W) || iters < 1 ||
        iters > 1000)
        return LB_ERR_INVALID_ARG;
    for (int p = 0; p < n_paths; ++p) {
        const lb_path_init &P = paths[p];
        if (!P.v_bits || !P.u_bits || !P.g || !P.l || !P.h || !aligned16(P.v_bits) ||
            !aligned16(P.u_bits) || !aligned16(P.g) || !aligned16(P.l) || !aligned16(P.h))
            return LB_ERR_INVALID_ARG;
    }
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_dual_svid_workspace_size(d_out, d_in, n_paths, paths))
        return LB_ERR_WORKSPACE;
    int ranks[2];
    uint32_t *vb[2], *ub[2];
    uint16_t *g[2], *l[2], *h[2];
    for (int p = 0; p < n_paths; ++p) {
        ranks[p] = paths[p].r;
        vb[p] = paths[p].v_bits;
        ub[p] = paths[p].u_bits;
        g[p] = paths[p].g;
        l[p] = paths[p].l;
        h[p] = paths[p].h;
    }
    return from_cuda(lb::launch_dual_svid(W, d_out, d_in, n_paths, ranks, vb, ub, g, l, h, iters,
                                          ws, (cudaStream_t)stream));
}

namespace {
// FNV-1a over a QAT linear's shapes and pointers, the input pointer and T:
// what a forward leaves in its workspace is keyed by it.
unsigned long long train_tag(const lb_train_linear *L, const float *x, int64_t T) {
    unsigned long long h = 1469598103934665603ull;
    auto mix = [&h](unsigned long long v) {
        for (int b = 0; b < 8; ++b) {
            h ^= (v >> (8 * b)) & 0xffu;
            h *= 1099511628211ull;
        }
    };
    mix((unsigned long long)L->d_in);
    mix((unsigned long long)L->d_out);
    mix((unsigned long long)L->n_paths);
    for (int p = 0; p < L->n_paths; ++p) {
        const lb_train_path &P = L->path[p];
        mix((unsigned long long)P.r);
        mix(reinterpret_cast<uintptr_t>(P.u));
        mix(reinterpret_cast<uintptr_t>(P.v));
        mix(reinterpret_cast<uintptr_t>(P.g));
        mix(reinterpret_cast<uintptr_t>(P.l));
        mix(reinterpret_cast<uintptr_t>(P.h));
    }
    mix(reinterpret_cast<uintptr_t>(x));
    mix((unsigned long long)T);
    return h;
}

lb_status check_train(const lb_train_linear *L) {
    if (!L || L->d_in <= 0 || L->d_out <= 0 || (L->n_paths != 1 && L->n_paths != 2))
        return LB_ERR_INVALID_ARG;
    for (int p = 0; p < L->n_paths; ++p) {
        const lb_train_path &P = L->path[p];
        if (P.r < 1 || P.r > lb::kMaxRank) return LB_ERR_INVALID_ARG;
        if (!P.u || !P.v || !P.g || !P.l || !P.h || !aligned16(P.u) || !aligned16(P.v) ||
            !aligned16(P.g) || !aligned16(P.l) || !aligned16(P.h))
            return LB_ERR_INVALID_ARG;
    }
    return LB_OK;
}
}  // namespace

size_t littlebit_train_workspace_size(const lb_train_linear *L, int64_t T) {
    if (check_train(L) != LB_OK || T < 0 || T > INT32_MAX) return 0;
    int rsum = 0;
    for (int p = 0; p < L->n_paths; ++p) rsum += L->path[p].r;
    return lb::qat_ws_bytes(L->d_in, L->d_out, rsum, T);
}

lb_status littlebit_train_forward(const lb_train_linear *L, const float *x, int64_t T, float *y,
                                  void *ws, size_t ws_bytes, lb_stream_t stream) {
    lb_status st = check_train(L);
    if (st != LB_OK) return st;
    if (T < 0 || T > INT32_MAX) return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_train_workspace_size(L, T))
        return LB_ERR_WORKSPACE;
    return from_cuda(lb::launch_train_forward(*L, x, T, y, ws, train_tag(L, x, T),
                                              (cudaStream_t)stream));
}

namespace {
lb_status train_backward(const lb_train_linear *L, const float *x, const float *dy, int64_t T,
                         float k_smooth, const lb_train_grad *grads, float *dx, void *ws,
                         size_t ws_bytes, bool saved, lb_stream_t stream) {
    lb_status st = check_train(L);
    if (st != LB_OK) return st;
    if (T < 0 || T > INT32_MAX || !grads || !(k_smooth > 0.f)) return LB_ERR_INVALID_ARG;
    if (T == 0) return LB_OK;
    if (!x || !dy || !aligned16(x) || !aligned16(dy) || (dx && !aligned16(dx)))
        return LB_ERR_INVALID_ARG;
    for (int p = 0; p < L->n_paths; ++p) {
        const lb_train_grad &G = grads[p];
        if (!G.du || !G.dv || !G.dg || !G.dl || !G.dh || !aligned16(G.du) || !aligned16(G.dv) ||
            !aligned16(G.dg) || !aligned16(G.dl) || !aligned16(G.dh))
            return LB_ERR_INVALID_ARG;
    }
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_train_workspace_size(L, T))
        return LB_ERR_WORKSPACE;
    return from_cuda(lb::launch_train_backward(*L, x, dy, T, k_smooth, grads, dx, ws, saved,
                                               train_tag(L, x, T), (cudaStream_t)stream));
}
}  // namespace

lb_status littlebit_train_backward(const lb_train_linear *L, const float *x, const float *dy,
                                   int64_t T, float k_smooth, const lb_train_grad *grads,
                                   float *dx, void *ws, size_t ws_bytes, lb_stream_t stream) {
    return train_backward(L, x, dy, T, k_smooth, grads, dx, ws, ws_bytes, false, stream);
}

lb_status littlebit_train_backward_saved(const lb_train_linear *L, const float *x,
                                         const float *dy, int64_t T, float k_smooth,
                                         const lb_train_grad *grads, float *dx, void *ws,
                                         size_t ws_bytes, lb_stream_t stream) {
    return train_backward(L, x, dy, T, k_smooth, grads, dx, ws, ws_bytes, true, stream);
}

size_t littlebit_stack_workspace_size(const lb_linear *lin, int32_t n_layers, int32_t head_dim) {
    lb::StackShape shape;
    if (check_stack(lin, n_layers, head_dim, &shape) != LB_OK) return 0;
    return kWsHeader + lb::stack_ws_bytes_after_header(lin, n_layers);
}

lb_status littlebit_stack_prepare(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                                  void *ws, size_t ws_bytes, lb_stream_t stream) {
    lb::StackShape shape;
    lb_status st = check_stack(lin, n_layers, head_dim, &shape);
    if (st != LB_OK) return st;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_stack_workspace_size(lin, n_layers, head_dim))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    if ((st = num_sms(&sms)) != LB_OK) return st;
    const int cl = stack_cluster();
    if ((sms = lb::stack_grid_ctas(lin, shape, sms, cl)) <= 0) return LB_ERR_UNSUPPORTED;
    const cudaError_t e = lb::launch_stack_prepare(
        lin, n_layers, shape, sms, cl, stack_fingerprint(lin, n_layers, head_dim, sms, cl),
        static_cast<unsigned *>(ws), static_cast<char *>(ws) + kWsHeader, (cudaStream_t)stream);
    return e == cudaErrorNotSupported ? LB_ERR_UNSUPPORTED : from_cuda(e);
}

lb_status littlebit_stack_forward(const lb_linear *lin, int32_t n_layers, int32_t head_dim,
                                  const uint16_t *x0, float *out, float *q_out, float *kv_out,
                                  void *ws, size_t ws_bytes, lb_stream_t stream) {
    lb::StackShape shape;
    lb_status st = check_stack(lin, n_layers, head_dim, &shape);
    if (st != LB_OK) return st;
    if (!x0 || !out || !aligned16(x0) || !aligned16(out) || (q_out && !aligned16(q_out)) ||
        (kv_out && !aligned16(kv_out)))
        return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < littlebit_stack_workspace_size(lin, n_layers, head_dim))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    if ((st = num_sms(&sms)) != LB_OK) return st;
    const int cl = stack_cluster();
    if ((sms = lb::stack_grid_ctas(lin, shape, sms, cl)) <= 0) return LB_ERR_UNSUPPORTED;
    if (!lb::stack_supported(lin, shape, sms, cl)) return LB_ERR_UNSUPPORTED;
    return from_cuda(lb::launch_stack(lin, n_layers, shape,
                                      stack_fingerprint(lin, n_layers, head_dim, sms, cl), x0,
                                      out, q_out, kv_out, static_cast<unsigned *>(ws),
                                      static_cast<char *>(ws) + kWsHeader, sms, cl,
                                      (cudaStream_t)stream));
}

lb_status littlebit_poll_error(void *ws, lb_stream_t stream) {
    if (!ws) return LB_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaStreamSynchronize(s) != cudaSuccess) return LB_ERR_CUDA;
    unsigned err = 0;
    if (cudaMemcpy(&err, ws, sizeof(unsigned), cudaMemcpyDeviceToHost) != cudaSuccess)
        return LB_ERR_CUDA;
    if (err != 0u) {
        // the error word, and the grid-barrier counters a failed launch may
        // have left behind
        const unsigned zero[3] = {0u, 0u, 0u};
        if (cudaMemcpy(ws, zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
            return LB_ERR_CUDA;
        return (lb_status)err;
    }
    return LB_OK;
}

lb_status littlebit_selftest_wait_timeout(void *ws, lb_stream_t stream) {
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0)) return LB_ERR_WORKSPACE;
    return from_cuda(lb::launch_wait_timeout(static_cast<unsigned *>(ws), (cudaStream_t)stream));
}

size_t littlebit_selftest_exchange_workspace_size(int32_t n_rounds, const int32_t *sizes,
                                                   int32_t n_sizes) {
    if (n_rounds < 1 || !sizes || n_sizes < 1 || n_sizes > 8) return 0;
    return lb::xchain_ws_bytes(n_rounds, sizes, n_sizes);
}

lb_status littlebit_selftest_exchange(int32_t n_rounds, const int32_t *sizes, int32_t n_sizes,
                                      int32_t cluster, int32_t words, void *ws, size_t ws_bytes,
                                      lb_stream_t stream) {
    if (n_rounds < 1 || !sizes || n_sizes < 1 || n_sizes > 8 || (cluster != 1 && cluster != 2) ||
        (words != 1 && words != 2))
        return LB_ERR_INVALID_ARG;
    for (int i = 0; i < n_sizes; ++i)
        if (sizes[i] < 1 || sizes[i] > 2048) return LB_ERR_INVALID_ARG;
    if (!ws || ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) ||
        ws_bytes < lb::xchain_ws_bytes(n_rounds, sizes, n_sizes))
        return LB_ERR_WORKSPACE;
    int sms = 0;
    lb_status st = num_sms(&sms);
    if (st != LB_OK) return st;
    return from_cuda(lb::launch_xchain(n_rounds, sizes, n_sizes, cluster, words,
                                       static_cast<unsigned *>(ws),
                                       static_cast<char *>(ws) + kWsHeader, sms,
                                       (cudaStream_t)stream));
}

}  // extern "C"
