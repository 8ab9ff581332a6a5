// lb_decoder.cu -- one decode step at position p of a Llama-shaped decoder
// whose linears are LittleBit (App. I.3 of LittleBit, arXiv 2506.13771: the
// end-to-end setting replaces only nn.Linear; attention and the norms stay
// dense).  Per layer, with lin[7 l + 0..6] = q, k, v, o, gate, up, down,
// D = head_dim and kv head g = h / (n_heads / n_kv_heads) of query head h:
//   n = rho(a);  q, k, v = Q(n), K(n), V(n)
//   q, k rotated to position p: pairs (i, i + D/2), theta_i = p base^(-2i/D)
//   cache[l][p] = (k, v);  attn_h = softmax_t(q_h . k_t,g / sqrt(D)) . v_t,g
//   a += O(attn);  n = rho(a);  a += Down(silu(G(n)) . U(n))
// with rho(v) = v / sqrt(mean(v^2)), all activations fp32 (as in the
// 70B-shaped stack: rounding them to bf16 before each linear makes a 32-layer
// chain drift by ~7e-3 from its exact value).  The linears run on the
// single-token kernel (k_decode, one cooperative launch each) with fp32
// inputs, every slot of the seven on a workspace of its own; the kernels
// here are the dense glue: the RMS norm and residual (one CTA), attention
// (one CTA per query head) and the SiLU product.  The position lives in
// device memory: every kernel reads it and the last one of the step
// increments it, so a step is a fixed sequence of launches that replays as a
// CUDA graph token after token.
#include <cuda_runtime.h>

#include <cmath>

#include "lb_common.cuh"
#include "lb_kernels.h"

namespace lb {

namespace {

constexpr int kNormThreads = 1024;
constexpr int kMaxHeadDim = 256;

// Word 0 of the decoder header: LB_ERR_RANGE once a step found its position
// outside the cache; every decoder kernel then returns at once.
__device__ __forceinline__ bool dec_ok(const unsigned *hdr) { return ld_relaxed_gpu(hdr) == 0u; }

__device__ __forceinline__ float warp_sum(float v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Reduction over the CTA (blockDim.x a multiple of 32, at most 1024),
// returned to every thread; red holds 32 floats.
template <bool MAX>
__device__ float cta_reduce(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    v = MAX ? warp_max(v) : warp_sum(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float r = lane < nw ? red[lane] : (MAX ? -INFINITY : 0.f);
    return MAX ? warp_max(r) : warp_sum(r);
}

// a = x, n = rho(a); a position outside [0, max_pos) records LB_ERR_RANGE.
__global__ void __launch_bounds__(kNormThreads)
    k_dec_start(const uint16_t *x, float *a, float *n, int d, const int *pos, int max_pos,
                unsigned *hdr) {
    __shared__ float red[32];
    if (!dec_ok(hdr)) return;
    const int p = *pos;
    if (p < 0 || p >= max_pos) {
        if (threadIdx.x == 0) atomicCAS(hdr, 0u, static_cast<unsigned>(LB_ERR_RANGE));
        return;
    }
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const float v = bf16_bits_to_float(x[i]);
        a[i] = v;
        ss += v * v;
    }
    const float inv = 1.f / sqrtf(cta_reduce<false>(ss, red) / (float)d);
    for (int i = threadIdx.x; i < d; i += blockDim.x) n[i] = a[i] * inv;
}

// a += y; then n = rho(a) (n non-null), or out = a and ++*pos (last step of
// the token).
__global__ void __launch_bounds__(kNormThreads)
    k_dec_residual(float *a, const float *y, float *n, int d, float *out, int *pos,
                   const unsigned *hdr) {
    __shared__ float red[32];
    if (!dec_ok(hdr)) return;
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const float v = a[i] + y[i];
        a[i] = v;
        ss += v * v;
    }
    if (n) {
        const float inv = 1.f / sqrtf(cta_reduce<false>(ss, red) / (float)d);
        for (int i = threadIdx.x; i < d; i += blockDim.x) n[i] = a[i] * inv;
    }
    if (out) {
        for (int i = threadIdx.x; i < d; i += blockDim.x) out[i] = a[i];
        __syncthreads();
        if (threadIdx.x == 0) *pos += 1;
    }
}

// Rotary inverse frequencies base^(-2j/D), j < D/2, computed on the host in
// fp64 (a kernel argument).
struct RopeFreq {
    double inv_freq[kMaxHeadDim / 2];
};

// Attention splits per query head: the positions 0..p are cut into kSplits
// runs handled by kSplits CTAs (flash-decoding), so that a long context
// spreads over the SMs instead of one CTA per head.
constexpr int kSplits = 8;

// Attention of query head h = blockIdx.x over its run sp = blockIdx.y of the
// positions, thread i = dimension i of the head (HD = head_dim threads).
// kc / vc: this layer's cache rows [max_pos][d_kv].  Rows t < p come from the
// cache (earlier steps); row p is this step's rotated k and v, which the run
// holding p of the first query head of each kv head also writes into the
// cache.  Scores and the weighted values each take kU positions per warp at a
// time with every load of those positions in flight together.  Each run
// leaves (sum_t e^(s_t - m) v_t, m, sum_t e^(s_t - m)) over its positions in
// part; the last run of a head to finish (a counter in cnt, which it resets)
// rescales the runs to their common maximum and writes the head's output.
template <int HD>
__global__ void __launch_bounds__(HD)
    k_dec_attention(const float *q, const float *k, const float *v, float *kc, float *vc,
                    float *attn, float *part, unsigned *cnt, int n_heads, int n_kv_heads,
                    int max_pos, const __grid_constant__ RopeFreq F, const int *pos,
                    const unsigned *hdr) {
    constexpr int kU = 8, NW = HD / 32, PER = HD / 32;
    extern __shared__ float sm[];
    __shared__ int s_last;
    if (!dec_ok(hdr)) return;
    const int half = HD / 2, i = threadIdx.x;
    const int h = blockIdx.x, sp = blockIdx.y, S = gridDim.y;
    const int group = n_heads / n_kv_heads, g = h / group;
    const int dkv = n_kv_heads * HD, p = *pos;
    // this run's positions [t_lo, t_hi), possibly none
    const int n = p + 1, chunk = (n + S - 1) / S;
    const int t_lo = min(n, sp * chunk), t_hi = min(n, t_lo + chunk);
    const bool has_p = t_lo <= p && p < t_hi;
    float *qs = sm, *ks = sm + HD, *red = sm + 2 * HD, *sc = sm + 2 * HD + 32;
    float *vsum = sc + max_pos;  // [NW][HD]
    qs[i] = q[h * HD + i];
    ks[i] = k[g * HD + i];
    __syncthreads();
    // rotation of the pair (j, j + D/2) by theta_j = p inv_freq_j: the angle in
    // fp64, reduced to [-pi, pi] before the fp32 sine and cosine
    const int j = i < half ? i : i - half;
    const double th = (double)p * F.inv_freq[j];
    const double two_pi = 6.283185307179586476925286766559;
    float sn, cs;
    sincosf((float)(th - two_pi * rint(th / two_pi)), &sn, &cs);
    const float qr = i < half ? qs[i] * cs - qs[i + half] * sn : qs[i - half] * sn + qs[i] * cs;
    const float kr = i < half ? ks[i] * cs - ks[i + half] * sn : ks[i - half] * sn + ks[i] * cs;
    const float vi = v[g * HD + i];
    __syncthreads();
    qs[i] = qr;
    ks[i] = kr;
    if (has_p && h % group == 0) {
        kc[(size_t)p * dkv + g * HD + i] = kr;
        vc[(size_t)p * dkv + g * HD + i] = vi;
    }
    __syncthreads();
    const int lane = i & 31, warp = i >> 5;
    float qreg[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e) qreg[e] = qs[lane + 32 * e];
    const float scale = 1.f / sqrtf((float)HD);
    for (int t0 = t_lo + warp * kU; t0 < t_hi; t0 += NW * kU) {
        float kv[kU][PER];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int t = t0 + u;
            const float *kt = t < p ? kc + (size_t)t * dkv + g * HD : ks;
#pragma unroll
            for (int e = 0; e < PER; ++e)
                kv[u][e] = t < min(p, t_hi) ? __ldg(kt + lane + 32 * e)
                                            : (t == p ? kt[lane + 32 * e] : 0.f);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            float acc = 0.f;
#pragma unroll
            for (int e = 0; e < PER; ++e) acc += qreg[e] * kv[u][e];
            acc = warp_sum(acc);
            if (lane == 0 && t0 + u < t_hi) sc[t0 + u - t_lo] = acc * scale;
        }
    }
    __syncthreads();
    const int len = t_hi - t_lo;
    float mx = -INFINITY;
    for (int t = i; t < len; t += HD) mx = fmaxf(mx, sc[t]);
    mx = cta_reduce<true>(mx, red);
    float sum = 0.f;
    for (int t = i; t < len; t += HD) {
        const float e = expf(sc[t] - mx);
        sc[t] = e;
        sum += e;
    }
    sum = cta_reduce<false>(sum, red);  // its barriers also publish sc
    // weighted values: the same split of positions over warps; the warps'
    // partial vectors meet in shared memory
    float pv[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e) pv[e] = 0.f;
    const int t_end = min(t_hi, p);  // cached rows of the run
    for (int t0 = t_lo + warp * kU; t0 < t_end; t0 += NW * kU) {
        float vv[kU][PER];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int t = t0 + u;
            const float *vt = vc + (size_t)(t < t_end ? t : t_lo) * dkv + g * HD + lane;
#pragma unroll
            for (int e = 0; e < PER; ++e) vv[u][e] = t < t_end ? __ldg(vt + 32 * e) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const float w = t0 + u < t_end ? sc[t0 + u - t_lo] : 0.f;
#pragma unroll
            for (int e = 0; e < PER; ++e) pv[e] += w * vv[u][e];
        }
    }
#pragma unroll
    for (int e = 0; e < PER; ++e) vsum[warp * HD + lane + 32 * e] = pv[e];
    __syncthreads();
    float acc = has_p ? sc[p - t_lo] * vi : 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) acc += vsum[w * HD + i];
    float *mine = part + ((size_t)h * S + sp) * (HD + 2);
    mine[i] = acc;
    if (i == 0) {
        mine[HD] = mx;    // -inf for a run without positions
        mine[HD + 1] = sum;
    }
    __threadfence();
    __syncthreads();
    if (i == 0) s_last = atomicAdd(cnt + h, 1u) == (unsigned)(S - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const float *runs = part + (size_t)h * S * (HD + 2);
    float M = -INFINITY;
    for (int r = 0; r < S; ++r) M = fmaxf(M, __ldcg(runs + r * (HD + 2) + HD));
    float L = 0.f, O = 0.f;
    for (int r = 0; r < S; ++r) {
        const float m_r = __ldcg(runs + r * (HD + 2) + HD);
        const float w = m_r == -INFINITY ? 0.f : expf(m_r - M);
        L += w * __ldcg(runs + r * (HD + 2) + HD + 1);
        O += w * __ldcg(runs + r * (HD + 2) + i);
    }
    attn[h * HD + i] = O / L;
    if (i == 0) cnt[h] = 0u;
}

size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

struct DecLayout {
    size_t slot[7];        // byte offsets of the seven single-linear workspaces
    size_t slot_bytes[7];
    size_t qkv_ws, qkv_bytes, gu_ws, gu_bytes;  // the two multi-linear workspaces
    size_t n, attn, q, k, v, y, g, u, a, part, cnt, end;
};

// The grouped launches of a layer: q with k and v when all three have one
// shape (else k and v together, q alone), gate with up.
struct DecGroups {
    int qkv;  // 3: q, k, v in one launch; 2: k, v in one launch; 0: none
    bool gu;
};

DecLayout dec_layout(const lb_linear *lin, const lb_decoder_shape &S) {
    DecLayout o{};
    size_t off = kWsHeader;
    for (int j = 0; j < 7; ++j) {
        o.slot[j] = off;
        o.slot_bytes[j] = kWsHeader + align256(decode_ws_bytes(lin[j]));
        off += o.slot_bytes[j];
    }
    o.qkv_ws = off;
    o.qkv_bytes = kWsHeader + align256(multi_ws_bytes(lin[1], 3));
    off += o.qkv_bytes;
    o.gu_ws = off;
    o.gu_bytes = kWsHeader + align256(multi_ws_bytes(lin[4], 2));
    off += o.gu_bytes;
    const size_t d = (size_t)S.n_heads * S.head_dim, dkv = (size_t)S.n_kv_heads * S.head_dim;
    const size_t dff = (size_t)lin[4].d_out;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off += align256(bytes);
        return at;
    };
    o.n = take(d * 4);
    o.attn = take(d * 4);
    o.q = take((d + 2 * dkv) * 4);  // q, k, v back to back (the rows of a grouped launch)
    o.k = o.q + d * 4;
    o.v = o.k + dkv * 4;
    o.y = take(d * 4);
    o.g = take(2 * dff * 4);        // gate, up back to back
    o.u = o.g + dff * 4;
    o.a = take(d * 4);
    o.part = take((size_t)S.n_heads * kSplits * (S.head_dim + 2) * 4);  // attention runs
    o.cnt = take((size_t)S.n_heads * 4);                                 // zero between steps
    o.end = off;
    return o;
}

bool same_shape(const lb_linear &A, const lb_linear &B) {
    if (A.d_in != B.d_in || A.d_out != B.d_out || A.n_paths != B.n_paths) return false;
    for (int p = 0; p < A.n_paths; ++p)
        if (A.path[p].r != B.path[p].r) return false;
    return true;
}

// Shapes: q d -> d, k and v d -> d_kv, o d -> d, gate and up d -> d_ff, down
// d_ff -> d, the same in every layer (the slot workspaces are sized once).
lb_status check_decoder(const lb_linear *lin, const lb_decoder_shape *S) {
    if (!lin || !S) return LB_ERR_INVALID_ARG;
    if (S->n_layers < 1 || S->n_heads < 1 || S->n_kv_heads < 1 || S->n_heads % S->n_kv_heads != 0 ||
        (S->head_dim != 64 && S->head_dim != 128 && S->head_dim != 256) ||
        S->max_pos < 1 || S->max_pos > 8192 || !(S->rope_base > 1.f))
        return LB_ERR_INVALID_ARG;
    const int d = S->n_heads * S->head_dim, dkv = S->n_kv_heads * S->head_dim;
    const int dff = lin[4].d_out;
    const int din[7] = {d, d, d, d, d, d, dff}, dout[7] = {d, dkv, dkv, d, dff, dff, d};
    for (int l = 0; l < S->n_layers; ++l)
        for (int j = 0; j < 7; ++j) {
            const lb_linear &L = lin[7 * (size_t)l + j];
            if (validate_linear(&L) != LB_OK) return LB_ERR_INVALID_ARG;
            if (L.d_in != din[j] || L.d_out != dout[j] || !same_shape(L, lin[j]))
                return LB_ERR_UNSUPPORTED;
            // the single-token kernel's shape rules
            if (L.d_out % 8 != 0) return LB_ERR_UNSUPPORTED;
            for (int p = 0; p < L.n_paths; ++p)
                if (L.path[p].r % 8 != 0) return LB_ERR_UNSUPPORTED;
        }
    return LB_OK;
}

lb_status from_err(cudaError_t e) { return e == cudaSuccess ? LB_OK : LB_ERR_CUDA; }

DecGroups groups_of(const lb_linear *lin, int sms) {
    DecGroups G{};
    const lb_linear qkv[3] = {lin[0], lin[1], lin[2]};
    if (multi_supported(qkv, 3, sms)) G.qkv = 3;
    else if (multi_supported(qkv + 1, 2, sms)) G.qkv = 2;
    const lb_linear gu[2] = {lin[4], lin[5]};
    G.gu = multi_supported(gu, 2, sms);
    return G;
}

// SM count of the current device (cached per device).
int sm_count() {
    static int sms[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        sms[dev] = n;
    }
    return sms[dev];
}

}  // namespace

}  // namespace lb

extern "C" {

size_t littlebit_decoder_workspace_size(const lb_linear *lin, const lb_decoder_shape *S) {
    if (lb::check_decoder(lin, S) != LB_OK) return 0;
    return lb::dec_layout(lin, *S).end;
}

lb_status littlebit_decoder_step(const lb_linear *lin, const lb_decoder_shape *S,
                                 const uint16_t *x, float *kcache, float *vcache, int32_t *pos,
                                 float *out, void *ws, size_t ws_bytes, lb_stream_t stream) {
    using namespace lb;
    lb_status st = check_decoder(lin, S);
    if (st != LB_OK) return st;
    if (!x || !kcache || !vcache || !pos || !out) return LB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(kcache) |
         reinterpret_cast<uintptr_t>(vcache) | reinterpret_cast<uintptr_t>(out)) & 15u)
        return LB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(pos) & 3u) != 0) return LB_ERR_INVALID_ARG;
    const DecLayout o = dec_layout(lin, *S);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < o.end)
        return LB_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    char *w = static_cast<char *>(ws);
    unsigned *hdr = reinterpret_cast<unsigned *>(w);
    float *n = reinterpret_cast<float *>(w + o.n);
    float *attn = reinterpret_cast<float *>(w + o.attn);
    float *q = reinterpret_cast<float *>(w + o.q), *k = reinterpret_cast<float *>(w + o.k);
    float *v = reinterpret_cast<float *>(w + o.v), *y = reinterpret_cast<float *>(w + o.y);
    float *g = reinterpret_cast<float *>(w + o.g), *u = reinterpret_cast<float *>(w + o.u);
    float *a = reinterpret_cast<float *>(w + o.a);
    float *part = reinterpret_cast<float *>(w + o.part);
    unsigned *cnt = reinterpret_cast<unsigned *>(w + o.cnt);
    const int d = S->n_heads * S->head_dim, dkv = S->n_kv_heads * S->head_dim;
    const int D = S->head_dim;
    const size_t layer_rows = (size_t)S->max_pos * dkv;
    const size_t attn_smem = (size_t)(2 * D + 32 + S->max_pos + D * D / 32) * sizeof(float);
    RopeFreq freq{};
    for (int j = 0; j < D / 2; ++j)
        freq.inv_freq[j] = std::pow((double)S->rope_base, -2.0 * (double)j / (double)D);
    const int sms = sm_count();
    if (sms < 1 || !decode_supported(lin[0], sms)) return LB_ERR_UNSUPPORTED;
    // x_mode 1: fp32 input; 2: silu(xin[i]) * xin[d_in + i] (gate, up back to back)
    auto linear = [&](int l, int j, const float *xin, float *yout, int x_mode = 1) {
        char *slot = w + o.slot[j];
        const cudaError_t e = launch_decode(lin[7 * (size_t)l + j], xin, x_mode, yout, 1,
                                            reinterpret_cast<unsigned *>(slot), slot + kWsHeader,
                                            sms, s);
        return e == cudaErrorCooperativeLaunchTooLarge ? LB_ERR_UNSUPPORTED : from_err(e);
    };
    // linears j .. j + M - 1 of layer l in one launch (outputs back to back);
    // with fold, their input is a += y and they apply rho themselves
    auto group = [&](int l, int j, int M, size_t ws_off, const float *xin, float *yout,
                     bool fold = false) {
        char *gw = w + ws_off;
        const cudaError_t e = launch_decode_multi(&lin[7 * (size_t)l + j], M, fold ? nullptr : xin,
                                                  fold ? 3 : 1, yout, 1,
                                                  reinterpret_cast<unsigned *>(gw),
                                                  gw + kWsHeader, sms, s, fold ? a : nullptr,
                                                  fold ? y : nullptr);
        return e == cudaErrorCooperativeLaunchTooLarge ? LB_ERR_UNSUPPORTED : from_err(e);
    };
    const DecGroups G = groups_of(lin, sms);
    k_dec_start<<<1, kNormThreads, 0, s>>>(x, a, n, d, pos, S->max_pos, hdr);
    if ((st = from_err(cudaGetLastError())) != LB_OK) return st;
    // The residual add and RMS norm ahead of a grouped launch run inside it
    // (a += y, its outputs scaled by 1 / rms(a)): ahead of gate / up always,
    // ahead of q / k / v when the three are grouped (from layer 1 on).
    for (int l = 0; l < S->n_layers; ++l) {
        const bool last = l + 1 == S->n_layers;
        if (G.qkv == 3) {
            if ((st = group(l, 0, 3, o.qkv_ws, n, q, l > 0)) != LB_OK) return st;
        } else if (G.qkv == 2) {
            if ((st = linear(l, 0, n, q)) != LB_OK || (st = group(l, 1, 2, o.qkv_ws, n, k)) != LB_OK)
                return st;
        } else if ((st = linear(l, 0, n, q)) != LB_OK || (st = linear(l, 1, n, k)) != LB_OK ||
                   (st = linear(l, 2, n, v)) != LB_OK) {
            return st;
        }
        float *kl = kcache + l * layer_rows, *vl = vcache + l * layer_rows;
        const dim3 agrid(S->n_heads, kSplits);
        if (D == 64)
            k_dec_attention<64><<<agrid, 64, attn_smem, s>>>(q, k, v, kl, vl, attn, part, cnt,
                                                            S->n_heads, S->n_kv_heads,
                                                            S->max_pos, freq, pos, hdr);
        else if (D == 128)
            k_dec_attention<128><<<agrid, 128, attn_smem, s>>>(q, k, v, kl, vl, attn, part, cnt,
                                                              S->n_heads, S->n_kv_heads,
                                                              S->max_pos, freq, pos, hdr);
        else
            k_dec_attention<256><<<agrid, 256, attn_smem, s>>>(q, k, v, kl, vl, attn, part, cnt,
                                                              S->n_heads, S->n_kv_heads,
                                                              S->max_pos, freq, pos, hdr);
        if ((st = from_err(cudaGetLastError())) != LB_OK) return st;
        if ((st = linear(l, 3, attn, y)) != LB_OK) return st;
        if (G.gu) {
            if ((st = group(l, 4, 2, o.gu_ws, nullptr, g, true)) != LB_OK) return st;
        } else {
            k_dec_residual<<<1, kNormThreads, 0, s>>>(a, y, n, d, nullptr, nullptr, hdr);
            if ((st = from_err(cudaGetLastError())) != LB_OK) return st;
            if ((st = linear(l, 4, n, g)) != LB_OK || (st = linear(l, 5, n, u)) != LB_OK)
                return st;
        }
        // down reads silu(gate) * up straight from the gate / up outputs
        if ((st = linear(l, 6, g, y, 2)) != LB_OK) return st;
        if (last || G.qkv != 3) {
            k_dec_residual<<<1, kNormThreads, 0, s>>>(a, y, last ? nullptr : n, d,
                                                      last ? out : nullptr, last ? pos : nullptr,
                                                      hdr);
            if ((st = from_err(cudaGetLastError())) != LB_OK) return st;
        }
    }
    return LB_OK;
}

lb_status littlebit_decoder_poll_error(const lb_linear *lin, const lb_decoder_shape *S, void *ws,
                                       lb_stream_t stream) {
    using namespace lb;
    lb_status st = check_decoder(lin, S);
    if (st != LB_OK) return st;
    if (!ws) return LB_ERR_WORKSPACE;
    const DecLayout o = dec_layout(lin, *S);
    char *w = static_cast<char *>(ws);
    // the decoder's own word first, then each linear slot's workspace
    lb_status first = littlebit_poll_error(w, stream);
    for (int j = 0; j < 9; ++j) {
        const size_t at = j < 7 ? o.slot[j] : (j == 7 ? o.qkv_ws : o.gu_ws);
        const lb_status e = littlebit_poll_error(w + at, stream);
        if (first == LB_OK) first = e;
    }
    return first;
}

}  // extern "C"
