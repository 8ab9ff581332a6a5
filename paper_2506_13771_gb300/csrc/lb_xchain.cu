// lb_xchain.cu -- exchange-chain diagnostic (littlebit_selftest_exchange):
// the latency floor of the all-reduce that the single-token kernels run
// between stage 1 and stage 2 of every linear (Prop. 1: t = V_sign^T (g . x)
// summed over the CTAs' input slices), with no weights and no arithmetic
// around it.
//
// One persistent launch, one CTA per SM (cooperative; 2-CTA clusters when
// asked), runs n_rounds dependent exchanges.  Round k has sizes[k % n_sizes]
// elements: every CTA contributes a value to every element exactly as the
// stack kernel's stage 1 does (with clusters: the pair's partials meet in the
// owner's shared memory through st.async + mbarrier, and the owner sends one
// contribution per cluster), then polls every element exactly as the stack
// kernel's stage-2 tables do (one gating lane per 128-element unit, then four
// elements per lane) until all are complete, and only then starts round k+1.
// W = 1 encodes every element as the stack does (one word at a scale set
// from a bound, send_fix1), W = 2 as the single-token kernels do (the exact
// hi / lo pair, send_fix2).  The time per round is the exchange's floor on
// the critical path: the kernels add their +-1 sums to it.  Every wait is
// bounded.
#include "lb_common.cuh"
#include "lb_kernels.h"
#include "lb_lut.cuh"

namespace lb {

namespace {

constexpr int kXT = 512;
constexpr int kXW = kXT / 32;
constexpr int kXMaxUnits = 64;  // 32-element units per round: at most 2048 elements

struct XchainParams {
    unsigned long long *buf;  // n_rounds buffers of `stride` words, zero
    unsigned *ws_words;
    int n_rounds, n_sizes, stride;
    int sizes[8];
    unsigned n_contrib;
    float limit;
};

__device__ __forceinline__ bool xc_sticky(const unsigned *w) {
    return ld_relaxed_gpu(w + kErrWord) != 0u;
}

template <int C, int W>
__global__ void __launch_bounds__(kXT, 1) k_xchain(const __grid_constant__ XchainParams P) {
    __shared__ __align__(8) unsigned long long ubar[kXMaxUnits / 2];
    __shared__ float slot[kXMaxUnits / 2][32];
    unsigned *ws = P.ws_words;
    if (xc_sticky(ws)) return;
    if (C > 1 && cluster_size() != (unsigned)C) {
        // not launched in clusters of C: no other CTA's memory is touched
        if (threadIdx.x == 0) atomicCAS(ws + kErrWord, 0u, static_cast<unsigned>(LB_ERR_UNSUPPORTED));
        return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const unsigned rank = C > 1 ? cluster_rank() : 0u;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kXMaxUnits / 2; ++i) mbar_init(ubar + i, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (C > 1) cluster_sync_all();
    // this CTA's contribution: 2^-10 * (blockIdx + 1), exactly representable;
    // a cluster's sum is below 2 gridDim 2^-10 (the one-word scale's bound)
    const float v = (float)(blockIdx.x + 1) * 0x1p-10f;
    const float sc = fix1_scale(2.f * (float)gridDim.x * 0x1p-10f, (int)P.n_contrib).x;

    unsigned long long *xk = P.buf;
    auto x_at = [&](int e) { return xk + e; };
    auto send = [&](int e, float a) {
        if (W == 1)
            send_fix1(x_at(e), a, sc, P.limit, ws + kErrWord);
        else
            send_fix2(fix2_at(xk, e), a, P.limit, ws + kErrWord);
    };
    for (int k = 0; k < P.n_rounds; ++k) {
        xk = P.buf + (size_t)k * P.stride;
        const int n = P.sizes[k % P.n_sizes];
        const int units = (n + 31) >> 5;
        const unsigned par = (unsigned)(k & 1);
        bool ok = true;
        // ---- contributions: unit u (32 elements) on warp u % 16.  Every
        //      mbarrier is armed once per round (with no bytes for units
        //      beyond this round's size), so its parity is the round's.
        if (C > 1 && lane == 0)
            for (int u = warp; u < kXMaxUnits; u += kXW)
                if ((unsigned)(u % C) == rank)
                    mbar_arrive_expect_tx(ubar + u / C,
                                          (unsigned)((C - 1) * 4 * max(0, min(32, n - 32 * u))));
        __syncwarp();
        for (int u = warp; u < units; u += kXW) {
            const int e = 32 * u + lane;
            if (C == 1) {
                if (e < n) send(e, v);
                continue;
            }
            const unsigned own = (unsigned)(u % C);
            if (own != rank) {
                if (e < n)
                    st_async_f32(mapa(saddr(&slot[u / C][lane]), own), v,
                                 mapa(saddr(ubar + u / C), own));
                continue;
            }
            if (!ok) continue;
            if (!mbar_try_wait_cluster(ubar + u / C, par)) {
                const unsigned long long t0 = globaltimer_ns();
                while (!mbar_try_wait_cluster(ubar + u / C, par)) {
                    if (xc_sticky(ws) || globaltimer_ns() - t0 > kWaitLimitNs) {
                        atomicCAS(ws + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                        ok = false;
                        break;
                    }
                }
                if (!ok) continue;
            }
            // the peer's partial beside this CTA's own, in rank order
            const float sum = rank == 0 ? v + slot[u / C][lane] : slot[u / C][lane] + v;
            if (e < n) send(e, sum);
        }
        // ---- polls: 128-element unit q on warp q % 16
        for (int q = warp; q < (n + 127) / 128 && ok; q += kXW) {
            const int e0 = 128 * q, m = min(128, n - e0);
            if (lane == 0) {
                // the last element's (lo) word
                const unsigned long long *gw = W == 1 ? x_at(e0 + m - 1) : fix2_at(xk, e0 + m - 1) + 32;
                const unsigned long long t0 = globaltimer_ns();
                for (int spin = 0; (unsigned)(ld_relaxed_u64(gw) & 0xffull) != P.n_contrib; ++spin)
                    if ((spin & 15) == 15 && globaltimer_ns() - t0 > kWaitLimitNs) break;
            }
            __syncwarp();
            if (4 * lane >= m) continue;
            // element groups of 4 stay inside one 32-element block (n is padded
            // to whole blocks in the buffer, and the padding stays zero)
            const unsigned long long *w = W == 1 ? x_at(e0 + 4 * lane) : fix2_at(xk, e0 + 4 * lane);
            const int have = min(4, m - 4 * lane);
            unsigned long long a[8];
            const unsigned long long t0 = globaltimer_ns();
            for (int spin = 0;; ++spin) {
                bool done = true;
                if (W == 1) {
                    ld_relaxed_v2_u64(w, a[0], a[1]);
                    ld_relaxed_v2_u64(w + 2, a[2], a[3]);
                    for (int j = 0; j < have; ++j) done = done && counted1(a[j], P.n_contrib);
                } else {
                    ld_fix2x4(w, a);
                    for (int j = 0; j < have; ++j)
                        done = done && counted2(a[2 * j], a[2 * j + 1], P.n_contrib);
                }
                if (done) break;
                if ((spin & 15) == 15 &&
                    (xc_sticky(ws) || globaltimer_ns() - t0 > kWaitLimitNs)) {
                    atomicCAS(ws + kErrWord, 0u, static_cast<unsigned>(LB_ERR_TIMEOUT));
                    ok = false;
                    break;
                }
            }
        }
        if (!__syncthreads_and(ok)) break;
    }
    // no CTA leaves while its cluster peer may still store into its shared memory
    if (C > 1) cluster_sync_all();
}

}  // namespace

size_t xchain_ws_bytes(int n_rounds, const int *sizes, int n_sizes) {
    int mx = 0;
    for (int i = 0; i < n_sizes; ++i) mx = sizes[i] > mx ? sizes[i] : mx;
    return kWsHeader + (size_t)n_rounds * fix2_words((size_t)mx) * sizeof(unsigned long long);
}

cudaError_t launch_xchain(int n_rounds, const int *sizes, int n_sizes, int cluster, int words,
                          unsigned *ws_words, void *buf, int num_sms, cudaStream_t s) {
    if (n_rounds < 1 || n_sizes < 1 || n_sizes > 8 || (cluster != 1 && cluster != 2) ||
        (words != 1 && words != 2))
        return cudaErrorInvalidValue;
    XchainParams P{};
    int mx = 0;
    for (int i = 0; i < n_sizes; ++i) {
        if (sizes[i] < 1 || sizes[i] > 32 * kXMaxUnits) return cudaErrorInvalidValue;
        P.sizes[i] = sizes[i];
        mx = sizes[i] > mx ? sizes[i] : mx;
    }
    const int N = num_sms - num_sms % cluster;
    if (N < cluster || N > 255) return cudaErrorInvalidValue;
    P.buf = static_cast<unsigned long long *>(buf);
    P.ws_words = ws_words;
    P.n_rounds = n_rounds;
    P.n_sizes = n_sizes;
    P.stride = (int)fix2_words((size_t)mx);
    P.n_contrib = (unsigned)(N / cluster);
    // one word: below 2^55 / n (n contributions then sum to less than 2^55)
    P.limit = words == 1 ? 0x1p54f / (float)P.n_contrib : fix2_limit(N);
    cudaError_t e = cudaMemsetAsync(buf, 0, (size_t)n_rounds * P.stride * sizeof(unsigned long long),
                                    s);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(N, 1, 1);
    cfg.blockDim = dim3(kXT, 1, 1);
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeCooperative;
    at[0].val.cooperative = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cluster;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    if (words == 1)
        return cluster == 2 ? cudaLaunchKernelEx(&cfg, k_xchain<2, 1>, P)
                            : cudaLaunchKernelEx(&cfg, k_xchain<1, 1>, P);
    return cluster == 2 ? cudaLaunchKernelEx(&cfg, k_xchain<2, 2>, P)
                        : cudaLaunchKernelEx(&cfg, k_xchain<1, 2>, P);
}

}  // namespace lb
